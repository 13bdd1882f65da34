// Decode-step attention for dynamic prediction (Sec. 3.2, t >= 1): one new
// query token per request attends to every cached draft key/value of its
// request plus its own (already appended to the paged cache).
//
// Cache layout: pools [pages][KVH][page_tokens = 64][hd]; a request's keys are
// the concatenation of its pages (page list uploaded per call).  The same
// kernels read the head-major K/V of a static prediction ([KVH, kv_ld, hd],
// "pages" of 64 rows from each prompt's first row) to attend from each
// prompt's last row: the first row of a page is page * page_stride + kv head
// * head_stride.
//
// bf16 path: split-KV.  One CTA = (request, split of <= split_len keys, kv
// head).  The G = H / KVH query heads of the kv head form the rows of one
// 16-row mma.sync tile, so every K/V byte is read from HBM once.  Page blocks
// (64 keys x hd) of K and V are staged by TMA (128-byte swizzle, 2 stages,
// three CTAs per SM so one CTA's start-up is covered by two streaming ones);
// each of the 4 warps takes 16 keys of a page, keeps its own online softmax,
// and the warps are merged through shared memory.  Requests with one split
// write the output directly; others write (o, m, l) partials, and the last
// split CTA of each (request, kv head) to finish merges them (a fenced
// completion counter; no CTA waits for another).
//
// f32 path: one warp per (request, head), lanes own head dims.
#include "common.cuh"
#include "kernels.h"
#include "mma_sync.cuh"

namespace outlets {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kStages = 2;

template <int HD>
struct DecCfg {
  static constexpr int PAGE_BYTES = 64 * HD * 2;    // one page-head block of K (or V)
  static constexpr int Q_BYTES = 16 * HD * 2;       // 16-row query tile
  static constexpr size_t SMEM = 1024 + Q_BYTES + kStages * 2 * PAGE_BYTES + 128;
};

// Merge the split partials of request b, heads h0 .. h0 + nh - 1:
// out = sum_s w_s o_s / sum_s w_s with w_s = l_s * 2^(m_s - max m), splits
// added in order.  The (m, l) pairs and the weights are staged in `scratch`
// (2 * nh * ns + nh floats); each output then issues the loads of up to eight
// splits together.  Partials written by other CTAs are read through L2.
template <int HD>
__device__ __forceinline__ void merge_splits(const DecodeArgs& a, int b, int h0, int nh, float* scratch) {
  const int w0 = a.work_off[b];
  const int ns = a.work_off[b + 1] - w0;
  float* ml = scratch;           // [nh][ns][2]
  float* wt = scratch + 2 * nh * ns;  // [nh][ns] weights, then [nh] their sums
  float* lsum = wt + nh * ns;
  for (int i = threadIdx.x; i < nh * ns * 2; i += blockDim.x) {
    const int r = i / (2 * ns), rem = i - r * 2 * ns;
    ml[i] = __ldcg(&a.part_ml[((long long)(w0 + (rem >> 1)) * a.H + h0 + r) * 2 + (rem & 1)]);
  }
  __syncthreads();
  for (int r = threadIdx.x; r < nh; r += blockDim.x) {
    float M = -INFINITY;
    for (int w = 0; w < ns; ++w) M = fmaxf(M, ml[(r * ns + w) * 2]);
    const float Mu = (M == -INFINITY) ? 0.f : M;
    float Ls = 0.f;
    for (int w = 0; w < ns; ++w) {
      const float f = exp2f(ml[(r * ns + w) * 2] - Mu) * ml[(r * ns + w) * 2 + 1];
      wt[r * ns + w] = f;
      Ls += f;
    }
    lsum[r] = Ls;
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < nh * HD; idx += blockDim.x) {
    const int r = idx / HD;
    const int d = idx - r * HD;
    const float* po = a.part_o + ((long long)w0 * a.H + h0 + r) * HD + d;
    const long long wstride = (long long)a.H * HD;
    float Os = 0.f;
    for (int w = 0; w < ns; w += 8) {
      float o[8];
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (w + k < ns) o[k] = __ldcg(po + (w + k) * wstride);
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (w + k < ns) Os += wt[r * ns + w + k] * o[k];
    }
    const long long oi = ((long long)b * a.H + h0 + r) * HD + d;
    const float gv = a.gate ? __bfloat162float(reinterpret_cast<const bf16*>(a.gate)[oi]) : 1.f;  // gated attention
    reinterpret_cast<bf16*>(a.out)[oi] = __float2bfloat16_rn(Os / lsum[r] * gv);
  }
}

template <int HD>
__global__ void __launch_bounds__(128, 3)
    k_attn_decode_bf16(const __grid_constant__ CUtensorMap k_map, const __grid_constant__ CUtensorMap v_map,
                       const DecodeArgs a) {
  pdl_trigger();
  pdl_wait();
  using C = DecCfg<HD>;
  constexpr int NB = HD / 64;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sKV = smem + C::Q_BYTES;  // stage s: K at s*2*PAGE, V at s*2*PAGE + PAGE
  uint64_t* full = reinterpret_cast<uint64_t*>(sKV + kStages * 2 * C::PAGE_BYTES);
  uint64_t* empty = full + kStages;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty + kStages);

  const int item = a.order ? a.order[blockIdx.x] : (int)blockIdx.x;  // work item of this CTA
  const int2 wk = reinterpret_cast<const int2*>(a.work)[item];
  const int b = wk.x;
  const int split = wk.y;
  const int g = blockIdx.y;
  const int G = a.H / a.KVH;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int L = a.seq_len[b];
  const int key_begin = split * a.split_len;
  const int key_end = min(L, key_begin + a.split_len);
  const int page_begin = key_begin / 64;
  const int n_pages = (key_end - key_begin + 63) / 64;
  const int* pages = a.page_list + a.page_off[b];

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 4);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  // query rows r < G: heads g*G + r of request b; rows >= G are zero
  {
    const bf16* qsrc = reinterpret_cast<const bf16*>(a.q) + ((long long)b * a.H + (long long)g * G) * HD;
    for (int c = threadIdx.x; c < 16 * (HD / 8); c += blockDim.x) {
      const int r = c / (HD / 8);
      const int d = (c % (HD / 8)) * 8;
      uint4 val = make_uint4(0, 0, 0, 0);
      if (r < G) val = *reinterpret_cast<const uint4*>(qsrc + r * HD + d);
      *reinterpret_cast<uint4*>(sQ + sw128_offset<16>(r, d)) = val;
    }
  }
  __syncthreads();

  // K/V pages are read once per call and the cache is far larger than L2:
  // evict them first, so the weights the next kernels prefetched stay in L2
  const uint64_t kv_policy = l2_evict_first_policy();
  auto issue = [&](int pi, int stage) {
    const int row = (int)((long long)pages[page_begin + pi] * a.page_stride + (long long)g * a.head_stride);
    uint8_t* dk = sKV + stage * 2 * C::PAGE_BYTES;
    mbar_arrive_expect_tx(&full[stage], 2 * C::PAGE_BYTES);
#pragma unroll
    for (int bx = 0; bx < NB; ++bx) {
      tma_load_2d_hint(dk + bx * 8192, &k_map, &full[stage], bx * 64, row, kv_policy);
      tma_load_2d_hint(dk + C::PAGE_BYTES + bx * 8192, &v_map, &full[stage], bx * 64, row, kv_policy);
    }
  };
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages && s < n_pages; ++s) issue(s, s);
  }

  uint32_t qf[HD / 16][4];
  {
    const uint32_t qbase = smem_u32(sQ);
    const int r = (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
      const int d = ks * 16 + ((lane >> 4) & 1) * 8;
      ldsm_x4(qbase + sw128_offset<16>(r, d), qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3]);
    }
  }

  float o[HD / 8][4];
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  const float sl2 = rsqrtf((float)HD) * kLog2e;
  bool ok = true;

  for (int pi = 0; pi < n_pages; ++pi) {
    const int stage = pi % kStages;
    const uint32_t par = (pi / kStages) & 1;
    if (!mbar_wait(&full[stage], par, abort_flag, a.err)) {
      ok = false;
      break;
    }
    const uint32_t kbase = smem_u32(sKV + stage * 2 * C::PAGE_BYTES);
    const uint32_t vbase = kbase + C::PAGE_BYTES;
    const int key_pg = (page_begin + pi) * 64;  // request-relative index of the page's first key

    float s[2][4];
#pragma unroll
    for (int j = 0; j < 2; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
      uint32_t b0, b1, b2, b3;
      const int key = warp * 16 + (lane & 7) + ((lane >> 4) & 1) * 8;
      const int d = ks * 16 + ((lane >> 3) & 1) * 8;
      ldsm_x4(kbase + sw128_offset<64>(key, d), b0, b1, b2, b3);
      mma_16816(s[0], qf[ks], b0, b1);
      mma_16816(s[1], qf[ks], b2, b3);
    }
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int kc = key_pg + warp * 16 + 8 * j + 2 * (lane & 3);
      const bool v0 = kc >= key_begin && kc < key_end;
      const bool v1 = kc + 1 >= key_begin && kc + 1 < key_end;
      s[j][0] = v0 ? s[j][0] * sl2 : -INFINITY;
      s[j][1] = v1 ? s[j][1] * sl2 : -INFINITY;
      s[j][2] = v0 ? s[j][2] * sl2 : -INFINITY;
      s[j][3] = v1 ? s[j][3] * sl2 : -INFINITY;
      mx0 = fmaxf(mx0, fmaxf(s[j][0], s[j][1]));
      mx1 = fmaxf(mx1, fmaxf(s[j][2], s[j][3]));
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float mn0 = fmaxf(m0, mx0);
    const float mn1 = fmaxf(m1, mx1);
    const float mu0 = (mn0 == -INFINITY) ? 0.f : mn0;
    const float mu1 = (mn1 == -INFINITY) ? 0.f : mn1;
    const float c0 = exp2f(m0 - mu0);
    const float c1 = exp2f(m1 - mu1);
    m0 = mn0;
    m1 = mn1;
    float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      s[j][0] = exp2f(s[j][0] - mu0);
      s[j][1] = exp2f(s[j][1] - mu0);
      s[j][2] = exp2f(s[j][2] - mu1);
      s[j][3] = exp2f(s[j][3] - mu1);
      ps0 += s[j][0] + s[j][1];
      ps1 += s[j][2] + s[j][3];
    }
    l0 = l0 * c0 + ps0;
    l1 = l1 * c1 + ps1;
    uint32_t pa[4];
    pa[0] = pack_bf16x2(s[0][0], s[0][1]);
    pa[1] = pack_bf16x2(s[0][2], s[0][3]);
    pa[2] = pack_bf16x2(s[1][0], s[1][1]);
    pa[3] = pack_bf16x2(s[1][2], s[1][3]);
#pragma unroll
    for (int dp = 0; dp < HD / 16; ++dp) {
      o[2 * dp][0] *= c0;
      o[2 * dp][1] *= c0;
      o[2 * dp][2] *= c1;
      o[2 * dp][3] *= c1;
      o[2 * dp + 1][0] *= c0;
      o[2 * dp + 1][1] *= c0;
      o[2 * dp + 1][2] *= c1;
      o[2 * dp + 1][3] *= c1;
      uint32_t b0, b1, b2, b3;
      const int key = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
      const int d = dp * 16 + ((lane >> 4) & 1) * 8;
      ldsm_x4_t(vbase + sw128_offset<64>(key, d), b0, b1, b2, b3);
      mma_16816(o[2 * dp], pa, b0, b1);
      mma_16816(o[2 * dp + 1], pa, b2, b3);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[stage]);
    if (threadIdx.x == 0 && pi + kStages < n_pages) {
      if (!mbar_wait(&empty[stage], par, abort_flag, a.err)) {
        ok = false;
        break;
      }
      issue(pi + kStages, stage);
    }
  }

  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);

  // merge the 4 warps: reuse the K/V ring (all copies have landed and been read)
  __syncthreads();
  float* sm_ml = reinterpret_cast<float*>(sKV);        // [4 warps][16 rows][2]
  float* sm_o = sm_ml + 4 * 16 * 2;                     // [4 warps][16 rows][HD]
  {
    const int r0 = lane >> 2, r1 = r0 + 8;
    if ((lane & 3) == 0) {
      sm_ml[(warp * 16 + r0) * 2 + 0] = m0;
      sm_ml[(warp * 16 + r0) * 2 + 1] = l0;
      sm_ml[(warp * 16 + r1) * 2 + 0] = m1;
      sm_ml[(warp * 16 + r1) * 2 + 1] = l1;
    }
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) {
      const int d = 8 * j + 2 * (lane & 3);
      sm_o[(warp * 16 + r0) * HD + d] = o[j][0];
      sm_o[(warp * 16 + r0) * HD + d + 1] = o[j][1];
      sm_o[(warp * 16 + r1) * HD + d] = o[j][2];
      sm_o[(warp * 16 + r1) * HD + d + 1] = o[j][3];
    }
  }
  __syncthreads();
  if (!ok || *abort_flag) return;
  const int n_split = a.work_off[b + 1] - a.work_off[b];
  for (int idx = threadIdx.x; idx < G * HD; idx += blockDim.x) {
    const int r = idx / HD;
    const int d = idx - r * HD;
    float M = -INFINITY;
    for (int w = 0; w < 4; ++w) M = fmaxf(M, sm_ml[(w * 16 + r) * 2]);
    const float Mu = (M == -INFINITY) ? 0.f : M;
    float Ls = 0.f, Os = 0.f;
    for (int w = 0; w < 4; ++w) {
      const float f = exp2f(sm_ml[(w * 16 + r) * 2] - Mu);
      Ls += f * sm_ml[(w * 16 + r) * 2 + 1];
      Os += f * sm_o[(w * 16 + r) * HD + d];
    }
    const int head = g * G + r;
    if (n_split == 1) {
      const long long oi = ((long long)b * a.H + head) * HD + d;
      const float gv = a.gate ? __bfloat162float(reinterpret_cast<const bf16*>(a.gate)[oi]) : 1.f;
      reinterpret_cast<bf16*>(a.out)[oi] = __float2bfloat16_rn(Os / Ls * gv);
    } else {
      const long long pi = (long long)item * a.H + head;  // partial index: (work item, head)
      a.part_o[pi * HD + d] = Os / Ls;
      if (d == 0) {
        a.part_ml[pi * 2 + 0] = M;
        a.part_ml[pi * 2 + 1] = Ls;
      }
    }
  }
  if (n_split == 1) return;
  // The last split CTA of (request, KV group) to finish merges all splits:
  // each CTA publishes its partial (fence, then count); the one that brings
  // the count to n_split reads every partial and resets the counter for the
  // next call.  No CTA waits for another.
  __shared__ int is_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int prev = atomicAdd(&a.combine_count[b * a.KVH + g], 1);
    is_last = prev == n_split - 1;
  }
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  merge_splits<HD>(a, b, g * G, G, reinterpret_cast<float*>(sKV));  // the K/V stages are idle now
  if (threadIdx.x == 0) a.combine_count[b * a.KVH + g] = 0;
}

// f32 path: warp per (request, head); keys walked through the page list.
template <typename Act>
__global__ void k_attn_decode_simt(const DecodeArgs a) {
  pdl_trigger();
  pdl_wait();
  constexpr int MAXD = 8;
  const int b = blockIdx.x;
  const int h = blockIdx.y * 4 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (h >= a.H) return;
  const int hd = a.hd;
  const int g = (h * a.KVH) / a.H;
  const int L = a.seq_len[b];
  const int* pages = a.page_list + a.page_off[b];
  const Act* qp = reinterpret_cast<const Act*>(a.q) + ((long long)b * a.H + h) * hd;
  const Act* kpool = reinterpret_cast<const Act*>(a.k_pool);
  const Act* vpool = reinterpret_cast<const Act*>(a.v_pool);
  float qv[MAXD], ov[MAXD];
#pragma unroll
  for (int i = 0; i < MAXD; ++i) {
    const int d = lane + 32 * i;
    qv[i] = d < hd ? to_f(qp[d]) : 0.f;
    ov[i] = 0.f;
  }
  const float scale = rsqrtf((float)hd);
  float m = -INFINITY, l = 0.f;
  for (int j = 0; j < L; ++j) {
    const long long base =
        ((long long)pages[j / a.page_tokens] * a.page_stride + (long long)g * a.head_stride + j % a.page_tokens) * hd;
    float part = 0.f;
#pragma unroll
    for (int i = 0; i < MAXD; ++i) {
      const int d = lane + 32 * i;
      if (d < hd) part += qv[i] * to_f(kpool[base + d]);
    }
    const float sc = warp_sum(part) * scale;
    const float mn = fmaxf(m, sc);
    const float c = __expf(m - mn);
    const float p = __expf(sc - mn);
    l = l * c + p;
#pragma unroll
    for (int i = 0; i < MAXD; ++i) {
      const int d = lane + 32 * i;
      ov[i] = ov[i] * c + (d < hd ? p * to_f(vpool[base + d]) : 0.f);
    }
    m = mn;
  }
  Act* op = reinterpret_cast<Act*>(a.out) + ((long long)b * a.H + h) * hd;
  const Act* gp = a.gate ? reinterpret_cast<const Act*>(a.gate) + ((long long)b * a.H + h) * hd : nullptr;
#pragma unroll
  for (int i = 0; i < MAXD; ++i) {
    const int d = lane + 32 * i;
    if (d < hd) op[d] = from_f<Act>(ov[i] / l * (gp ? to_f(gp[d]) : 1.f));
  }
}

template <int HD>
cudaError_t launch_decode_tc(const CUtensorMap& k_map, const CUtensorMap& v_map, const DecodeArgs& a,
                             cudaStream_t stream) {
  using C = DecCfg<HD>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_attn_decode_bf16<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  // the split merge stages (3 * splits + 1) floats per query head in the K/V stages
  if ((3LL * a.max_splits + 1) * (a.H / a.KVH) * 4 > (long long)kStages * 2 * C::PAGE_BYTES) return cudaErrorInvalidValue;
  dim3 grid(a.n_work, a.KVH);
  OUTLETS_TRY_LAUNCH(launch_k(k_attn_decode_bf16<HD>, dim3(grid), dim3(128), C::SMEM, stream, k_map, v_map, a));
  return cudaGetLastError();
}

}  // namespace

cudaError_t attn_decode_bf16_launch(const CUtensorMap& k_map, const CUtensorMap& v_map, const DecodeArgs& a,
                                    cudaStream_t stream) {
  if (a.B == 0) return cudaSuccess;
  if (a.H / a.KVH > 16 || a.page_tokens != 64 || a.page_stride < 1 || a.head_stride < 1) return cudaErrorInvalidValue;
  if (a.hd == 128) return launch_decode_tc<128>(k_map, v_map, a, stream);
  if (a.hd == 64) return launch_decode_tc<64>(k_map, v_map, a, stream);
  return cudaErrorInvalidValue;
}

template <typename Act>
cudaError_t attn_decode_simt_launch(const DecodeArgs& a, cudaStream_t stream) {
  if (a.B == 0) return cudaSuccess;
  if (a.hd > 256 || a.page_stride < 1 || a.head_stride < 1) return cudaErrorInvalidValue;
  OUTLETS_TRY_LAUNCH(launch_k(k_attn_decode_simt<Act>, dim3(dim3(a.B, (a.H + 3) / 4)), dim3(128), 0, stream, a));
  return cudaGetLastError();
}
template cudaError_t attn_decode_simt_launch<float>(const DecodeArgs&, cudaStream_t);
template cudaError_t attn_decode_simt_launch<bf16>(const DecodeArgs&, cudaStream_t);

}  // namespace outlets
