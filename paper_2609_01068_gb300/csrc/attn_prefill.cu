// Causal GQA self-attention over a packed varlen batch (the draft decoder's
// self-attention, Sec. 4.1), o = softmax(q k^T / sqrt(hd) + causal mask) v per
// sequence, q-head h reading kv-head floor(h * KVH / H).
//
// bf16 path: flash attention with online softmax in f32.  One CTA = one
// 64-row query tile of one sequence x one query head; 4 warps x 16 rows.
// Q, K and V tiles are staged into shared memory by TMA (128-byte swizzle,
// two K/V stages); QK^T and PV run on mma.sync m16n8k16.  K/V are head-major
// [KVH, T, hd] so one kv-head's keys of a sequence are contiguous rows.
//
// f32 path: one warp per (query row, head), lanes own head dims, keys walked
// in order with an online softmax.  Only the small f32 configuration uses it.
#include "common.cuh"
#include "kernels.h"
#include "mma_sync.cuh"

namespace outlets {
namespace {

constexpr float kLog2e = 1.4426950408889634f;

template <int HD>
struct PrefillCfg {
  static constexpr int TILE_BYTES = 64 * HD * 2;
  static constexpr size_t SMEM = 1024 + 5 * TILE_BYTES + 64;
};

template <int HD>
__global__ void __launch_bounds__(128)
    k_attn_prefill_bf16(const __grid_constant__ CUtensorMap q_map, const __grid_constant__ CUtensorMap k_map,
                        const __grid_constant__ CUtensorMap v_map, const AttnTile* __restrict__ tiles, int T,
                        int H, int KVH, bf16* __restrict__ out, const bf16* __restrict__ gate, int* err) {
  pdl_trigger();
  pdl_wait();
  using C = PrefillCfg<HD>;
  constexpr int NB = HD / 64;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = smem + C::TILE_BYTES;
  uint8_t* sV = sK + 2 * C::TILE_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + 2 * C::TILE_BYTES);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;
  uint64_t* kv_empty = bars + 3;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 5);

  const int h = blockIdx.x;
  const AttnTile tile = tiles[blockIdx.y];
  const int g = (h * KVH) / H;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int seq_end = tile.seq_start + tile.seq_len;
  const int n_kt = (tile.q_start + tile.q_len - tile.seq_start + 63) / 64;
  const int kv_row0 = g * T + tile.seq_start;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 4);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  auto issue_kv = [&](int kt, int stage) {
    mbar_arrive_expect_tx(&kv_full[stage], 2 * C::TILE_BYTES);
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      tma_load_2d(sK + stage * C::TILE_BYTES + b * 8192, &k_map, &kv_full[stage], b * 64, kv_row0 + kt * 64);
      tma_load_2d(sV + stage * C::TILE_BYTES + b * 8192, &v_map, &kv_full[stage], b * 64, kv_row0 + kt * 64);
    }
  };

  if (threadIdx.x == 0) {
    mbar_arrive_expect_tx(q_full, C::TILE_BYTES);
#pragma unroll
    for (int b = 0; b < NB; ++b) tma_load_2d(sQ + b * 8192, &q_map, q_full, h * HD + b * 64, tile.q_start);
    for (int s = 0; s < 2 && s < n_kt; ++s) issue_kv(s, s);
  }

  bool ok = mbar_wait(q_full, 0, abort_flag, err);

  // Q fragments of this warp's 16 rows
  uint32_t qf[HD / 16][4];
  {
    const uint32_t qbase = smem_u32(sQ);
    const int r = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
      const int d = ks * 16 + ((lane >> 4) & 1) * 8;
      ldsm_x4(qbase + sw128_offset<64>(r, d), qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3]);
    }
  }

  float o[HD / 8][4];
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  const int row0 = tile.q_start + warp * 16 + (lane >> 2);
  const int row1 = row0 + 8;
  const int r0e = min(row0, seq_end - 1);
  const int r1e = min(row1, seq_end - 1);
  const float sl2 = rsqrtf((float)HD) * kLog2e;

  for (int kt = 0; kt < n_kt && ok; ++kt) {
    const int stage = kt & 1;
    if (!mbar_wait(&kv_full[stage], (kt >> 1) & 1, abort_flag, err)) {
      ok = false;
      break;
    }
    const uint32_t kbase = smem_u32(sK + stage * C::TILE_BYTES);
    const uint32_t vbase = smem_u32(sV + stage * C::TILE_BYTES);
    const int key0 = tile.seq_start + kt * 64;

    float s[8][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t b0, b1, b2, b3;
        const int key = np * 16 + (lane & 7) + ((lane >> 4) & 1) * 8;
        const int d = ks * 16 + ((lane >> 3) & 1) * 8;
        ldsm_x4(kbase + sw128_offset<64>(key, d), b0, b1, b2, b3);
        mma_16816(s[2 * np], qf[ks], b0, b1);
        mma_16816(s[2 * np + 1], qf[ks], b2, b3);
      }
    }

    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int kc = key0 + 8 * j + 2 * (lane & 3);
      s[j][0] = (kc <= r0e) ? s[j][0] * sl2 : -INFINITY;
      s[j][1] = (kc + 1 <= r0e) ? s[j][1] * sl2 : -INFINITY;
      s[j][2] = (kc <= r1e) ? s[j][2] * sl2 : -INFINITY;
      s[j][3] = (kc + 1 <= r1e) ? s[j][3] * sl2 : -INFINITY;
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
    for (int j = 0; j < 8; ++j) {
      s[j][0] = exp2f(s[j][0] - mu0);
      s[j][1] = exp2f(s[j][1] - mu0);
      s[j][2] = exp2f(s[j][2] - mu1);
      s[j][3] = exp2f(s[j][3] - mu1);
      ps0 += s[j][0] + s[j][1];
      ps1 += s[j][2] + s[j][3];
    }
    l0 = l0 * c0 + ps0;
    l1 = l1 * c1 + ps1;
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) {
      o[j][0] *= c0;
      o[j][1] *= c0;
      o[j][2] *= c1;
      o[j][3] *= c1;
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t a[4];
      a[0] = pack_bf16x2(s[2 * kk][0], s[2 * kk][1]);
      a[1] = pack_bf16x2(s[2 * kk][2], s[2 * kk][3]);
      a[2] = pack_bf16x2(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      a[3] = pack_bf16x2(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int dp = 0; dp < HD / 16; ++dp) {
        uint32_t b0, b1, b2, b3;
        const int key = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int d = dp * 16 + ((lane >> 4) & 1) * 8;
        ldsm_x4_t(vbase + sw128_offset<64>(key, d), b0, b1, b2, b3);
        mma_16816(o[2 * dp], a, b0, b1);
        mma_16816(o[2 * dp + 1], a, b2, b3);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&kv_empty[stage]);
    if (threadIdx.x == 0 && kt + 2 < n_kt) {
      if (!mbar_wait(&kv_empty[stage], (kt >> 1) & 1, abort_flag, err)) {
        ok = false;
        break;
      }
      issue_kv(kt + 2, stage);
    }
  }

  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  if (!ok) return;
  const float inv0 = 1.f / l0;
  const float inv1 = 1.f / l1;
  const int q_end = tile.q_start + tile.q_len;
  const long long ld = (long long)H * HD;
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) {
    const int d = h * HD + 8 * j + 2 * (lane & 3);
    if (row0 < q_end) {
      float2 gv = make_float2(1.f, 1.f);  // gated attention: elementwise output gate
      if (gate) gv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(gate + row0 * ld + d));
      *reinterpret_cast<uint32_t*>(out + row0 * ld + d) = pack_bf16x2(o[j][0] * inv0 * gv.x, o[j][1] * inv0 * gv.y);
    }
    if (row1 < q_end) {
      float2 gv = make_float2(1.f, 1.f);
      if (gate) gv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(gate + row1 * ld + d));
      *reinterpret_cast<uint32_t*>(out + row1 * ld + d) = pack_bf16x2(o[j][2] * inv1 * gv.x, o[j][3] * inv1 * gv.y);
    }
  }
}

// ---------------------------------------------------------------- plain warp-per-row path
template <typename Act, int MAXD>
__device__ __forceinline__ void load_dims(const Act* p, int hd, int lane, float* v) {
#pragma unroll
  for (int i = 0; i < MAXD; ++i) {
    const int d = lane + 32 * i;
    v[i] = d < hd ? to_f(p[d]) : 0.f;
  }
}

template <typename Act>
__global__ void k_attn_prefill_simt(const Act* __restrict__ q, const Act* __restrict__ k,
                                    const Act* __restrict__ v, const int* __restrict__ cu, int B, int kv_ld, int H,
                                    int KVH, int hd, Act* __restrict__ out, const Act* __restrict__ gate) {
  pdl_trigger();
  pdl_wait();
  constexpr int MAXD = 8;  // hd <= 256
  const int row = blockIdx.x;
  const int h = blockIdx.y * 4 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (h >= H) return;
  int lo = 0, hi = B;  // sequence of this row: cu[b] <= row < cu[b+1]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (cu[mid] <= row) lo = mid;
    else hi = mid;
  }
  const int s0 = cu[lo];
  const int g = (h * KVH) / H;
  const float scale = rsqrtf((float)hd);
  float qv[MAXD], ov[MAXD];
  load_dims<Act, MAXD>(q + ((long long)row * H + h) * hd, hd, lane, qv);
#pragma unroll
  for (int i = 0; i < MAXD; ++i) ov[i] = 0.f;
  float m = -INFINITY, l = 0.f;
  for (int j = s0; j <= row; ++j) {
    const Act* kp = k + ((long long)g * kv_ld + j) * hd;
    const Act* vp = v + ((long long)g * kv_ld + j) * hd;
    float part = 0.f;
#pragma unroll
    for (int i = 0; i < MAXD; ++i) {
      const int d = lane + 32 * i;
      if (d < hd) part += qv[i] * to_f(kp[d]);
    }
    const float sc = warp_sum(part) * scale;
    const float mn = fmaxf(m, sc);
    const float c = __expf(m - mn);
    const float p = __expf(sc - mn);
    l = l * c + p;
#pragma unroll
    for (int i = 0; i < MAXD; ++i) {
      const int d = lane + 32 * i;
      ov[i] = ov[i] * c + (d < hd ? p * to_f(vp[d]) : 0.f);
    }
    m = mn;
  }
  Act* op = out + ((long long)row * H + h) * hd;
  const Act* gp = gate ? gate + ((long long)row * H + h) * hd : nullptr;
#pragma unroll
  for (int i = 0; i < MAXD; ++i) {
    const int d = lane + 32 * i;
    if (d < hd) op[d] = from_f<Act>(ov[i] / l * (gp ? to_f(gp[d]) : 1.f));
  }
}

}  // namespace

cudaError_t attn_prefill_bf16_launch(const CUtensorMap& q_map, const CUtensorMap& k_map, const CUtensorMap& v_map,
                                     const AttnTile* tiles, int n_tiles, int T, int H, int KVH, int hd, void* out,
                                     const void* gate, int* err, cudaStream_t stream) {
  if (n_tiles == 0) return cudaSuccess;
  if (hd == 128) {
    using C = PrefillCfg<128>;
    static bool attr = false;
    if (!attr) {
      cudaError_t e = cudaFuncSetAttribute(k_attn_prefill_bf16<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)C::SMEM);
      if (e != cudaSuccess) return e;
      attr = true;
    }
    dim3 grid(H, n_tiles);
    OUTLETS_TRY_LAUNCH(launch_k(k_attn_prefill_bf16<128>, dim3(grid), dim3(128), C::SMEM, stream, q_map, k_map, v_map, tiles, T, H, KVH,
                                                             reinterpret_cast<bf16*>(out), reinterpret_cast<const bf16*>(gate), err));
    return cudaGetLastError();
  }
  if (hd == 64) {
    using C = PrefillCfg<64>;
    static bool attr = false;
    if (!attr) {
      cudaError_t e = cudaFuncSetAttribute(k_attn_prefill_bf16<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)C::SMEM);
      if (e != cudaSuccess) return e;
      attr = true;
    }
    dim3 grid(H, n_tiles);
    OUTLETS_TRY_LAUNCH(launch_k(k_attn_prefill_bf16<64>, dim3(grid), dim3(128), C::SMEM, stream, q_map, k_map, v_map, tiles, T, H, KVH,
                                                            reinterpret_cast<bf16*>(out), reinterpret_cast<const bf16*>(gate), err));
    return cudaGetLastError();
  }
  return cudaErrorInvalidValue;
}

template <typename Act>
cudaError_t attn_prefill_simt_launch(const Act* q, const Act* k, const Act* v, const int* cu, int B, int n_rows,
                                     int kv_ld, int H, int KVH, int hd, Act* out, const Act* gate,
                                     cudaStream_t stream) {
  if (n_rows == 0) return cudaSuccess;
  if (hd > 256) return cudaErrorInvalidValue;
  dim3 grid(n_rows, (H + 3) / 4);
  OUTLETS_TRY_LAUNCH(launch_k(k_attn_prefill_simt<Act>, dim3(grid), dim3(128), 0, stream, q, k, v, cu, B, kv_ld, H, KVH, hd, out, gate));
  return cudaGetLastError();
}

template cudaError_t attn_prefill_simt_launch<float>(const float*, const float*, const float*, const int*, int,
                                                     int, int, int, int, int, float*, const float*, cudaStream_t);
template cudaError_t attn_prefill_simt_launch<bf16>(const bf16*, const bf16*, const bf16*, const int*, int, int,
                                                    int, int, int, int, bf16*, const bf16*, cudaStream_t);

}  // namespace outlets
