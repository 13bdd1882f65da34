// Causal GQA self-attention over a packed varlen batch (the draft decoder's
// self-attention, Sec. 4.1), o = softmax(q k^T / sqrt(hd) + causal mask) v per
// sequence, q-head h reading kv-head floor(h * KVH / H).
//
// This file holds the f32 (CUDA-core) path: one warp per (query row, head),
// lanes own head dims, keys walked in order with an online softmax.  Only the
// small f32 configuration uses it; the bf16 path is the tcgen05 kernel of
// attn_prefill_tc.cu.
#include "common.cuh"
#include "kernels.h"

namespace outlets {
namespace {

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
