// Draft LM head of the dual head (Sec. 4.2, Eq. 2): P_draft = softmax(W_lm h^draft).
//
// The tensor-core GEMM (k_gemm_small with an EPI_LM* epilogue) never writes
// the [rows, V] logits unless asked to; it leaves per (row, N tile) partials:
// the tile's maximum logit m_t, the sum s_t of exp(logit - m_t) over its
// columns, and its best KT (logit, token id) pairs.  This file holds
//   k_lm_merge          one CTA per row: logsumexp = m + log(sum_t s_t exp(m_t - m)),
//                       m = max_t m_t, and the k best tokens of the row (every
//                       token of the row's top-k is in its tile's list, at or
//                       above the row's bound): the list entries that reach the
//                       bound are gathered in shared memory and the k best
//                       taken from there, one at a time;
//   k_lm_tile_stats_f32 the same partials from f32 logits (CUDA-core path).
#include "common.cuh"
#include "kernels.h"
#include "lm_topk.cuh"

namespace outlets {
namespace {

constexpr int kMergeThreads = 256;
constexpr int kMaxTilesPerThread = 16;  // n_tiles <= 4096

// Best (value, id, owner) over the block; every thread gets the result.
__device__ __forceinline__ void block_best(float& v, int& i, float* sv, int* si) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, i, o);
    if (lm_better(ov, oi, v, i)) {
      v = ov;
      i = oi;
    }
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();  // the previous round's readers are done with sv / si
  if (lane == 0) {
    sv[warp] = v;
    si[warp] = i;
  }
  __syncthreads();
  v = sv[0];
  i = si[0];
#pragma unroll
  for (int w = 1; w < kMergeThreads / 32; ++w)
    if (lm_better(sv[w], si[w], v, i)) {
      v = sv[w];
      i = si[w];
    }
}

__device__ __forceinline__ float block_reduce(float v, bool is_max, float* sv) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmaxf(v, ov) : v + ov;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) sv[warp] = v;
  __syncthreads();
  v = sv[0];
#pragma unroll
  for (int w = 1; w < kMergeThreads / 32; ++w) v = is_max ? fmaxf(v, sv[w]) : v + sv[w];
  return v;
}

// Candidates of a row the merge collects in shared memory (beyond this the
// merge takes the k rounds over the tiles' lists in global memory instead).
constexpr int kMergeCap = 2048;

template <int KT>
__global__ void __launch_bounds__(kMergeThreads) k_lm_merge(const float2* __restrict__ stats,
                                                            const int2* __restrict__ top, int n_tiles, int k,
                                                            int* __restrict__ ids, float* __restrict__ logprob,
                                                            float* __restrict__ lse_out, int* __restrict__ bound) {
  __shared__ float sv[kMergeThreads / 32];
  __shared__ int si[kMergeThreads / 32];
  __shared__ float cv[kMergeCap];
  __shared__ int ci[kMergeCap];
  __shared__ int ncand;
  pdl_trigger();
  pdl_wait();
  const int row = blockIdx.x;
  const float2* st = stats + (long long)row * n_tiles;
  const int2* tp = top + (long long)row * n_tiles * KT;
  // logsumexp in one pass: each thread keeps (max, sum relative to it)
  float m = -INFINITY, sm = 0.f;
  for (int t = threadIdx.x; t < n_tiles; t += kMergeThreads) {
    const float2 e = st[t];
    if (e.y == 0.f) continue;  // a partial tile past the vocabulary
    if (e.x > m) {
      sm = sm * exp2f((m - e.x) * kLog2e) + e.y;
      m = e.x;
    } else {
      sm += e.y * exp2f((e.x - m) * kLog2e);
    }
  }
  const float M = block_reduce(m, true, sv);
  const float S = block_reduce(m == -INFINITY ? 0.f : sm * exp2f((m - M) * kLog2e), false, sv);
  const float lse = M + logf(S);

  // The row's bound slots (written by the GEMM epilogue) bound the row's 8th
  // best logit from below, so every token of the top-k is at or above it:
  // collect the tiles' list entries that reach it (the lists are sorted, so a
  // thread stops at the first entry below it), then take the k best of those.
  float thr = -INFINITY;
  if (KT > 1 && bound) {
    int kmin = INT_MAX;
#pragma unroll
    for (int q = 0; q < kLmBoundSlots; ++q) kmin = min(kmin, __ldcg(bound + (long long)row * kLmBoundSlots + q));
    thr = lm_unkey(kmin);
  }
  if (threadIdx.x == 0) ncand = 0;
  __syncthreads();
  if (KT > 1) {
    for (int t = threadIdx.x; t < n_tiles; t += kMergeThreads) {
#pragma unroll 1
      for (int q = 0; q < KT; ++q) {
        const int2 e = tp[(long long)t * KT + q];
        const float v = __int_as_float(e.x);
        if (e.y == INT_MAX || v < thr) break;
        const int pos = atomicAdd(&ncand, 1);
        if (pos < kMergeCap) {
          cv[pos] = v;
          ci[pos] = e.y;
        }
      }
    }
  }
  __syncthreads();
  const int nc = ncand;
  if (KT > 1 && nc <= kMergeCap) {
    for (int r = 0; r < k; ++r) {
      float bv = -INFINITY;
      int bi = INT_MAX, bp = -1;
      for (int c = threadIdx.x; c < nc; c += kMergeThreads)
        if (lm_better(cv[c], ci[c], bv, bi)) {
          bv = cv[c];
          bi = ci[c];
          bp = c;
        }
      const float mv = bv;
      const int mi = bi;
      block_best(bv, bi, sv, si);
      if (bp >= 0 && mi == bi && mv == bv) cv[bp] = -INFINITY, ci[bp] = INT_MAX;  // taken
      if (threadIdx.x == 0) {
        ids[(long long)row * k + r] = bi;
        logprob[(long long)row * k + r] = bv - lse;
      }
    }
  } else {
    // k rounds over the heads of the tiles' sorted lists in global memory
    int head[kMaxTilesPerThread];
#pragma unroll
    for (int j = 0; j < kMaxTilesPerThread; ++j) head[j] = 0;
    for (int r = 0; r < k; ++r) {
      float bv = -INFINITY;
      int bi = INT_MAX, bj = -1;
#pragma unroll
      for (int j = 0; j < kMaxTilesPerThread; ++j) {
        const int t = threadIdx.x + j * kMergeThreads;
        if (t < n_tiles && head[j] < KT) {
          const int2 e = tp[(long long)t * KT + head[j]];
          const float v = __int_as_float(e.x);
          if (lm_better(v, e.y, bv, bi)) {
            bv = v;
            bi = e.y;
            bj = j;
          }
        }
      }
      const float mv = bv;
      const int mi = bi;
      block_best(bv, bi, sv, si);
      // token ids are unique, so exactly one thread owns the winner
      if (bj >= 0 && mi == bi && mv == bv) {
#pragma unroll
        for (int j = 0; j < kMaxTilesPerThread; ++j)
          if (j == bj) ++head[j];
      }
      if (threadIdx.x == 0) {
        ids[(long long)row * k + r] = bi;
        logprob[(long long)row * k + r] = bv - lse;
      }
    }
  }
  if (threadIdx.x == 0 && lse_out) lse_out[row] = lse;
  if (bound && threadIdx.x < kLmBoundSlots)
    bound[(long long)row * kLmBoundSlots + threadIdx.x] = kLmBoundInit;  // ready for the next pass over these rows
}

template <int KT>
__global__ void __launch_bounds__(128) k_lm_tile_stats_f32(const float* __restrict__ logits, long long ld, int rows,
                                                           int V, int tile_w, float2* __restrict__ stats,
                                                           int2* __restrict__ top) {
  pdl_trigger();
  pdl_wait();
  const int n_tiles = (V + tile_w - 1) / tile_w;
  const long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= (long long)rows * n_tiles) return;
  const int row = (int)(u / n_tiles), tile = (int)(u - (long long)row * n_tiles);
  const int c0 = tile * tile_w, c1 = min(V, c0 + tile_w);
  const float* x = logits + (long long)row * ld;
  float m = -INFINITY;
  for (int c = c0; c < c1; ++c) m = fmaxf(m, x[c]);
  float s = 0.f;
  float tv[KT];
  int ti[KT];
  lm_init<KT>(tv, ti);
  for (int c = c0; c < c1; ++c) {
    s += exp2f((x[c] - m) * kLog2e);
    lm_insert<KT>(tv, ti, x[c], c);
  }
  stats[u] = make_float2(m, s);
#pragma unroll
  for (int i = 0; i < KT; ++i) top[u * KT + i] = make_int2(__float_as_int(tv[i]), ti[i]);
}

}  // namespace

cudaError_t lm_merge_launch(const float2* stats, const int2* top, int n_tiles, int kt, int rows, int k, int* ids,
                            float* logprob, float* lse, int* bound, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  if (n_tiles < 1 || n_tiles > kMergeThreads * kMaxTilesPerThread || k < 1 || k > kt) return cudaErrorInvalidValue;
  if (kt == 1)
    return launch_k(k_lm_merge<1>, dim3(rows), dim3(kMergeThreads), 0, stream, stats, top, n_tiles, k, ids, logprob,
                    lse, bound);
  if (kt == 8)
    return launch_k(k_lm_merge<8>, dim3(rows), dim3(kMergeThreads), 0, stream, stats, top, n_tiles, k, ids, logprob,
                    lse, bound);
  return cudaErrorInvalidValue;
}

cudaError_t lm_tile_stats_f32_launch(const float* logits, long long ld, int rows, int V, int tile_w, int kt,
                                     float2* stats, int2* top, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  const long long n = (long long)rows * ((V + tile_w - 1) / tile_w);
  const dim3 grid((unsigned)((n + 127) / 128));
  if (kt == 1) return launch_k(k_lm_tile_stats_f32<1>, grid, dim3(128), 0, stream, logits, ld, rows, V, tile_w, stats, top);
  if (kt == 8) return launch_k(k_lm_tile_stats_f32<8>, grid, dim3(128), 0, stream, logits, ld, rows, V, tile_w, stats, top);
  return cudaErrorInvalidValue;
}

}  // namespace outlets
