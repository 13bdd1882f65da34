// Device helpers of the draft LM head (Eq. 2): running top-k lists of
// (logit, token id) pairs and the softmax statistics of a block of logits.
//
// Order: a larger logit ranks first; equal logits rank by smaller token id.
// This is a total order on (logit, id) pairs, so the top-k of a row does not
// depend on the order in which its pairs are visited (tiles, candidates).
#pragma once

#include <climits>

#include "common.cuh"

namespace outlets {

constexpr float kLog2e = 1.4426950408889634f;

// Order-preserving map between floats and signed ints (for atomicMax on logits).
__device__ __forceinline__ int lm_key(float f) {
  const int i = __float_as_int(f);
  return i >= 0 ? i : i ^ 0x7FFFFFFF;
}
__device__ __forceinline__ float lm_unkey(int k) { return __int_as_float(k >= 0 ? k : k ^ 0x7FFFFFFF); }

__device__ __forceinline__ bool lm_better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

// tv/ti: KT pairs sorted best first.  Inserts (v, i) when it ranks above the
// last entry, shifting the rest down.
template <int KT>
__device__ __forceinline__ void lm_insert(float (&tv)[KT], int (&ti)[KT], float v, int i) {
  if (!lm_better(v, i, tv[KT - 1], ti[KT - 1])) return;
  bool above[KT];
#pragma unroll
  for (int j = 0; j < KT; ++j) above[j] = lm_better(v, i, tv[j], ti[j]);
#pragma unroll
  for (int j = KT - 1; j > 0; --j) {
    // entry j becomes entry j-1 if (v, i) goes above j-1, else (v, i) if it goes above j
    const float nv = above[j - 1] ? tv[j - 1] : (above[j] ? v : tv[j]);
    const int ni = above[j - 1] ? ti[j - 1] : (above[j] ? i : ti[j]);
    tv[j] = nv;
    ti[j] = ni;
  }
  if (above[0]) {
    tv[0] = v;
    ti[0] = i;
  }
}

template <int KT>
__device__ __forceinline__ void lm_init(float (&tv)[KT], int (&ti)[KT]) {
#pragma unroll
  for (int j = 0; j < KT; ++j) {
    tv[j] = -INFINITY;
    ti[j] = INT_MAX;
  }
}

}  // namespace outlets
