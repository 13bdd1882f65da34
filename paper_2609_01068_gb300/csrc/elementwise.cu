// Row-wise and elementwise kernels of the draft layer and the length head,
// plus the plain CUDA-core GEMM of the f32 configuration.
//
//   RMSNorm           x * g / sqrt(mean(x^2) + eps) (pre-norm reading of the
//                     decoder layer of Sec. 4.1; also the final norm that
//                     yields h^draft for the heads of Sec. 4.2)
//   RoPE + scatter    rotate pairs (i, i + hd/2) of q and k by pos * theta^(-2i/hd)
//                     (table built in fp64 on the host), write q, head-major
//                     k/v for prefill attention, and k/v into the paged cache
//   SwiGLU            silu(gate) * up (the decoder layer's MLP block)
//   head tail         z_hat = w . relu(h + b) + b_out, length = max(0, expm1(z_hat))
//                     (Sec. 4.2: log-space target z = log(1 + length))
#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "kernels.h"

namespace outlets {
namespace {

__device__ __forceinline__ float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  const int nw = blockDim.x >> 5;
  float t = (threadIdx.x < nw) ? red[threadIdx.x] : 0.f;
  if (warp == 0) t = warp_sum(t);
  if (threadIdx.x == 0) red[32] = t;
  __syncthreads();
  return red[32];
}

// Split-K slices: s[0] + s[1] + ... + s[n-1] at p, p + stride, ..., added in
// slice order (the same order on every call); the loads of up to U + 1 slices
// are in flight together.
__device__ __forceinline__ void add4(float4& a, const float4& b) {
  a.x += b.x;
  a.y += b.y;
  a.z += b.z;
  a.w += b.w;
}
template <int U = 8>
__device__ __forceinline__ float4 ld_sum4(const float* p, int n, long long stride) {
  float4 acc = *reinterpret_cast<const float4*>(p);
  for (int s0 = 1; s0 < n; s0 += U) {
    float4 v[U];
#pragma unroll
    for (int k = 0; k < U; ++k)
      if (s0 + k < n) v[k] = *reinterpret_cast<const float4*>(p + (s0 + k) * stride);
#pragma unroll
    for (int k = 0; k < U; ++k)
      if (s0 + k < n) add4(acc, v[k]);
  }
  return acc;
}
// Two float4 runs (8 floats at p and 8 at q) summed over the slices; up to
// three slices of both in flight together.
__device__ __forceinline__ void ld_sum16(const float* p, const float* q, int n, long long stride, float4 (&o)[4]) {
  o[0] = *reinterpret_cast<const float4*>(p);
  o[1] = *reinterpret_cast<const float4*>(p + 4);
  o[2] = *reinterpret_cast<const float4*>(q);
  o[3] = *reinterpret_cast<const float4*>(q + 4);
  for (int s0 = 1; s0 < n; s0 += 2) {
    float4 v[2][4];
#pragma unroll
    for (int k = 0; k < 2; ++k)
      if (s0 + k < n) {
        const long long off = (s0 + k) * stride;
        v[k][0] = *reinterpret_cast<const float4*>(p + off);
        v[k][1] = *reinterpret_cast<const float4*>(p + off + 4);
        v[k][2] = *reinterpret_cast<const float4*>(q + off);
        v[k][3] = *reinterpret_cast<const float4*>(q + off + 4);
      }
#pragma unroll
    for (int k = 0; k < 2; ++k)
      if (s0 + k < n) {
#pragma unroll
        for (int j = 0; j < 4; ++j) add4(o[j], v[k][j]);
      }
  }
}

// Drops row `row` (ld floats) of every split-K slice from L2 once the block has
// read it: the slices are scratch, rewritten before they are read again, and
// their dirty lines would otherwise be written back to DRAM when evicted (in
// the step, largely while the attention stage streams the K/V cache).  The
// caller has passed a __syncthreads after its last read of the slices.  Only
// whole, aligned 128-byte lines: nothing is done unless ld, the slice stride
// and the base are multiples of 32 floats.
__device__ __forceinline__ void discard_slice_rows(const float* x, int n_split, long long stride, long long row,
                                                   int ld) {
  if ((ld & 31) || (stride & 31) || (reinterpret_cast<uintptr_t>(x) & 127)) return;
  const int lines = ld >> 5;
  const float* r0 = x + row * ld;
  for (int t = threadIdx.x; t < n_split * lines; t += blockDim.x) {
    const int s = t / lines;
    discard_l2_line(r0 + s * stride + (long long)(t - s * lines) * 32);
  }
}

template <typename Act>
__device__ __forceinline__ void store4(Act* p, float a, float b, float c, float d);
template <>
__device__ __forceinline__ void store4<float>(float* p, float a, float b, float c, float d) {
  *reinterpret_cast<float4*>(p) = make_float4(a, b, c, d);
}
template <>
__device__ __forceinline__ void store4<bf16>(bf16* p, float a, float b, float c, float d) {
  uint2 v;
  v.x = pack_bf16x2(a, b);
  v.y = pack_bf16x2(c, d);
  *reinterpret_cast<uint2*>(p) = v;
}

// v = (sum_s x[s][src]) + residual[src] (split-K slices of the producing GEMM, in slice order);
// y[r] = v * g * rsqrt(mean(v^2) + eps); copy_out[r] = v (f32) when given.
// REDUCE = false: v = x[src] (one slice, no residual).
template <typename Act, bool REDUCE>
__global__ void __launch_bounds__(512, 2) k_rmsnorm(const float* __restrict__ x, int n_split, long long split_stride,
                          const float* __restrict__ residual, const int* __restrict__ row_index,
                          const float* __restrict__ g, Act* __restrict__ y, float* __restrict__ copy_out, int d,
                          float eps, bool discard) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[33];
  extern __shared__ float4 rowbuf[];  // the reduced row (REDUCE only)
  const int r = blockIdx.x;
  const long long src = row_index ? row_index[r] : r;
  float ss = 0.f;
  for (int i = threadIdx.x * 4; i < d; i += blockDim.x * 4) {
    float4 v;
    if constexpr (REDUCE) {
      v = ld_sum4(x + src * d + i, n_split, split_stride);
      if (residual) add4(v, *reinterpret_cast<const float4*>(residual + src * d + i));
      rowbuf[i >> 2] = v;
    } else {
      v = *reinterpret_cast<const float4*>(x + src * d + i);
    }
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)d + eps);  // every slice read of the block is done
  if constexpr (REDUCE)
    if (discard && !row_index) discard_slice_rows(x, n_split, split_stride, r, d);
  Act* yr = y + (long long)r * d;
  for (int i = threadIdx.x * 4; i < d; i += blockDim.x * 4) {
    float4 v;
    if constexpr (REDUCE) v = rowbuf[i >> 2];
    else v = *reinterpret_cast<const float4*>(x + src * d + i);
    const float4 gg = *reinterpret_cast<const float4*>(g + i);
    store4<Act>(yr + i, v.x * inv * gg.x, v.y * inv * gg.y, v.z * inv * gg.z, v.w * inv * gg.w);
    if (copy_out) *reinterpret_cast<float4*>(copy_out + (long long)r * d + i) = v;
  }
}

// 8 consecutive elements of a row as f32, summed over n_split slices.
template <typename In>
__device__ __forceinline__ void load8(const In* p, long long idx, int n_split, long long stride, float* v);
template <>
__device__ __forceinline__ void load8<bf16>(const bf16* p, long long idx, int, long long, float* v) {
  const uint4 u = *reinterpret_cast<const uint4*>(p + idx);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float2 f = __bfloat1622float2(h[k]);
    v[2 * k] = f.x;
    v[2 * k + 1] = f.y;
  }
}
template <>
__device__ __forceinline__ void load8<float>(const float* p, long long idx, int n_split, long long stride,
                                             float* v) {
  const float4 a = ld_sum4<4>(p + idx, n_split, stride);
  const float4 b = ld_sum4<4>(p + idx + 4, n_split, stride);
  v[0] = a.x, v[1] = a.y, v[2] = a.z, v[3] = a.w, v[4] = b.x, v[5] = b.y, v[6] = b.z, v[7] = b.w;
}
// Both halves of a rotation pair (8 elements at idx and at idx + half).
template <typename In>
__device__ __forceinline__ void load8x2(const In* p, long long idx, long long half, int n_split, long long stride,
                                        float* v1, float* v2) {
  load8<In>(p, idx, n_split, stride, v1);
  load8<In>(p, idx + half, n_split, stride, v2);
}
template <>
__device__ __forceinline__ void load8x2<float>(const float* p, long long idx, long long half, int n_split,
                                               long long stride, float* v1, float* v2) {
  float4 o[4];
  ld_sum16(p + idx, p + idx + half, n_split, stride, o);
  v1[0] = o[0].x, v1[1] = o[0].y, v1[2] = o[0].z, v1[3] = o[0].w;
  v1[4] = o[1].x, v1[5] = o[1].y, v1[6] = o[1].z, v1[7] = o[1].w;
  v2[0] = o[2].x, v2[1] = o[2].y, v2[2] = o[2].z, v2[3] = o[2].w;
  v2[4] = o[3].x, v2[5] = o[3].y, v2[6] = o[3].z, v2[7] = o[3].w;
}

template <typename Act>
__device__ __forceinline__ void store8(Act* p, const float* v);
template <>
__device__ __forceinline__ void store8<bf16>(bf16* p, const float* v) {
  uint4 u;
  u.x = pack_bf16x2(v[0], v[1]);
  u.y = pack_bf16x2(v[2], v[3]);
  u.z = pack_bf16x2(v[4], v[5]);
  u.w = pack_bf16x2(v[6], v[7]);
  *reinterpret_cast<uint4*>(p) = u;
}
template <>
__device__ __forceinline__ void store8<float>(float* p, const float* v) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
}

// Input-embedding branch (EAGLE-3-style layer input): y[r] = RMSNorm(E[tok[r]]) * g,
// one CTA per row, 8 elements per thread step (d is a multiple of 64).  A token
// outside [0, V) raises ERR_BAD_INDEX and reads row 0 instead.
template <typename Act>
__global__ void __launch_bounds__(256) k_embed_rmsnorm(const int* __restrict__ tok, const Act* __restrict__ E, int V,
                                                       const float* __restrict__ g, Act* __restrict__ y, int d,
                                                       float eps, int* __restrict__ err) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[33];
  const int r = blockIdx.x;
  int t = tok[r];
  if (t < 0 || t >= V) {
    if (threadIdx.x == 0) atomicOr(err, ERR_BAD_INDEX);
    t = 0;
  }
  const long long base = (long long)t * d;
  float ss = 0.f;
  for (int i = threadIdx.x * 8; i < d; i += blockDim.x * 8) {
    float v[8];
    load8<Act>(E, base + i, 1, 0, v);
#pragma unroll
    for (int k = 0; k < 8; ++k) ss += v[k] * v[k];
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)d + eps);
  for (int i = threadIdx.x * 8; i < d; i += blockDim.x * 8) {
    float v[8];
    load8<Act>(E, base + i, 1, 0, v);
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] *= inv * g[i + k];
    store8<Act>(y + (long long)r * d + i, v);
  }
}

// One CTA per row; a thread rotates 8 pairs (i..i+7 with i+hd/2..i+hd/2+7) of
// one head and copies 8 values of V.  hd is a multiple of 16.
// Block shape of the RoPE/scatter kernel.  f32 input (split-K slices, small
// batches): one rotation chunk per thread, two CTAs (rows) per SM.  bf16 input
// (prefill, one CTA per token over ~T rows): small CTAs, many per SM.
template <typename In>
struct RopeBlock {
  static constexpr int kThreads = std::is_same<In, float>::value ? 320 : 128;
  static constexpr int kMinBlocks = std::is_same<In, float>::value ? 2 : 10;  // bf16: 51 registers, no spills
};

template <typename In, typename Act>
__global__ void __launch_bounds__(RopeBlock<In>::kThreads, RopeBlock<In>::kMinBlocks) k_rope_scatter(const In* __restrict__ qkv, const RopeArgs a) {
  pdl_trigger();
  pdl_wait();
  const int row = a.row0 + (int)blockIdx.x;
  int pos, seq;
  if (a.cu) {
    int lo = 0, hi = a.B;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (a.cu[mid] <= row) lo = mid;
      else hi = mid;
    }
    seq = lo;
    pos = row - a.cu[lo];
  } else {
    seq = row;
    pos = a.pos[row];
  }
  if (pos < 0 || pos >= a.max_pos) {
    if (threadIdx.x == 0) atomicOr(a.err, ERR_BAD_INDEX);
    pos = 0;
  }
  const int hd = a.hd, half = hd / 2, H = a.H, KVH = a.KVH;
  const long long W = a.qkv_ld;
  const In* src = qkv + (long long)row * W;
  const float* cs = a.cos_tab + (long long)pos * half;
  const float* sn = a.sin_tab + (long long)pos * half;
  Act* q_out = reinterpret_cast<Act*>(a.q_out);
  Act* k_out = reinterpret_cast<Act*>(a.k_out);
  Act* v_out = reinterpret_cast<Act*>(a.v_out);
  Act* k_pool = reinterpret_cast<Act*>(a.k_pool);
  Act* v_pool = reinterpret_cast<Act*>(a.v_pool);
  long long cache_base = -1;
  if (k_pool) {
    const int page = a.page_list[a.page_off[seq] + pos / a.page_tokens];
    cache_base = ((long long)page * KVH) * a.page_tokens + pos % a.page_tokens;
  }
  const int cpr = half / 8;  // 8-element chunks per half head
  for (int idx = (q_out ? 0 : H * cpr) + threadIdx.x; idx < (H + KVH) * cpr; idx += blockDim.x) {
    const int head = idx / cpr;
    const int i = (idx - head * cpr) * 8;
    float x1[8], x2[8], y1[8], y2[8];
    load8x2<In>(src, head * hd + i, half, a.n_split, a.split_stride, x1, x2);
    const float4 c0 = *reinterpret_cast<const float4*>(cs + i);
    const float4 c1 = *reinterpret_cast<const float4*>(cs + i + 4);
    const float4 s0 = *reinterpret_cast<const float4*>(sn + i);
    const float4 s1 = *reinterpret_cast<const float4*>(sn + i + 4);
    const float c[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
    const float sv[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      y1[k] = x1[k] * c[k] - x2[k] * sv[k];
      y2[k] = x2[k] * c[k] + x1[k] * sv[k];
    }
    if (head < H) {
      Act* qo = q_out + ((long long)row * H + head) * hd;
      store8<Act>(qo + i, y1);
      store8<Act>(qo + i + half, y2);
    } else {
      const int kh = head - H;
      if (k_out) {
        Act* ko = k_out + ((long long)kh * a.kv_ld_rows + row) * hd;
        store8<Act>(ko + i, y1);
        store8<Act>(ko + i + half, y2);
      }
      if (k_pool) {
        Act* kc = k_pool + (cache_base + (long long)kh * a.page_tokens) * hd;
        store8<Act>(kc + i, y1);
        store8<Act>(kc + i + half, y2);
      }
    }
  }
  const long long voff = (long long)(H + KVH) * hd;
  for (int idx = threadIdx.x; idx < KVH * hd / 8; idx += blockDim.x) {
    const int e = idx * 8;
    const int kh = e / hd;
    const int dd = e - kh * hd;
    float v[8];
    load8<In>(src, voff + e, a.n_split, a.split_stride, v);
    if (v_out) store8<Act>(v_out + ((long long)kh * a.kv_ld_rows + row) * hd + dd, v);
    if (v_pool) store8<Act>(v_pool + (cache_base + (long long)kh * a.page_tokens) * hd + dd, v);
  }
  if (a.gate_out) {
    // gated attention (Sec. 4.1): the gate columns follow q, k, v in the qkv
    // row; the attention kernels multiply their output by sigmoid(gate)
    const long long goff = (long long)(H + 2 * KVH) * hd;
    Act* go = reinterpret_cast<Act*>(a.gate_out) + (long long)row * H * hd;
    for (int idx = threadIdx.x; idx < H * hd / 8; idx += blockDim.x) {
      float g[8];
      load8<In>(src, goff + idx * 8, a.n_split, a.split_stride, g);
#pragma unroll
      for (int k = 0; k < 8; ++k) g[k] = 1.f / (1.f + __expf(-g[k]));
      store8<Act>(go + idx * 8, g);
    }
  }
  if constexpr (std::is_same<In, float>::value) {
    if (a.discard) {  // block-uniform
      __syncthreads();  // every slice read of the block is done
      discard_slice_rows(qkv, a.n_split, a.split_stride, row, a.qkv_ld);
    }
  }
}

// dst[r] = src[idx[r]], 16 bytes per thread step.
__global__ void __launch_bounds__(256) k_gather_rows(const uint4* __restrict__ src, const int* __restrict__ idx,
                                                     uint4* __restrict__ dst, int rows, long long row_vec) {
  pdl_trigger();
  pdl_wait();
  const long long n = (long long)rows * row_vec;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
    const long long r = i / row_vec, c = i - r * row_vec;
    dst[i] = src[(long long)idx[r] * row_vec + c];
  }
}

template <typename Act>
__global__ void k_swiglu(const float* __restrict__ gu, Act* __restrict__ u, int rows, int f_pad) {
  pdl_trigger();
  pdl_wait();
  const long long n = (long long)rows * f_pad;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < n;
       idx += (long long)gridDim.x * blockDim.x) {
    const long long r = idx / f_pad;
    const int j = (int)(idx - r * f_pad);
    const float* row = gu + r * 2 * f_pad + (j >> 5) * 64 + (j & 31);
    const float gt = row[0], up = row[32];
    u[idx] = from_f<Act>(gt / (1.f + __expf(-gt)) * up);
  }
}

// One CTA per row: h = sum of slices, a = relu(h + b_prev), z = w_last . a + b_last.
__global__ void __launch_bounds__(512) k_head_tail(const float* __restrict__ h, int n_split, long long split_stride,
                            const float* __restrict__ b_prev, const float* __restrict__ w_last,
                            const float* __restrict__ b_last, int rows, int width, float* __restrict__ z,
                            float* __restrict__ len, bool discard) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[33];
  const int r = blockIdx.x;
  const float* hr = h + (long long)r * width;
  float acc = 0.f;
  if ((width & 3) == 0) {
    for (int j = threadIdx.x * 4; j < width; j += blockDim.x * 4) {
      float4 x = ld_sum4(hr + j, n_split, split_stride);
      if (b_prev) {
        const float4 b = *reinterpret_cast<const float4*>(b_prev + j);
        x = make_float4(fmaxf(x.x + b.x, 0.f), fmaxf(x.y + b.y, 0.f), fmaxf(x.z + b.z, 0.f), fmaxf(x.w + b.w, 0.f));
      }
      const float4 wl = *reinterpret_cast<const float4*>(w_last + j);
      acc += wl.x * x.x + wl.y * x.y + wl.z * x.z + wl.w * x.w;
    }
  } else {
    for (int j = threadIdx.x; j < width; j += blockDim.x) {
      float x = hr[j];
      for (int sp = 1; sp < n_split; ++sp) x += hr[sp * split_stride + j];
      if (b_prev) x = fmaxf(x + b_prev[j], 0.f);
      acc += w_last[j] * x;
    }
  }
  acc = block_sum(acc, red);  // every slice read of the block is done
  if (discard) discard_slice_rows(h, n_split, split_stride, r, width);
  if (threadIdx.x == 0) {
    const float zz = acc + b_last[0];
    z[r] = zz;
    if (len) len[r] = fmaxf(0.f, expm1f(zz));
  }
}

template <typename Act>
__global__ void k_convert_rows(const float* __restrict__ src, Act* __restrict__ dst, int rows, int cols,
                               long long dst_ld, int row_mode, int row_base, long long kb_np,
                               const float* __restrict__ col_scale) {
  const long long n = (long long)rows * cols;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < n;
       idx += (long long)gridDim.x * blockDim.x) {
    const int r = (int)(idx / cols);
    const int c = (int)(idx - (long long)r * cols);
    const int rg = row_base + r;
    long long dr;
    if (row_mode == 0) dr = rg;
    else if (row_mode == 1) dr = (rg >> 5) * 64 + (rg & 31);        // gate rows of an interleaved [gate 32 | up 32] block
    else dr = (rg >> 5) * 64 + 32 + (rg & 31);                      // up rows
    long long o;
    if (kb_np > 0) {
      const int cc = c & 63;
      o = ((long long)(c >> 6) * kb_np + dr) * 64 + ((((cc >> 3) ^ (int)(dr & 7)) << 3) | (cc & 7));
    } else {
      o = dr * dst_ld + c;
    }
    dst[o] = from_f<Act>(col_scale ? src[idx] * col_scale[c] : src[idx]);
  }
}

// ---------------------------------------------------------------- f32 GEMM (CUDA cores)
constexpr int ST = 64, SK = 16;

__global__ void __launch_bounds__(256) k_gemm_simt(const float* __restrict__ a0, const float* __restrict__ a1,
                                                   const float* __restrict__ a2, const float* __restrict__ bm,
                                                   int epi, const GemmArgs p) {
  pdl_trigger();
  pdl_wait();
  __shared__ float As[SK][ST + 1];
  __shared__ float Bs[SK][ST + 1];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int m0 = blockIdx.y * ST, n0 = blockIdx.x * ST;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < p.K; k0 += SK) {
    for (int i = threadIdx.x; i < ST * SK; i += 256) {
      const int r = i / SK, kk = i % SK;
      const int m = m0 + r, n = n0 + r, k = k0 + kk;
      float av = 0.f, bv = 0.f;
      if (m < p.M && k < p.K) {
        const int piece = k / p.k_per_map;
        const float* ap = piece == 0 ? a0 : (piece == 1 ? a1 : a2);
        av = ap[(long long)m * p.k_per_map + (k - piece * p.k_per_map)];
      }
      if (n < p.N && k < p.K) bv = bm[(long long)n * p.K + k];
      As[kk][r] = av;
      Bs[kk][r] = bv;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < SK; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] += av[i] * bv[j];
    }
    __syncthreads();
  }
  float* out = reinterpret_cast<float*>(p.out);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= p.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= p.N) continue;
      float v = acc[i][j];
      if (epi == EPI_F32 && p.residual) v += p.residual[(long long)m * p.ldr + n];
      if (epi == EPI_BIAS_RELU) v = fmaxf(v + p.bias[n], 0.f);
      out[(long long)m * p.ldo + n] = v;
    }
  }
}

// A wait that nothing completes: the bounded-wait path every pipeline uses
// (mbar_wait) gives up after timeout_ns and raises ERR_TIMEOUT.
__global__ void k_wait_selftest(int* err, unsigned long long timeout_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(&bar, 0, &abort_flag, err, timeout_ns);
  __syncthreads();
}

inline int grid_for(long long n, int threads) {
  long long g = (n + threads - 1) / threads;
  if (g > 152LL * 32) g = 152LL * 32;
  return (int)(g < 1 ? 1 : g);
}

}  // namespace

template <typename Act>
cudaError_t rmsnorm_launch(const float* x, const float* g, Act* y, float* copy_out, int rows, int d, float eps,
                           cudaStream_t stream) {
  return rmsnorm_reduce_launch<Act>(x, 1, 0, nullptr, nullptr, g, y, copy_out, rows, d, eps, stream, false);
}

template <typename Act>
cudaError_t rmsnorm_gather_launch(const float* x, const int* row_index, const float* g, Act* y, int rows, int d,
                                  float eps, cudaStream_t stream) {
  return rmsnorm_reduce_launch<Act>(x, 1, 0, nullptr, row_index, g, y, nullptr, rows, d, eps, stream, false);
}

template <typename Act>
cudaError_t rmsnorm_reduce_launch(const float* x, int n_split, long long split_stride, const float* residual,
                                  const int* row_index, const float* g, Act* y, float* copy_out, int rows, int d,
                                  float eps, cudaStream_t stream, bool discard) {
  if (rows == 0) return cudaSuccess;
  if (n_split > 1 || residual) {
    const size_t smem = (size_t)d * sizeof(float);
    if (smem > 48 * 1024) {
      static bool attr = false;
      if (!attr) {
        cudaError_t e =
            cudaFuncSetAttribute(k_rmsnorm<Act, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
        if (e != cudaSuccess) return e;
        attr = true;
      }
    }
    // two CTAs (rows) per SM fit beside each other: a one-wave grid for up to 2 x SMs rows
    const int threads = std::min(512, std::max(64, ((d / 4 + 31) / 32) * 32));
    OUTLETS_TRY_LAUNCH(launch_k(k_rmsnorm<Act, true>, dim3(rows), dim3(threads), smem, stream, x, n_split, split_stride, residual, row_index, g, y, copy_out,
                                                      d, eps, discard));
  } else {
    OUTLETS_TRY_LAUNCH(launch_k(k_rmsnorm<Act, false>, dim3(rows), dim3(256), 0, stream, x, 1, 0, nullptr, row_index, g, y, copy_out, d, eps, false));
  }
  return cudaGetLastError();
}

template <typename In, typename Act>
cudaError_t rope_scatter_launch(const In* qkv, const RopeArgs& a, cudaStream_t stream) {
  if (a.T == 0) return cudaSuccess;
  const int items = (a.H + a.KVH) * (a.hd / 16);  // rotation chunks per row
  const int threads = std::min(RopeBlock<In>::kThreads, std::max(64, ((items + 31) / 32) * 32));
  OUTLETS_TRY_LAUNCH(launch_k(k_rope_scatter<In, Act>, dim3(a.T), dim3(threads), 0, stream, qkv, a));
  return cudaGetLastError();
}

template <typename Act>
cudaError_t swiglu_launch(const float* gu, Act* u, int rows, int f_pad, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  OUTLETS_TRY_LAUNCH(launch_k(k_swiglu<Act>, dim3(grid_for((long long)rows * f_pad, 256)), dim3(256), 0, stream, gu, u, rows, f_pad));
  return cudaGetLastError();
}

template <typename Act>
cudaError_t embed_rmsnorm_launch(const int* tokens, const Act* table, int vocab, const float* g, Act* y, int rows,
                                 int d, float eps, int* err, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  const int threads = std::min(256, std::max(32, ((d / 8 + 31) / 32) * 32));
  OUTLETS_TRY_LAUNCH(launch_k(k_embed_rmsnorm<Act>, dim3(rows), dim3(threads), 0, stream, tokens, table, vocab, g, y, d,
                              eps, err));
  return cudaGetLastError();
}

cudaError_t head_tail_launch(const float* h_pre, int n_split, long long split_stride, const float* b_prev,
                             const float* w_last, const float* b_last, int rows, int width, float* z, float* len,
                             cudaStream_t stream, bool discard) {
  if (rows == 0) return cudaSuccess;
  const int threads = std::min(512, std::max(64, ((width / 4 + 31) / 32) * 32));
  OUTLETS_TRY_LAUNCH(launch_k(k_head_tail, dim3(rows), dim3(threads), 0, stream, h_pre, n_split, split_stride, b_prev, w_last, b_last, rows, width, z, len, discard));
  return cudaGetLastError();
}

cudaError_t gather_rows_launch(const void* src, const int* idx, void* dst, int rows, long long row_bytes,
                               cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  if (row_bytes % 16 || (reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) % 16)
    return cudaErrorInvalidValue;
  const long long vec = row_bytes / 16;
  OUTLETS_TRY_LAUNCH(launch_k(k_gather_rows, dim3(grid_for((long long)rows * vec, 256)), dim3(256), 0, stream,
                              reinterpret_cast<const uint4*>(src), idx, reinterpret_cast<uint4*>(dst), rows, vec));
  return cudaGetLastError();
}

template <typename Act>
cudaError_t convert_rows_launch(const float* src, Act* dst, int rows, int cols, long long dst_ld, int row_mode,
                                int row_base, long long kb_np, const float* col_scale, cudaStream_t stream) {
  if (rows == 0 || cols == 0) return cudaSuccess;
  OUTLETS_TRY_LAUNCH(launch_k(k_convert_rows<Act>, dim3(grid_for((long long)rows * cols, 256)), dim3(256), 0, stream, src, dst, rows, cols, dst_ld,
                                                                                row_mode, row_base, kb_np, col_scale));
  return cudaGetLastError();
}

cudaError_t wait_selftest_launch(int* err, unsigned long long timeout_ns, cudaStream_t stream) {
  k_wait_selftest<<<1, 32, 0, stream>>>(err, timeout_ns);
  return cudaGetLastError();
}

cudaError_t gemm_simt_f32_launch(const float* const a[3], const float* b, int epi, const GemmArgs& args,
                                 cudaStream_t stream) {
  if (args.M == 0 || args.N == 0) return cudaSuccess;
  dim3 grid((args.N + ST - 1) / ST, (args.M + ST - 1) / ST);
  OUTLETS_TRY_LAUNCH(launch_k(k_gemm_simt, dim3(grid), dim3(256), 0, stream, a[0], a[1], a[2], b, epi, args));
  return cudaGetLastError();
}

#define OUTLETS_INST_ACT(Act)                                                                                   \
  template cudaError_t rmsnorm_reduce_launch<Act>(const float*, int, long long, const float*, const int*,        \
                                                  const float*, Act*, float*, int, int, float, cudaStream_t,    \
                                                  bool);                                                        \
  template cudaError_t rmsnorm_launch<Act>(const float*, const float*, Act*, float*, int, int, float,          \
                                           cudaStream_t);                                                      \
  template cudaError_t rmsnorm_gather_launch<Act>(const float*, const int*, const float*, Act*, int, int, float, \
                                                  cudaStream_t);                                               \
  template cudaError_t swiglu_launch<Act>(const float*, Act*, int, int, cudaStream_t);                         \
  template cudaError_t embed_rmsnorm_launch<Act>(const int*, const Act*, int, const float*, Act*, int, int, float, \
                                                 int*, cudaStream_t);                                          \
  template cudaError_t convert_rows_launch<Act>(const float*, Act*, int, int, long long, int, int, long long,       \
                                                const float*, cudaStream_t);                                    \
  template cudaError_t rope_scatter_launch<float, Act>(const float*, const RopeArgs&, cudaStream_t);           \
  template cudaError_t rope_scatter_launch<Act, Act>(const Act*, const RopeArgs&, cudaStream_t);
OUTLETS_INST_ACT(bf16)
template cudaError_t rmsnorm_reduce_launch<float>(const float*, int, long long, const float*, const int*,
                                                  const float*, float*, float*, int, int, float, cudaStream_t, bool);
template cudaError_t rmsnorm_launch<float>(const float*, const float*, float*, float*, int, int, float, cudaStream_t);
template cudaError_t rmsnorm_gather_launch<float>(const float*, const int*, const float*, float*, int, int, float,
                                                  cudaStream_t);
template cudaError_t swiglu_launch<float>(const float*, float*, int, int, cudaStream_t);
template cudaError_t embed_rmsnorm_launch<float>(const int*, const float*, int, const float*, float*, int, int, float,
                                                 int*, cudaStream_t);
template cudaError_t convert_rows_launch<float>(const float*, float*, int, int, long long, int, int, long long,
                                                const float*, cudaStream_t);
template cudaError_t rope_scatter_launch<float, float>(const float*, const RopeArgs&, cudaStream_t);
#undef OUTLETS_INST_ACT

}  // namespace outlets
