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

template <typename Act>
__global__ void k_rmsnorm(const float* __restrict__ x, const int* __restrict__ row_index,
                          const float* __restrict__ g, Act* __restrict__ y, float* __restrict__ copy_out, int d,
                          float eps) {
  __shared__ float red[33];
  const int r = blockIdx.x;
  const long long src = row_index ? row_index[r] : r;
  const float* xr = x + src * d;
  float ss = 0.f;
  for (int i = threadIdx.x * 4; i < d; i += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(xr + i);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)d + eps);
  Act* yr = y + (long long)r * d;
  for (int i = threadIdx.x * 4; i < d; i += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(xr + i);
    const float4 gg = *reinterpret_cast<const float4*>(g + i);
    store4<Act>(yr + i, v.x * inv * gg.x, v.y * inv * gg.y, v.z * inv * gg.z, v.w * inv * gg.w);
    if (copy_out) *reinterpret_cast<float4*>(copy_out + (long long)r * d + i) = v;
  }
}

template <typename In, typename Act>
__global__ void k_rope_scatter(const In* __restrict__ qkv, const RopeArgs a) {
  const int row = blockIdx.x;
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
  const long long W = (long long)(H + 2 * KVH) * hd;
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
  for (int idx = threadIdx.x; idx < (H + KVH) * half; idx += blockDim.x) {
    const int head = idx / half;
    const int i = idx - head * half;
    const float x1 = to_f(src[head * hd + i]);
    const float x2 = to_f(src[head * hd + i + half]);
    const float c = cs[i], s = sn[i];
    const float y1 = x1 * c - x2 * s;
    const float y2 = x2 * c + x1 * s;
    if (head < H) {
      Act* qo = q_out + ((long long)row * H + head) * hd;
      qo[i] = from_f<Act>(y1);
      qo[i + half] = from_f<Act>(y2);
    } else {
      const int kh = head - H;
      if (k_out) {
        Act* ko = k_out + ((long long)kh * a.kv_ld_rows + row) * hd;
        ko[i] = from_f<Act>(y1);
        ko[i + half] = from_f<Act>(y2);
      }
      if (k_pool) {
        Act* kc = k_pool + (cache_base + (long long)kh * a.page_tokens) * hd;
        kc[i] = from_f<Act>(y1);
        kc[i + half] = from_f<Act>(y2);
      }
    }
  }
  const In* vs = src + (long long)(H + KVH) * hd;
  for (int idx = threadIdx.x; idx < KVH * hd; idx += blockDim.x) {
    const int kh = idx / hd;
    const int dd = idx - kh * hd;
    const Act val = from_f<Act>(to_f(vs[idx]));
    if (v_out) v_out[((long long)kh * a.kv_ld_rows + row) * hd + dd] = val;
    if (v_pool) v_pool[(cache_base + (long long)kh * a.page_tokens) * hd + dd] = val;
  }
}

template <typename Act>
__global__ void k_swiglu(const float* __restrict__ gu, Act* __restrict__ u, int rows, int f_pad) {
  const long long n = (long long)rows * f_pad;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < n;
       idx += (long long)gridDim.x * blockDim.x) {
    const long long r = idx / f_pad;
    const int j = (int)(idx - r * f_pad);
    const float* row = gu + r * 2 * f_pad + (j >> 7) * 256 + (j & 127);
    const float gt = row[0], up = row[128];
    u[idx] = from_f<Act>(gt / (1.f + __expf(-gt)) * up);
  }
}

__global__ void k_head_tail(const float* __restrict__ h, const float* __restrict__ b_prev,
                            const float* __restrict__ w_last, const float* __restrict__ b_last, int rows, int width,
                            float* __restrict__ z, float* __restrict__ len) {
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const float* hr = h + (long long)r * width;
  float acc = 0.f;
  for (int j = lane; j < width; j += 32) {
    float x = hr[j];
    if (b_prev) x = fmaxf(x + b_prev[j], 0.f);
    acc += w_last[j] * x;
  }
  acc = warp_sum(acc);
  if (lane == 0) {
    const float zz = acc + b_last[0];
    z[r] = zz;
    if (len) len[r] = fmaxf(0.f, expm1f(zz));
  }
}

template <typename Act>
__global__ void k_convert_rows(const float* __restrict__ src, Act* __restrict__ dst, int rows, int cols,
                               long long dst_ld, int row_mode, int row_base) {
  const long long n = (long long)rows * cols;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < n;
       idx += (long long)gridDim.x * blockDim.x) {
    const int r = (int)(idx / cols);
    const int c = (int)(idx - (long long)r * cols);
    int dr;
    if (row_mode == 0) dr = row_base + r;
    else if (row_mode == 1) dr = (r >> 7) * 256 + (r & 127);        // gate rows of an interleaved [gate|up] block
    else dr = (r >> 7) * 256 + 128 + (r & 127);                      // up rows
    dst[(long long)dr * dst_ld + c] = from_f<Act>(src[idx]);
  }
}

// ---------------------------------------------------------------- f32 GEMM (CUDA cores)
constexpr int ST = 64, SK = 16;

__global__ void __launch_bounds__(256) k_gemm_simt(const float* __restrict__ a0, const float* __restrict__ a1,
                                                   const float* __restrict__ a2, const float* __restrict__ bm,
                                                   int epi, const GemmArgs p) {
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

inline int grid_for(long long n, int threads) {
  long long g = (n + threads - 1) / threads;
  if (g > 152LL * 32) g = 152LL * 32;
  return (int)(g < 1 ? 1 : g);
}

}  // namespace

template <typename Act>
cudaError_t rmsnorm_launch(const float* x, const float* g, Act* y, float* copy_out, int rows, int d, float eps,
                           cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  k_rmsnorm<Act><<<rows, 256, 0, stream>>>(x, nullptr, g, y, copy_out, d, eps);
  return cudaGetLastError();
}

template <typename Act>
cudaError_t rmsnorm_gather_launch(const float* x, const int* row_index, const float* g, Act* y, int rows, int d,
                                  float eps, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  k_rmsnorm<Act><<<rows, 256, 0, stream>>>(x, row_index, g, y, nullptr, d, eps);
  return cudaGetLastError();
}

template <typename In, typename Act>
cudaError_t rope_scatter_launch(const In* qkv, const RopeArgs& a, cudaStream_t stream) {
  if (a.T == 0) return cudaSuccess;
  k_rope_scatter<In, Act><<<a.T, 128, 0, stream>>>(qkv, a);
  return cudaGetLastError();
}

template <typename Act>
cudaError_t swiglu_launch(const float* gu, Act* u, int rows, int f_pad, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  k_swiglu<Act><<<grid_for((long long)rows * f_pad, 256), 256, 0, stream>>>(gu, u, rows, f_pad);
  return cudaGetLastError();
}

cudaError_t head_tail_launch(const float* h_pre, const float* b_prev, const float* w_last, const float* b_last,
                             int rows, int width, float* z, float* len, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  k_head_tail<<<(rows + 7) / 8, 256, 0, stream>>>(h_pre, b_prev, w_last, b_last, rows, width, z, len);
  return cudaGetLastError();
}

template <typename Act>
cudaError_t convert_rows_launch(const float* src, Act* dst, int rows, int cols, long long dst_ld, int row_mode,
                                int row_base, cudaStream_t stream) {
  if (rows == 0 || cols == 0) return cudaSuccess;
  k_convert_rows<Act><<<grid_for((long long)rows * cols, 256), 256, 0, stream>>>(src, dst, rows, cols, dst_ld,
                                                                                row_mode, row_base);
  return cudaGetLastError();
}

cudaError_t gemm_simt_f32_launch(const float* const a[3], const float* b, int epi, const GemmArgs& args,
                                 cudaStream_t stream) {
  if (args.M == 0 || args.N == 0) return cudaSuccess;
  dim3 grid((args.N + ST - 1) / ST, (args.M + ST - 1) / ST);
  k_gemm_simt<<<grid, 256, 0, stream>>>(a[0], a[1], a[2], b, epi, args);
  return cudaGetLastError();
}

#define OUTLETS_INST_ACT(Act)                                                                                   \
  template cudaError_t rmsnorm_launch<Act>(const float*, const float*, Act*, float*, int, int, float,          \
                                           cudaStream_t);                                                      \
  template cudaError_t rmsnorm_gather_launch<Act>(const float*, const int*, const float*, Act*, int, int, float, \
                                                  cudaStream_t);                                               \
  template cudaError_t swiglu_launch<Act>(const float*, Act*, int, int, cudaStream_t);                         \
  template cudaError_t convert_rows_launch<Act>(const float*, Act*, int, int, long long, int, int, cudaStream_t); \
  template cudaError_t rope_scatter_launch<float, Act>(const float*, const RopeArgs&, cudaStream_t);           \
  template cudaError_t rope_scatter_launch<Act, Act>(const Act*, const RopeArgs&, cudaStream_t);
OUTLETS_INST_ACT(bf16)
template cudaError_t rmsnorm_launch<float>(const float*, const float*, float*, float*, int, int, float, cudaStream_t);
template cudaError_t rmsnorm_gather_launch<float>(const float*, const int*, const float*, float*, int, int, float,
                                                  cudaStream_t);
template cudaError_t swiglu_launch<float>(const float*, float*, int, int, cudaStream_t);
template cudaError_t convert_rows_launch<float>(const float*, float*, int, int, long long, int, int, cudaStream_t);
template cudaError_t rope_scatter_launch<float, float>(const float*, const RopeArgs&, cudaStream_t);
#undef OUTLETS_INST_ACT

}  // namespace outlets
