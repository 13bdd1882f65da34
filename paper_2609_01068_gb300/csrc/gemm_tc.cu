// tcgen05 GEMMs for sm_103a: C[M, N] = A[M, K] * B[N, K]^T, bf16 in, f32 accumulate.
// A (activations) is loaded by TMA tensor copies (128-byte swizzle); B (weights)
// lives in a k-block-major, pre-swizzled layout and is loaded by bulk copies.
//
// k_gemm_tc (large M, prefill): persistent, one CTA per SM, 6 warps:
//   warp 0      TMA producer (one thread): A and B K-blocks into a smem ring
//   warp 1      MMA issuer (one thread): tcgen05.mma 128 x BN x 16 into TMEM;
//               also owns the TMEM allocation
//   warps 2..5  epilogue: tcgen05.ld the accumulator, fuse the epilogue op,
//               store to global.  Warp w reads TMEM lanes 32*(w%4) .. +31.
// Two TMEM accumulators (2 * BN columns) let the epilogue of tile i overlap
// the main loop of tile i+1.  Every mbarrier wait is bounded.
//
// k_gemm_small (M <= 256, dynamic prediction and the head): one output tile and
// one K split per CTA, every weight tile streamed once; each K split writes an
// f32 slice that the consuming kernel adds up.
//
// Used for Eq. 1 (three-tap fusion: A is split along K over the three taps),
// the QKV / O / gate-up / down projections of the draft decoder layer, the
// first Linear of the length head and the draft LM head (Sec. 4.2, Eq. 2).
#include <stdlib.h>

#include "common.cuh"
#include "kernels.h"
#include "lm_topk.cuh"

namespace outlets {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // one 128-byte swizzle row of bf16

// BN: tile width (N); MT: 128-row M sub-tiles per tile (1 or 2).  With MT = 2 a
// CTA computes 256 rows against one staged B tile (two MMAs per K step into two
// TMEM accumulators), so each weight tile is read once for up to 256 rows.
template <int BN, int MT>
struct TcCfg {
  static constexpr int ACC = (512 / (MT * BN)) >= 2 ? 2 : 1;  // TMEM accumulator stages
  static_assert(BN % 64 == 0 && BN <= 256, "tile width");
  static constexpr uint32_t A_BYTES = MT * BM * BK * 2;
  static constexpr uint32_t B_BYTES = BN * BK * 2;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  // epilogue staging: one 32 x 32 f32 chunk per epilogue warp, rows padded to 36 words
  static constexpr uint32_t EPI_BYTES = 4 * 32 * 36 * 4;
  // the rest of the 227 KB a CTA may use goes to the ring (1 KB alignment + barriers aside)
  static constexpr int STAGES = ((232448 - 1024 - 256 - EPI_BYTES) / STAGE_BYTES) > 8
                                    ? 8
                                    : ((232448 - 1024 - 256 - EPI_BYTES) / STAGE_BYTES);
  static constexpr uint32_t TMEM_USED = ACC * MT * BN;
  static constexpr uint32_t TMEM_COLS = TMEM_USED <= 32 ? 32 : TMEM_USED <= 64 ? 64 : TMEM_USED <= 128 ? 128
                                                               : TMEM_USED <= 256 ? 256 : 512;  // power of 2
  static constexpr size_t SMEM = 1024 + STAGES * STAGE_BYTES + 256 + EPI_BYTES;
  static_assert(TMEM_USED <= 512, "TMEM columns");
};

struct Tile {
  int m_blk, n_blk, kb0, kb1, split;
};

__device__ __forceinline__ Tile decode_tile(int t, int num_m, int num_n, int group_m, int kb_total, int kb_per) {
  const int per_split = num_m * num_n;
  const int split = t / per_split;
  const int r = t - split * per_split;
  const int width = group_m * num_n;
  const int group = r / width;
  const int first_m = group * group_m;
  const int gm = min(num_m - first_m, group_m);
  const int rr = r - group * width;
  Tile tl;
  tl.m_blk = first_m + rr % gm;
  tl.n_blk = rr / gm;
  tl.kb0 = split * kb_per;
  tl.kb1 = min(kb_total, tl.kb0 + kb_per);
  tl.split = split;
  return tl;
}

// silu(x) = x * sigmoid(x); the fast division is exact to ~2 ulp (the result is rounded to bf16)
__device__ __forceinline__ float silu_f(float x) { return __fdividef(x, 1.0f + __expf(-x)); }

// RMSNorm folded into the GEMMs: row m's scale rsqrt(mean(x^2) + eps) from the
// per-N-tile sums of squares its producer left (summed in tile order).
__device__ __forceinline__ float fold_row_scale(const GemmArgs& p, int m) {
  if (!p.row_ss || m >= p.M) return 1.0f;
  const float* ss = p.row_ss + (long long)m * p.nrm_tiles;
  float t = 0.f;
#pragma unroll 8
  for (int i = 0; i < p.nrm_tiles; ++i) t += ss[i];
  return rsqrtf(t / (float)p.nrm_d + p.nrm_eps);
}

// Producer side: the 8 lanes (lane & 7) that share a row add up their
// columns' squares; the first writes the row's sum for this 64-column group.
// Groups of 64 columns whatever the tile width, so the consumer's sum over the
// groups (in group order) does not depend on how the producer was tiled.
__device__ __forceinline__ void fold_store_ss(const GemmArgs& p, float (&ssr)[8], int row0, int group, int lane) {
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    float v = ssr[k];
    v += __shfl_xor_sync(0xffffffffu, v, 1);
    v += __shfl_xor_sync(0xffffffffu, v, 2);
    v += __shfl_xor_sync(0xffffffffu, v, 4);
    const int mm = row0 + k * 4 + (lane >> 3);
    if ((lane & 7) == 0 && mm < p.M) p.nrm_ss[(long long)mm * p.nrm_tiles + group] = v;
    ssr[k] = 0.f;
  }
}

template <typename T>
__device__ __forceinline__ void store_row32(T* dst, const float* v, int valid);

template <>
__device__ __forceinline__ void store_row32<float>(float* dst, const float* v, int valid) {
  if (valid >= 32) {
#pragma unroll
    for (int j = 0; j < 32; j += 4)
      *reinterpret_cast<float4*>(dst + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
  } else {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (j < valid) dst[j] = v[j];
  }
}

template <>
__device__ __forceinline__ void store_row32<bf16>(bf16* dst, const float* v, int valid) {
  if (valid >= 32) {
#pragma unroll
    for (int j = 0; j < 32; j += 8) {
      uint4 p;
      p.x = pack_bf16x2(v[j], v[j + 1]);
      p.y = pack_bf16x2(v[j + 2], v[j + 3]);
      p.z = pack_bf16x2(v[j + 4], v[j + 5]);
      p.w = pack_bf16x2(v[j + 6], v[j + 7]);
      *reinterpret_cast<uint4*>(dst + j) = p;
    }
  } else {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (j < valid) dst[j] = __float2bfloat16_rn(v[j]);
  }
}

template <int BN, int EPI, int MT>
__global__ void __launch_bounds__(192, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap map_a0, const __grid_constant__ CUtensorMap map_a1,
              const __grid_constant__ CUtensorMap map_a2, const GemmArgs p) {
  using C = TcCfg<BN, MT>;
  constexpr int TM = BM * MT;  // rows per tile
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* epi_stage = reinterpret_cast<float*>(smem + C::STAGES * C::STAGE_BYTES + 256);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < C::ACC; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 128);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&map_a0);
    tma_prefetch_map(&map_a1);
    tma_prefetch_map(&map_a2);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_trigger();
  if (warp == 0 && lane == 0 && p.prefetch) {
    // weights never change: start pulling this CTA's first weight tiles toward L2
    // while the previous kernel finishes
    const int nm = (p.M + TM - 1) / TM, nn = (p.N + BN - 1) / BN, kbt = (p.K + BK - 1) / BK;
    if ((int)blockIdx.x < nm * nn * p.splits) {
    const Tile t0 = decode_tile(blockIdx.x, nm, nn, p.group_m, kbt, (kbt + p.splits - 1) / p.splits);
    const bf16* bt = reinterpret_cast<const bf16*>(p.b) + (long long)t0.n_blk * BN * BK;
    for (int kb = t0.kb0; kb < min(t0.kb1, t0.kb0 + p.prefetch); ++kb)
      bulk_prefetch_l2(bt + (long long)kb * p.b_np * BK, C::B_BYTES);
    }
  }
  pdl_wait();  // activations and outputs are touched only after the previous kernel is done

  const int num_m = (p.M + TM - 1) / TM;
  const int num_n = (p.N + BN - 1) / BN;
  const int kb_total = (p.K + BK - 1) / BK;
  const int kb_per = (kb_total + p.splits - 1) / p.splits;
  const int num_tiles = num_m * num_n * p.splits;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
        const Tile tl = decode_tile(t, num_m, num_n, p.group_m, kb_total, kb_per);
        const bf16* btile = reinterpret_cast<const bf16*>(p.b) + (long long)tl.n_blk * BN * BK;
        // weights streamed once: keep p.prefetch K blocks of B in flight toward L2
        for (int kb = tl.kb0; kb < min(tl.kb1, tl.kb0 + p.prefetch); ++kb)
          bulk_prefetch_l2(btile + (long long)kb * p.b_np * BK, C::B_BYTES);
        for (int kb = tl.kb0; kb < tl.kb1; ++kb) {
          if (p.prefetch && kb + p.prefetch < tl.kb1)
            bulk_prefetch_l2(btile + (long long)(kb + p.prefetch) * p.b_np * BK, C::B_BYTES);
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, p.err)) goto producer_done;
          uint8_t* sa = smem + stage * C::STAGE_BYTES;
          uint8_t* sb = sa + C::A_BYTES;
          mbar_arrive_expect_tx(&full[stage], C::STAGE_BYTES);
          const int kg = kb * BK;
          const int piece = kg / p.k_per_map;
          const int kl = kg - piece * p.k_per_map;
          const CUtensorMap* am = piece == 0 ? &map_a0 : (piece == 1 ? &map_a1 : &map_a2);
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
            tma_load_2d(sa + mt * (BM * BK * 2), am, &full[stage], kl, tl.m_blk * TM + mt * BM);
          bulk_load(sb, reinterpret_cast<const bf16*>(p.b) + ((long long)kb * p.b_np + tl.n_blk * BN) * BK,
                    C::B_BYTES, &full[stage]);
          if (++stage == C::STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    producer_done:;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
        const Tile tl = decode_tile(t, num_m, num_n, p.group_m, kb_total, kb_per);
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, p.err)) goto mma_done;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * MT * BN);
        for (int kb = tl.kb0; kb < tl.kb1; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, p.err)) goto mma_done;
          tc_fence_after();
          const uint32_t a_addr = smem_u32(smem + stage * C::STAGE_BYTES);
          const uint32_t b_addr = a_addr + C::A_BYTES;
          const uint64_t bdesc = sw128_kmajor_desc(b_addr);
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            const uint64_t adesc = sw128_kmajor_desc(a_addr + mt * (BM * BK * 2));
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
              // advance 16 elements (32 bytes = 2 units of 16 bytes) along K
              tc_mma_bf16(d_tmem + mt * BN, adesc + 2u * kk, bdesc + 2u * kk, idesc,
                          (kb > tl.kb0 || kk > 0) ? 1u : 0u);
            }
          }
          tc_commit(&empty[stage]);
          if (++stage == C::STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        tc_commit(&tfull[acc]);
        if (++acc == C::ACC) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
    mma_done:;
    }
  } else {
    // epilogue warps 2..5
    const int quarter = warp & 3;
    const int row_in_tile = quarter * 32 + lane;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
      const Tile tl = decode_tile(t, num_m, num_n, p.group_m, kb_total, kb_per);
      // folded RMSNorm: this thread's row scales, read while the main loop runs
      float rs_rows[MT];
#pragma unroll
      for (int mt = 0; mt < MT; ++mt)
        rs_rows[mt] = (EPI == EPI_SWIGLU || EPI == EPI_ACT) ? fold_row_scale(p, tl.m_blk * TM + mt * BM + row_in_tile)
                                                            : 1.0f;
      if (!mbar_wait(&tfull[acc], acc_phase, abort_flag, p.err)) break;
      tc_fence_after();
#pragma unroll 1
      for (int mt = 0; mt < MT; ++mt) {
      const int m = tl.m_blk * TM + mt * BM + row_in_tile;
      const bool row_ok = m < p.M;
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                             static_cast<uint32_t>((acc * MT + mt) * BN);
      if constexpr (EPI == EPI_SWIGLU) {
        // B rows are interleaved in blocks of 32: tile columns [64j, 64j+32) are
        // gate and [64j+32, 64j+64) up for the same 32 outputs
        const int n_out = p.N / 2;
        const float rs = rs_rows[mt];  // 1 unless the norm is folded in
        for (int c = 0; c < BN; c += 64) {
          uint32_t g[32], u[32];
          tmem_ld_32x32b_x32(tbase + c, g);
          tmem_ld_32x32b_x32(tbase + c + 32, u);
          tmem_ld_wait();
          const int n0 = (tl.n_blk * BN + c) / 2;
          if (row_ok && n0 < n_out) {
            float v[32];
#pragma unroll
            for (int j = 0; j < 32; ++j)
              v[j] = silu_f(__uint_as_float(g[j]) * rs) * (__uint_as_float(u[j]) * rs);
            store_row32(reinterpret_cast<bf16*>(p.out) + (long long)m * p.ldo + n0, v, min(32, n_out - n0));
          }
        }
      } else if (EPI == EPI_F32 && p.residual) {
        // f32 out + residual: the chunk loop is unrolled so the residual loads
        // of the next LA chunks are in flight while a chunk is written (a short
        // K loop, as in the O projection, leaves no time to wait for each).
        constexpr int NC = BN / 32;
        constexpr int LA = NC < 3 ? NC : 3;
        const int row0 = tl.m_blk * TM + mt * BM + quarter * 32;
        const int cq = (lane & 7) * 4;
        float* stg = epi_stage + (warp - 2) * (32 * 36);
        float4 res[LA][8];
        auto load_res = [&](int ci, float4 (&rr)[8]) {
          const int n = tl.n_blk * BN + ci * 32 + cq;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int mm = row0 + k * 4 + (lane >> 3);
            rr[k] = (mm < p.M && n < p.N)
                        ? __ldg(reinterpret_cast<const float4*>(p.residual + (long long)mm * p.ldr + n))
                        : make_float4(0.f, 0.f, 0.f, 0.f);
          }
        };
#pragma unroll
        for (int i = 0; i < LA; ++i) load_res(i, res[i]);
        float ssr[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int ci = 0; ci < NC; ++ci) {
          uint32_t r[32];
          tmem_ld_32x32b_x32(tbase + ci * 32, r);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 32; j += 4)
            *reinterpret_cast<float4*>(stg + lane * 36 + j) = make_float4(
                __uint_as_float(r[j]), __uint_as_float(r[j + 1]), __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3]));
          __syncwarp();
          const int n = tl.n_blk * BN + ci * 32 + cq;
          if (n < p.N) {
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const int rr = k * 4 + (lane >> 3);
              if (row0 + rr < p.M) {
                const float4 v = *reinterpret_cast<const float4*>(stg + rr * 36 + cq);
                const float4 q = res[ci % LA][k];
                const float4 o = make_float4(v.x + q.x, v.y + q.y, v.z + q.z, v.w + q.w);
                *reinterpret_cast<float4*>(reinterpret_cast<float*>(p.out) + (long long)(row0 + rr) * p.ldo + n) = o;
                if (p.nrm_out) {
                  uint2 packed;
                  packed.x = pack_bf16x2(o.x, o.y);
                  packed.y = pack_bf16x2(o.z, o.w);
                  *reinterpret_cast<uint2*>(p.nrm_out + (long long)(row0 + rr) * p.ldo + n) = packed;
                  ssr[k] += o.x * o.x + o.y * o.y + o.z * o.z + o.w * o.w;
                }
              }
            }
          }
          if (ci + LA < NC) load_res(ci + LA, res[ci % LA]);
          __syncwarp();
          if ((ci & 1) && p.nrm_out) fold_store_ss(p, ssr, row0, (tl.n_blk * BN + ci * 32) / 64, lane);
        }
      } else {
        float ssr[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};  // EPI_F32 producer of a folded norm
        const float rs_mine = rs_rows[mt];  // EPI_ACT consumer of a folded norm (else 1)
        for (int c = 0; c < BN; c += 32) {
          uint32_t r[32];
          tmem_ld_32x32b_x32(tbase + c, r);
          tmem_ld_wait();
          const int n0 = tl.n_blk * BN + c;
          if constexpr (EPI == EPI_F32 || EPI == EPI_ACT) {
            // stage the 32 x 32 chunk (thread = row) in shared memory, then write it
            // out line by line: 8 lanes x 16 bytes cover one row's 32 columns, 4 rows
            // per instruction.  Row stride 36 words: both directions conflict-free.
            float* stg = epi_stage + (warp - 2) * (32 * 36);
#pragma unroll
            for (int j = 0; j < 32; j += 4)
              *reinterpret_cast<float4*>(stg + lane * 36 + j) = make_float4(
                  __uint_as_float(r[j]), __uint_as_float(r[j + 1]), __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3]));
            __syncwarp();
            const int row0 = tl.m_blk * TM + mt * BM + quarter * 32;
            const int cq = (lane & 7) * 4;  // this lane's 4 columns of the chunk
            const int n = n0 + cq;
            float rsk[8];                   // EPI_ACT: the scales of the 8 rows this lane writes
#pragma unroll
            for (int k = 0; k < 8; ++k)
              rsk[k] = EPI == EPI_ACT ? __shfl_sync(0xffffffffu, rs_mine, k * 4 + (lane >> 3)) : 1.0f;
            if (n < p.N) {                  // N % 4 == 0: a lane's 4 columns are all in or all out
              if constexpr (EPI == EPI_F32) {
                float4 res[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) {  // all residual loads first, then the stores
                  const int mm = row0 + k * 4 + (lane >> 3);
                  res[k] = (p.residual && mm < p.M)
                               ? __ldg(reinterpret_cast<const float4*>(p.residual + (long long)mm * p.ldr + n))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
                }
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                  const int rr = k * 4 + (lane >> 3);
                  if (row0 + rr < p.M) {
                    const float4 v = *reinterpret_cast<const float4*>(stg + rr * 36 + cq);
                    const float4 o = make_float4(v.x + res[k].x, v.y + res[k].y, v.z + res[k].z, v.w + res[k].w);
                    *reinterpret_cast<float4*>(reinterpret_cast<float*>(p.out) + (long long)(row0 + rr) * p.ldo + n) = o;
                    if (p.nrm_out) {
                      uint2 packed;
                      packed.x = pack_bf16x2(o.x, o.y);
                      packed.y = pack_bf16x2(o.z, o.w);
                      *reinterpret_cast<uint2*>(p.nrm_out + (long long)(row0 + rr) * p.ldo + n) = packed;
                      ssr[k] += o.x * o.x + o.y * o.y + o.z * o.z + o.w * o.w;
                    }
                  }
                }
              } else {
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                  const int rr = k * 4 + (lane >> 3);
                  const float rs = rsk[k];
                  if (row0 + rr < p.M) {
                    const float4 v = *reinterpret_cast<const float4*>(stg + rr * 36 + cq);
                    uint2 packed;
                    packed.x = pack_bf16x2(v.x * rs, v.y * rs);
                    packed.y = pack_bf16x2(v.z * rs, v.w * rs);
                    *reinterpret_cast<uint2*>(reinterpret_cast<bf16*>(p.out) + (long long)(row0 + rr) * p.ldo + n) =
                        packed;
                  }
                }
              }
            }
            if constexpr (EPI == EPI_F32) {  // after every second 32-column chunk (all lanes together)
              if ((c & 32) && p.nrm_out) fold_store_ss(p, ssr, row0, n0 / 64, lane);
            }
            __syncwarp();
          } else if (row_ok && n0 < p.N) {  // EPI_BIAS_RELU
            const int valid = min(32, p.N - n0);
            float v[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = j < valid ? fmaxf(__uint_as_float(r[j]) + p.bias[n0 + j], 0.0f) : 0.0f;
            store_row32(reinterpret_cast<float*>(p.out) + (long long)m * p.ldo + n0, v, valid);
          }
        }
      }
      }  // mt
      tc_fence_before();
      mbar_arrive(&tempty[acc]);
      if (++acc == C::ACC) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

template <int BN, int EPI, int MT>
cudaError_t launch_one(const CUtensorMap a_maps[3], const GemmArgs& args, int num_sms,
                       cudaStream_t stream) {
  using C = TcCfg<BN, MT>;
  auto kern = k_gemm_tc<BN, EPI, MT>;
  static bool attr_set = false;  // per (BN, EPI) instantiation
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const long long tiles = (long long)((args.M + BM * MT - 1) / (BM * MT)) * ((args.N + BN - 1) / BN) * args.splits;
  const int grid = (int)(tiles < num_sms ? tiles : num_sms);
  if (grid <= 0) return cudaSuccess;
  OUTLETS_TRY_LAUNCH(launch_k(kern, dim3(grid), dim3(192), C::SMEM, stream, a_maps[0], a_maps[1], a_maps[2], args));
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Small-M kernel.  A CTA computes one (up to 256) x BN output tile over one
// K split (balanced, never empty).  Activations and weights have their own
// ring barriers (AS and WS slots; the producer may run the weight ring
// WS - AS blocks ahead); with AS == WS this is one ring holding both tiles of
// a K block, which is what the latency of both operands needs.
// ---------------------------------------------------------------- draft LM head epilogue (Eq. 2)
// Epilogue warps of the draft LM head kernel: 8 (two per TMEM lane quarter;
// the two warps of a quarter take the two column halves of the tile).
constexpr int kLmEpiWarps = 8;
constexpr int kLmEpiThreads = kLmEpiWarps * 32;
// Candidate places per epilogue thread in the idle operand ring.
constexpr int kLmCap = 64;

__device__ __forceinline__ float lm_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void lm_store32(float* dst, const uint32_t (&r)[32], int n, bool vec) {
  if (vec && n >= 32) {
#pragma unroll
    for (int j = 0; j < 32; j += 4)
      *reinterpret_cast<float4*>(dst + j) = make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]),
                                                        __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3]));
  } else {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (j < n) dst[j] = __uint_as_float(r[j]);
  }
}

// Inserts candidate list entries 0 .. cnt-1 of thread et into the sorted list.
template <int KT>
__device__ __forceinline__ void lm_flush(float (&tv)[KT], int (&ti)[KT], const float* cval, const int* cidx, int et,
                                         int n0, int cnt) {
#pragma unroll 1
  for (int i = 0; i < cnt; ++i)
    lm_insert<KT>(tv, ti, cval[i * kLmEpiThreads + et], n0 + cidx[i * kLmEpiThreads + et]);
}

// One row of one column half of a draft LM head tile.  The calling thread
// owns TMEM lane `tb`'s row (global row m) and chunks ch0 .. ch1-1 of 32
// columns (tile columns n0 + 32 ch ..; the first lim tile columns are inside
// the vocabulary when MASK), and writes the partials (kernels.h) of partial
// tile pt (num_pt partial tiles per row).
//  pass 1 reads the columns from TMEM and takes the maximum of each of 8
//         column groups (column mod 8); the smallest group maximum is reached
//         by 8 distinct columns, so it bounds the half's 8th best logit from
//         below.  A bound over the whole row comes from the row's 8 slots:
//         slot pt mod 8 keeps the largest maximum of the partial tiles it has
//         seen, so the slots hold logits of 8 distinct columns and their
//         minimum never exceeds the row's 8th best logit.  The slots are read
//         before pass 1 (the loads overlap it) and this half's maximum is
//         added after it.  Once every slot has seen a few tiles the bound is
//         close to the row's 8th best and later tiles keep almost no
//         candidates; which tile sees which bound depends on timing, the
//         merged top-k does not.
//  pass 2 re-reads the columns and sums exp(logit - max) in one branch-free
//         block per chunk; only a chunk in which some lane of the warp has a
//         logit at or above the bound goes through candidate collection,
//         which moves those logits to the thread's list in shared memory.
//  The list goes through the sorted insertion after the scan (and before a
//  chunk whenever fewer than 32 places are left, raising the bound to the
//  current KT-th best), so the lanes of a warp do not diverge on every logit.
template <int BN, int KT, bool MASK>
__device__ __forceinline__ void lm_row(const GemmArgs& p, uint32_t tb, int m, int n0, int lim, int ch0, int ch1,
                                       int pt, int num_pt, float* cval, int* cidx, int et) {
  static_assert(kLmCap >= 64, "a flushed list takes a whole chunk");
  // rows past M read zero-filled A: nothing to do there (tcgen05.ld is
  // warp-collective, so a warp with any live row runs the scan as a whole)
  const bool live = m < p.M;
  if (!__any_sync(0xffffffffu, live)) return;
  int* slot = p.lm_bound + (long long)(live ? m : 0) * kLmBoundSlots;
  int4 sa = make_int4(kLmBoundInit, kLmBoundInit, kLmBoundInit, kLmBoundInit), sb = sa;
  if (KT > 1 && live) {
    sa = __ldcg(reinterpret_cast<const int4*>(slot));
    sb = __ldcg(reinterpret_cast<const int4*>(slot) + 1);
  }
  float gmax[8];
#pragma unroll
  for (int g = 0; g < 8; ++g) gmax[g] = -INFINITY;
  float best = -INFINITY;
  int best_c = INT_MAX;
#pragma unroll 1
  for (int ch = ch0; ch < ch1; ++ch) {
    uint32_t r[32];
    tmem_ld_32x32b_x32(tb + ch * 32, r);
    tmem_ld_wait();
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int col = ch * 32 + j;
      float v = __uint_as_float(r[j]);
      if (MASK && col >= lim) v = -INFINITY;
      if constexpr (KT == 1) {
        if (v > best) {  // strict: the first (smallest) column keeps a tie
          best = v;
          best_c = col;
        }
      } else {
        gmax[j & 7] = fmaxf(gmax[j & 7], v);
      }
    }
  }
  float mx = best, thr = gmax[0];
  if constexpr (KT > 1) {
    mx = gmax[0];
#pragma unroll
    for (int g = 1; g < 8; ++g) {
      mx = fmaxf(mx, gmax[g]);
      thr = fminf(thr, gmax[g]);
    }
    if (live) {
      atomicMax(slot + (pt & (kLmBoundSlots - 1)), lm_key(mx));
      const int kmin = min(min(min(sa.x, sa.y), min(sa.z, sa.w)), min(min(sb.x, sb.y), min(sb.z, sb.w)));
      thr = fmaxf(thr, lm_unkey(kmin));
    }
  }
  const float mxl = mx == -INFINITY ? 0.f : mx * kLog2e;  // a half past the vocabulary: sum 0
  float tv[KT];
  int ti[KT];
  lm_init<KT>(tv, ti);
  float se = 0.f;
  int cnt = 0;
  float* lrow = (p.lm_logits && live) ? p.lm_logits + (long long)m * p.ldo + n0 : nullptr;
  const bool vec = (reinterpret_cast<uintptr_t>(lrow) & 15) == 0;
#pragma unroll 1
  for (int ch = ch0; ch < ch1; ++ch) {
    if constexpr (KT > 1) {
      if (cnt > kLmCap - 32) {
        lm_flush<KT>(tv, ti, cval, cidx, et, n0, cnt);
        cnt = 0;
        thr = fmaxf(thr, tv[KT - 1]);
      }
    }
    uint32_t r[32];
    tmem_ld_32x32b_x32(tb + ch * 32, r);
    tmem_ld_wait();
    if (MASK) {
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (ch * 32 + j >= lim) r[j] = __float_as_uint(-INFINITY);
    }
    // softmax sum: one branch-free block (four partial sums), the chunk's max on the side
    float s4[4] = {0.f, 0.f, 0.f, 0.f};
    float cmx = -INFINITY;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float v = __uint_as_float(r[j]);
      s4[j & 3] += lm_ex2(fmaf(v, kLog2e, -mxl));
      cmx = fmaxf(cmx, v);
    }
    se += (s4[0] + s4[1]) + (s4[2] + s4[3]);
    if constexpr (KT > 1) {
      if (__any_sync(0xffffffffu, live && cmx >= thr)) {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float v = __uint_as_float(r[j]);
          const bool take = live && v >= thr;
          if (take) {
            cval[cnt * kLmEpiThreads + et] = v;
            cidx[cnt * kLmEpiThreads + et] = ch * 32 + j;
          }
          cnt += take ? 1 : 0;
        }
      }
    }
    if (lrow) lm_store32(lrow + ch * 32, r, MASK ? lim - ch * 32 : 32, vec);
  }
  if constexpr (KT == 1) {
    tv[0] = best;
    ti[0] = best_c == INT_MAX ? INT_MAX : n0 + best_c;
  } else {
    lm_flush<KT>(tv, ti, cval, cidx, et, n0, cnt);
  }
  if (live) {
    const long long e = (long long)m * num_pt + pt;
    p.lm_stats[e] = make_float2(mx, se);
    int2* tp = p.lm_top + e * KT;
#pragma unroll
    for (int i = 0; i < KT; ++i) tp[i] = make_int2(__float_as_int(tv[i]), ti[i]);
  }
}

template <int BN, int MT>
struct SmCfg {
  static constexpr uint32_t A_BYTES = MT * BM * BK * 2;
  static constexpr uint32_t B_BYTES = BN * BK * 2;
  // one ring slot per K block for activations and weights alike: latency hides
  // behind total bytes in flight, so the ring takes every byte of the 227 KB
  static constexpr int FIT = (int)((232448u - 1024u - 256u) / (A_BYTES + B_BYTES));
  static constexpr int AS = FIT > 8 ? 8 : FIT;
  static constexpr int WS = AS;
  static constexpr uint32_t RING_BYTES = AS * A_BYTES + WS * B_BYTES;
  static constexpr uint32_t TMEM_USED = MT * BN;
  static constexpr uint32_t TMEM_COLS = TMEM_USED <= 64 ? 64 : TMEM_USED <= 128 ? 128 : TMEM_USED <= 256 ? 256 : 512;
  static constexpr size_t SMEM = 1024 + RING_BYTES + 256;
  static_assert(AS >= 2, "ring");
  static_assert(TMEM_USED <= 512, "TMEM columns");
};

// Threads of a small-M GEMM CTA: producer warp, MMA warp, epilogue warps
// (4; 8 for the draft LM head, whose epilogue is the longer part of a tile).
template <int EPI>
constexpr int small_threads() {
  return (EPI == EPI_LM1 || EPI == EPI_LM8) ? 64 + kLmEpiThreads : 192;
}

template <int BN, int EPI, int MT>
__global__ void __launch_bounds__(small_threads<EPI>(), 1)
    k_gemm_small(const __grid_constant__ CUtensorMap map_a0, const __grid_constant__ CUtensorMap map_a1,
                 const __grid_constant__ CUtensorMap map_a2, const GemmArgs p) {
  using C = SmCfg<BN, MT>;
  constexpr int TM = BM * MT;
  constexpr int AS = C::AS, WS = C::WS;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sW = smem + AS * C::A_BYTES;
  uint64_t* fullA = reinterpret_cast<uint64_t*>(smem + C::RING_BYTES);
  uint64_t* emptyA = fullA + AS;
  uint64_t* fullW = emptyA + AS;
  uint64_t* emptyW = fullW + WS;
  uint64_t* tfull = emptyW + WS;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tfull + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < AS; ++i) {
      mbar_init(&fullA[i], 1);
      mbar_init(&emptyA[i], 1);
    }
    for (int i = 0; i < WS; ++i) {
      mbar_init(&fullW[i], 1);
      mbar_init(&emptyW[i], 1);
    }
    mbar_init(&tfull[0], 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&map_a0);
    tma_prefetch_map(&map_a1);
    tma_prefetch_map(&map_a2);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_trigger();

  const int S = p.splits;
  const int tile = blockIdx.x / S;
  const int split = blockIdx.x - tile * S;
  const int num_n = (p.N + BN - 1) / BN;
  const int m_blk = tile / num_n;
  const int n_blk = tile - m_blk * num_n;
  const int kb_total = (p.K + BK - 1) / BK;
  // balanced split: every split gets floor or ceil of kb_total / S blocks (S <= kb_total)
  const int kb0 = (int)(((long long)split * kb_total) / S);
  const int kb1 = (int)(((long long)(split + 1) * kb_total) / S);
  const bf16* wt = reinterpret_cast<const bf16*>(p.b) + (long long)n_blk * BN * BK;
  // Weights do not depend on the previous kernel: fill the first weight slots
  // while it is still running, before waiting for its outputs (activations).
  const int pre = min(WS, kb1 - kb0);
  if (warp == 0 && lane == 0) {
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(&fullW[i], C::B_BYTES);
      bulk_load(sW + i * C::B_BYTES, wt + (long long)(kb0 + i) * p.b_np * BK, C::B_BYTES, &fullW[i]);
    }
  }
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      constexpr int lag = WS - AS;  // >= 0
      int ws = pre % WS, as = 0;
      uint32_t wph = pre == WS ? 1u : 0u, aph = 0;
      for (int i = kb0; i < kb1 + lag; ++i) {
        if (i < kb1 && i >= kb0 + pre) {
          if (!mbar_wait(&emptyW[ws], wph ^ 1u, abort_flag, p.err)) break;
          mbar_arrive_expect_tx(&fullW[ws], C::B_BYTES);
          bulk_load(sW + ws * C::B_BYTES, wt + (long long)i * p.b_np * BK, C::B_BYTES, &fullW[ws]);
          if (++ws == WS) {
            ws = 0;
            wph ^= 1u;
          }
        }
        const int j = i - lag;
        if (j >= kb0 && j < kb1) {
          if (!mbar_wait(&emptyA[as], aph ^ 1u, abort_flag, p.err)) break;
          mbar_arrive_expect_tx(&fullA[as], C::A_BYTES);
          const int kg = j * BK;
          const int piece = kg / p.k_per_map;
          const int kl = kg - piece * p.k_per_map;
          const CUtensorMap* am = piece == 0 ? &map_a0 : (piece == 1 ? &map_a1 : &map_a2);
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
            tma_load_2d(sA + as * C::A_BYTES + mt * (BM * BK * 2), am, &fullA[as], kl, m_blk * TM + mt * BM);
          if (++as == AS) {
            as = 0;
            aph ^= 1u;
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
      int ws = 0, as = 0;
      uint32_t wph = 0, aph = 0;
      for (int kb = kb0; kb < kb1; ++kb) {
        if (!mbar_wait(&fullA[as], aph, abort_flag, p.err)) break;
        if (!mbar_wait(&fullW[ws], wph, abort_flag, p.err)) break;
        tc_fence_after();
        const uint32_t a_addr = smem_u32(sA + as * C::A_BYTES);
        const uint64_t bdesc = sw128_kmajor_desc(smem_u32(sW + ws * C::B_BYTES));
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          const uint64_t adesc = sw128_kmajor_desc(a_addr + mt * (BM * BK * 2));
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            tc_mma_bf16(tmem_base + mt * BN, adesc + 2u * kk, bdesc + 2u * kk, idesc, (kb > kb0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(&emptyA[as]);
        tc_commit(&emptyW[ws]);
        if (++ws == WS) {
          ws = 0;
          wph ^= 1u;
        }
        if (++as == AS) {
          as = 0;
          aph ^= 1u;
        }
      }
      tc_commit(&tfull[0]);
    }
  }
  __syncwarp();

  bool have = false;
  if (warp >= 2) {
    have = mbar_wait(&tfull[0], 0, abort_flag, p.err);
    tc_fence_after();
  }
  const int quarter = warp & 3;
  if constexpr (EPI == EPI_SWIGLU) {
    if (warp >= 2 && have) {
      const int n_out = p.N / 2;
#pragma unroll 1
      for (int mt = 0; mt < MT; ++mt) {
        const int m = m_blk * TM + mt * BM + quarter * 32 + lane;
        const uint32_t tb = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(mt * BN);
        for (int c = 0; c < BN; c += 64) {
          uint32_t g[32], u[32];
          tmem_ld_32x32b_x32(tb + c, g);
          tmem_ld_32x32b_x32(tb + c + 32, u);
          tmem_ld_wait();
          const int n0 = (n_blk * BN + c) / 2;
          if (m < p.M && n0 < n_out) {
            float v[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = silu_f(__uint_as_float(g[j])) * __uint_as_float(u[j]);
            store_row32(reinterpret_cast<bf16*>(p.out) + (long long)m * p.ldo + n0, v, min(32, n_out - n0));
          }
        }
      }
    }
  } else if constexpr (EPI == EPI_LM1 || EPI == EPI_LM8) {
    // warps 2..9: lane quarter warp % 4, column half (warp - 2) / 4; each half
    // is its own partial tile (2 per N tile), so nothing is combined here
    constexpr int KT = EPI == EPI_LM1 ? 1 : 8;
    constexpr int NCH = BN / 32, SPLIT = (NCH + 1) / 2;
    static_assert((size_t)kLmCap * kLmEpiThreads * 8 <= C::RING_BYTES, "candidate lists fit in the ring");
    if (warp >= 2 && have) {
      const int et = threadIdx.x - 64;
      const int half = (warp - 2) >> 2;
      float* cval = reinterpret_cast<float*>(smem);
      int* cidx = reinterpret_cast<int*>(smem + kLmCap * kLmEpiThreads * 4);
      const int n0 = n_blk * BN;
      const int lim = p.N - n0;
      const int ch0 = half ? SPLIT : 0, ch1 = half ? NCH : SPLIT;
#pragma unroll 1
      for (int mt = 0; mt < MT; ++mt) {
        const int m = m_blk * TM + mt * BM + quarter * 32 + lane;
        const uint32_t tb = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(mt * BN);
        if (lim >= BN)
          lm_row<BN, KT, false>(p, tb, m, n0, lim, ch0, ch1, 2 * n_blk + half, 2 * num_n, cval, cidx, et);
        else
          lm_row<BN, KT, true>(p, tb, m, n0, lim, ch0, ch1, 2 * n_blk + half, 2 * num_n, cval, cidx, et);
      }
    }
  } else {
    // Split-K partial: the f32 tile of this K split goes to slice `split`
    // (out + split * group_stride); the consuming kernel adds the slices in
    // slice order, so the sum does not depend on scheduling.  The tile is
    // staged in the idle ring CW columns at a time (warps 2..5 read TMEM, one
    // row per thread) and written by all six warps with row-contiguous float4
    // stores (a warp store covers one 512-byte row segment).
    constexpr int CW = BN < 128 ? BN : 128;
    constexpr int LD = CW + 4;  // 16-byte row skew: conflict-free thread-per-row staging
    constexpr int Q = CW / 4;   // float4 per staged row
    constexpr int ITEMS = TM * Q;
    static_assert((size_t)TM * LD * 4 <= C::RING_BYTES, "stage fits in the ring");
    float* stage = reinterpret_cast<float*>(smem);
    float* out = reinterpret_cast<float*>(p.out) + (long long)split * p.group_stride;
    for (int rd = 0; rd < BN / CW; ++rd) {
      if (rd > 0) __syncthreads();  // the previous round's reads of the stage are done
      if (warp >= 2 && have) {
#pragma unroll 1
        for (int mt = 0; mt < MT; ++mt) {
          const int row = mt * BM + quarter * 32 + lane;
          const uint32_t tb = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                              static_cast<uint32_t>(mt * BN + rd * CW);
#pragma unroll 1
          for (int c = 0; c < CW; c += 32) {
            uint32_t r[32];
            tmem_ld_32x32b_x32(tb + c, r);
            tmem_ld_wait();
            float* dst = stage + row * LD + c;
#pragma unroll
            for (int j = 0; j < 32; j += 4)
              *reinterpret_cast<float4*>(dst + j) = make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]),
                                                                __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3]));
          }
        }
      }
      __syncthreads();
      if (!*abort_flag) {
        const int n0 = n_blk * BN + rd * CW;
#pragma unroll 4
        for (int it = threadIdx.x; it < ITEMS; it += 192) {
          const int row = it / Q;
          const int col = (it - row * Q) * 4;
          const int m = m_blk * TM + row;
          const int n = n0 + col;
          if (m < p.M && n < p.N)
            *reinterpret_cast<float4*>(out + (long long)m * p.ldo + n) =
                *reinterpret_cast<const float4*>(stage + row * LD + col);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

template <int BN, int EPI, int MT>
cudaError_t launch_small(const CUtensorMap a_maps[3], const GemmArgs& args, cudaStream_t stream) {
  using C = SmCfg<BN, MT>;
  auto kern = k_gemm_small<BN, EPI, MT>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const int tiles = ((args.M + BM * MT - 1) / (BM * MT)) * ((args.N + BN - 1) / BN);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(tiles * args.splits);
  cfg.blockDim = dim3(small_threads<EPI>());
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = stream;
  cudaLaunchAttribute at[1];
  int n = 0;
  if (pdl_enabled()) {
    at[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = at;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kern, a_maps[0], a_maps[1], a_maps[2], args);
}

}  // namespace

bool pdl_enabled() {
  static const bool on = [] {
    const char* v = getenv("OUTLETS_PDL");
    return !(v && v[0] == '0');
  }();
  return on;
}

cudaError_t gemm_small_launch(const CUtensorMap a_maps[3], int bn, int epi, int mt, const GemmArgs& args,
                              cudaStream_t stream) {
  if (args.splits < 1 || (epi == EPI_SLICES && args.N % 4)) return cudaErrorInvalidValue;
  if ((epi == EPI_LM1 || epi == EPI_LM8) && (args.splits != 1 || !args.lm_stats || !args.lm_top))
    return cudaErrorInvalidValue;
  if (epi == EPI_LM8 && !args.lm_bound) return cudaErrorInvalidValue;
#define OUTLETS_SM_CASE(BNV, EV, MTV) \
  if (bn == BNV && epi == EV && mt == MTV) return launch_small<BNV, EV, MTV>(a_maps, args, stream);
  OUTLETS_SM_CASE(256, EPI_SLICES, 2)
  OUTLETS_SM_CASE(256, EPI_SLICES, 1)
  OUTLETS_SM_CASE(128, EPI_SLICES, 2)
  OUTLETS_SM_CASE(128, EPI_SLICES, 1)
  OUTLETS_SM_CASE(256, EPI_SWIGLU, 2)
  OUTLETS_SM_CASE(256, EPI_SWIGLU, 1)
  OUTLETS_SM_CASE(192, EPI_SWIGLU, 2)  // 4 slots of 56 KB
  OUTLETS_SM_CASE(192, EPI_SWIGLU, 1)
  OUTLETS_SM_CASE(128, EPI_SWIGLU, 2)
  OUTLETS_SM_CASE(128, EPI_SWIGLU, 1)
  // draft LM head: tile widths the host's wave model chooses from
  OUTLETS_SM_CASE(256, EPI_LM8, 2)
  OUTLETS_SM_CASE(256, EPI_LM8, 1)
  OUTLETS_SM_CASE(224, EPI_LM8, 2)
  OUTLETS_SM_CASE(224, EPI_LM8, 1)
  OUTLETS_SM_CASE(128, EPI_LM8, 2)
  OUTLETS_SM_CASE(128, EPI_LM8, 1)
  OUTLETS_SM_CASE(256, EPI_LM1, 2)
  OUTLETS_SM_CASE(256, EPI_LM1, 1)
  OUTLETS_SM_CASE(224, EPI_LM1, 2)
  OUTLETS_SM_CASE(224, EPI_LM1, 1)
  OUTLETS_SM_CASE(128, EPI_LM1, 2)
  OUTLETS_SM_CASE(128, EPI_LM1, 1)
#undef OUTLETS_SM_CASE
  return cudaErrorInvalidValue;
}

cudaError_t gemm_tc_launch(const CUtensorMap a_maps[3], int bn, int epi, int mt, const GemmArgs& args, int num_sms,
                           cudaStream_t stream) {
#define OUTLETS_TC_CASE(BNV, EV, MTV) \
  if (bn == BNV && epi == EV && mt == MTV) return launch_one<BNV, EV, MTV>(a_maps, args, num_sms, stream);
  // large M (prefill): one 128-row sub-tile per tile, two TMEM accumulators
  OUTLETS_TC_CASE(256, EPI_F32, 1)
  OUTLETS_TC_CASE(256, EPI_ACT, 1)
  OUTLETS_TC_CASE(256, EPI_SWIGLU, 1)
  // large M, 256 x 256 tiles (two 128-row MMAs per staged weight tile)
  OUTLETS_TC_CASE(256, EPI_F32, 2)
  OUTLETS_TC_CASE(256, EPI_ACT, 2)
  OUTLETS_TC_CASE(128, EPI_F32, 1)
  OUTLETS_TC_CASE(128, EPI_ACT, 1)
  OUTLETS_TC_CASE(64, EPI_F32, 1)
  OUTLETS_TC_CASE(64, EPI_ACT, 1)
  OUTLETS_TC_CASE(64, EPI_BIAS_RELU, 1)
  // small M (dynamic prediction): fused SwiGLU, one wave of tiles
  OUTLETS_TC_CASE(256, EPI_SWIGLU, 2)
  OUTLETS_TC_CASE(192, EPI_SWIGLU, 2)
  OUTLETS_TC_CASE(192, EPI_SWIGLU, 1)
  OUTLETS_TC_CASE(128, EPI_SWIGLU, 2)
  OUTLETS_TC_CASE(128, EPI_SWIGLU, 1)
#undef OUTLETS_TC_CASE
  return cudaErrorInvalidValue;
}

}  // namespace outlets
