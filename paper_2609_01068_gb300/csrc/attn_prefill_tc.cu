// Causal GQA self-attention of the static-prediction pass (the draft decoder's
// self-attention, Sec. 4.1) on the tcgen05 tensor cores:
// o = softmax(q k^T / sqrt(hd) + causal mask) v per packed sequence, q-head h
// reading kv-head floor(h * KVH / H), optionally gated (o * gate).
//
// Persistent kernel, one CTA per SM, 8 + 4 kParts warps.  A work item is one 128-row
// query tile of one sequence x one query head; items are taken longest first
// (most key tiles) with a grid stride.
//   warps 0, 2   TMA producers, one thread each: Q tiles (two buffers) and
//                K tiles of 128 keys (warp 0), V^T tiles (warp 2), in rings of
//                their own (a K stage is freed by its S, a V stage by its PV),
//                continuously across items
//   warp 1       TMEM owner; one thread issues the S MMAs
//                  S_j = Q K_j^T     M=128 N=128 K=hd, into one of two TMEM S buffers
//                as soon as their inputs are there (S_{j+2} once PV_j has
//                completed), so the next scores are computed while the
//                softmax of this tile runs
//   warp 3       one thread issues the PV MMAs
//                  O  += P_j V_j     M=128 N=hd K=128, into O[item & 1] in TMEM
//                as soon as the softmax releases P_j
//   warps 4..    softmax, kParts threads per query row (TMEM lane), each
//                over a part of the tile's keys: the scores are read from TMEM
//                once into registers; the parts exchange their maxima of the
//                masked raw scores through shared memory; P = exp2(s - m) is
//                written as bf16 pairs back into the S buffer it came from
//                (the PV MMA reads its A operand from TMEM, so P is
//                double-buffered with S and PV_j overlaps the softmax of the
//                next tile); O and l are rescaled in place only when a row max
//                grows by more than 2^8 over the one in use (the result is
//                exact either way)
//   last 4 warps epilogue: O / l (x gate) of item k as bf16 from O[k & 1],
//                while the softmax and the MMAs run item k + 1
// V is read through a transposed copy V^T [KVH*hd, columns] (keys contiguous)
// so both MMAs take K-major operands; each sequence starts at a column that is
// a multiple of 8 (TMA coordinates in 16-byte units).  Every wait is bounded.
#include "common.cuh"
#include "kernels.h"

namespace outlets {
namespace {

constexpr int kBQ = 128;                         // query rows per work item
constexpr int kBK = 128;                         // keys per K/V tile
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescaleLog2 = 8.f;              // tolerated growth of a row max before O is rescaled
constexpr int kMaxLanes = 8;                     // independent partial maxima of a score row
// Threads of a query row in the softmax (each over kBK / kParts keys of a tile)
#ifndef OUTLETS_ATTN_PARTS
#define OUTLETS_ATTN_PARTS 2
#endif
constexpr int kParts = OUTLETS_ATTN_PARTS;
static_assert(kParts == 2 || kParts == 4, "softmax parts of a row");
constexpr int kSoftmaxWarps = 4 * kParts;
constexpr int kEpiWarp0 = 4 + kSoftmaxWarps;    // first epilogue warp
// Q/K producer, S issuer, V producer, PV issuer, the softmax warps, 4 epilogue warps
constexpr int kThreads = 32 * (4 + kSoftmaxWarps + 4);
constexpr int kSoftmaxThreads = 32 * kSoftmaxWarps;

__device__ __forceinline__ void tmem_st_32x32b_x16(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};"
      ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// 2^x with the hardware approximation (ex2.approx.ftz: -inf -> 0); the result
// is rounded to bf16 or divided out by the row sum, far coarser than its error.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int HD>
struct TcAttnCfg {
  static constexpr int NB = HD / 64;                   // 64-wide blocks of a head
  static constexpr uint32_t Q_BYTES = kBQ * HD * 2;    // [NB][128 rows][64]
  static constexpr uint32_t K_BYTES = kBK * HD * 2;    // [NB][128 keys][64]
  static constexpr uint32_t V_BYTES = HD * kBK * 2;    // V^T: [2][hd rows][64 keys]
  // Q buffers and K/V stages share the 227 KB; a second Q buffer lets the
  // first S of an item start while the previous item's last S runs
  static constexpr int NQ = 2;
  static constexpr uint32_t BAR_BYTES = 512;          // mbarriers, TMEM address, abort flag
  static constexpr uint32_t L_BYTES = 2 * kParts * kBQ * 4;  // row sums: [O buffer][part of the keys][row]
  static constexpr uint32_t X_BYTES = kParts * kBQ * 8;      // row max exchange: [part of the keys][row] x (max, ok)
  // K and V^T stages in what is left: as many of each as fit, one more K
  // stage where it fits (a K stage is held from its load to its S, a V
  // stage from its load to its PV, later)
  static constexpr uint32_t KV_BUDGET = 232448u - 1024u - BAR_BYTES - L_BYTES - X_BYTES - NQ * Q_BYTES;
  static constexpr int NV_FIT = (int)(KV_BUDGET / (K_BYTES + V_BYTES));
  static constexpr int NV = NV_FIT > 6 ? 6 : NV_FIT;
  static constexpr int NK = (NV < 6 && KV_BUDGET - NV * (K_BYTES + V_BYTES) >= K_BYTES) ? NV + 1 : NV;
  static constexpr size_t SMEM =
      1024 + NQ * Q_BYTES + NK * K_BYTES + NV * V_BYTES + BAR_BYTES + L_BYTES + X_BYTES;
  static_assert(NV >= 2 && NK >= 2, "K/V stages");
  // TMEM: S0 [0,128), S1 [128,256), O0 [256, 256+hd), O1 [256+hd, 256+2hd)
  static constexpr uint32_t O_COL = 2 * kBK;
  static_assert(O_COL + 2 * HD <= 512, "TMEM columns");
  static_assert(SMEM <= 232448, "shared memory");
};

template <int HD>
__global__ void __launch_bounds__(kThreads, 1)
    k_attn_prefill_tc(const __grid_constant__ CUtensorMap q_map, const __grid_constant__ CUtensorMap k_map,
                      const __grid_constant__ CUtensorMap vt_map, const TcAttnItem* __restrict__ items,
                      int n_items, int kv_ld, int H, int KVH, bf16* __restrict__ out, const bf16* __restrict__ gate,
                      int* err) {
  using C = TcAttnCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  constexpr int NQ = C::NQ, NK = C::NK, NV = C::NV;
  uint8_t* sQ = smem;                     // NQ buffers
  uint8_t* sK = sQ + NQ * C::Q_BYTES;     // NK stages
  uint8_t* sV = sK + NK * C::K_BYTES;     // NV stages
  uint64_t* q_full = reinterpret_cast<uint64_t*>(sV + NV * C::V_BYTES);
  uint64_t* q_empty = q_full + NQ;
  // K and V^T stages have their own rings: a K stage is free once its S is
  // computed, a V stage once its PV is (long before, in the K case)
  uint64_t* k_full = q_empty + NQ;
  uint64_t* k_empty = k_full + NK;
  uint64_t* v_full = k_empty + NK;
  uint64_t* v_empty = v_full + NV;
  uint64_t* s_full = v_empty + NV;
  uint64_t* p_full = s_full + 2;
  uint64_t* pv_done = p_full + 1;
  // O is double-buffered in TMEM: item k accumulates into O[k & 1] while the
  // epilogue warps store item k - 1 from the other buffer
  uint64_t* o_full = pv_done + 1;   // [2] last PV of the item complete
  uint64_t* o_empty = o_full + 2;   // [2] the epilogue has read O and l
  uint64_t* l_full = o_empty + 2;   // [2] the softmax has written the row sums
  // PV_n complete, for the S issuer (S_{n+2} overwrites the buffer P_n is read
  // from): two barriers, n & 1, so that neither runs two phases ahead of it
  uint64_t* pv_free = l_full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(pv_free + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* l_buf = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(q_full) + C::BAR_BYTES);  // [2][kParts][128]
  float2* m_xchg = reinterpret_cast<float2*>(l_buf + 2 * kParts * kBQ);  // [kParts][128]: partial max, wait status
  static_assert((2 * NQ + 2 * NK + 2 * NV + 12) * 8 + 8 <= (int)C::BAR_BYTES, "barrier area");
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < NQ; ++i) {
      mbar_init(&q_full[i], 1);
      mbar_init(&q_empty[i], 1);
    }
    for (int i = 0; i < NK; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
    }
    for (int i = 0; i < NV; ++i) {
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&o_full[i], 1);
      mbar_init(&o_empty[i], 4 * 32);
      mbar_init(&l_full[i], kSoftmaxThreads);
      mbar_init(&pv_free[i], 1);
    }
    mbar_init(p_full, kSoftmaxThreads);
    mbar_init(pv_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&q_map);
    tma_prefetch_map(&k_map);
    tma_prefetch_map(&vt_map);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_trigger();
  pdl_wait();  // q, k and V^T are written by the kernels before this one

  if (warp == 0) {
    if (lane == 0) {
      // Q and K producer: each item's Q (into buffer k % NQ, once the last S
      // of item k - NQ has read it), then its K tiles into the K ring (a
      // stage once the S that read it has completed).  It blocks in its
      // waits, which leaves the issue slots to the softmax warps of this SM
      // sub-partition (a polling producer delayed them).
      int g = 0;  // key tiles of this CTA
      int k = 0;  // items of this CTA
      for (int it = blockIdx.x; it < n_items; it += gridDim.x, ++k) {
        const TcAttnItem w = items[it];
        const int kvh = (w.head * KVH) / H;
        const int qb = k % NQ;
        bool ok = k < NQ || mbar_wait(&q_empty[qb], ((k - NQ) / NQ) & 1, abort_flag, err);
        if (!ok) break;
        mbar_arrive_expect_tx(&q_full[qb], C::Q_BYTES);
#pragma unroll
        for (int b = 0; b < C::NB; ++b)
          tma_load_2d(sQ + qb * C::Q_BYTES + b * (kBQ * 128), &q_map, &q_full[qb], w.head * HD + 64 * b, w.q_start);
        for (int j = 0; j < w.n_kv; ++j, ++g) {
          const int st = g % NK;
          ok = g < NK || mbar_wait(&k_empty[st], ((g - NK) / NK) & 1, abort_flag, err);
          if (!ok) break;
          mbar_arrive_expect_tx(&k_full[st], C::K_BYTES);
#pragma unroll
          for (int b = 0; b < C::NB; ++b)
            tma_load_2d(sK + st * C::K_BYTES + b * (kBK * 128), &k_map, &k_full[st], 64 * b,
                        kvh * kv_ld + w.seq_start + kBK * j);
        }
        if (!ok) break;
      }
    }
  } else if (warp == 2) {
    if (lane == 0) {
      // V^T producer: the V^T tiles into the V ring (a stage once the PV
      // that read it has completed), blocking like the Q and K producer
      int g = 0;
      for (int it = blockIdx.x; it < n_items; it += gridDim.x) {
        const TcAttnItem w = items[it];
        const int kvh = (w.head * KVH) / H;
        bool ok = true;
        for (int j = 0; j < w.n_kv; ++j, ++g) {
          const int st = g % NV;
          ok = g < NV || mbar_wait(&v_empty[st], ((g - NV) / NV) & 1, abort_flag, err);
          if (!ok) break;
          mbar_arrive_expect_tx(&v_full[st], C::V_BYTES);
#pragma unroll
          for (int b = 0; b < 2; ++b)
            tma_load_2d(sV + st * C::V_BYTES + b * (HD * 128), &vt_map, &v_full[st], w.v_start + kBK * j + 64 * b,
                        kvh * HD);
        }
        if (!ok) break;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // S issuer: S_n = Q K_n^T (M=128 N=128 K=hd) into TMEM buffer n & 1, as
      // soon as the item's Q, K tile n and the buffer are there (the PV that
      // read P_{n-2} from it complete).  The PV issuer is another thread: the
      // issue of an MMA blocks while the pipe's short queue is full, and a PV
      // the softmax waits for does not queue behind the issue of an S.
      constexpr uint32_t id_s = idesc_bf16_f32(kBQ, kBK);
      int g = 0;  // key tiles of this CTA
      int k = 0;  // items of this CTA
      for (int it = blockIdx.x; it < n_items; it += gridDim.x, ++k) {
        const int nkv = items[it].n_kv;
        const int qb = k % NQ;
        bool ok = mbar_wait(&q_full[qb], (k / NQ) & 1, abort_flag, err);
        for (int j = 0; ok && j < nkv; ++j, ++g) {
          const int st = g % NK;
          const int sb = g & 1;
          ok = mbar_wait(&k_full[st], (g / NK) & 1, abort_flag, err) &&
               (g < 2 || mbar_wait(&pv_free[sb], ((g - 2) >> 1) & 1, abort_flag, err));
          if (!ok) break;
          tc_fence_after();
          const uint32_t qa = smem_u32(sQ + qb * C::Q_BYTES);
          const uint32_t ka = smem_u32(sK + st * C::K_BYTES);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (128 * 128);
            tc_mma_bf16(tmem_base + sb * kBK, sw128_kmajor_desc(qa + off) + 2u * (kk & 3),
                        sw128_kmajor_desc(ka + off) + 2u * (kk & 3), id_s, kk > 0 ? 1u : 0u);
          }
          tc_commit(&s_full[sb]);
          tc_commit(&k_empty[st]);                      // S_n has read its K tile
          if (j == nkv - 1) tc_commit(&q_empty[qb]);  // last S of the item: its Q buffer is free
        }
        if (!ok) break;
      }
    }
  } else if (warp == 3) {
    if (lane == 0) {
      // PV issuer: O[item & 1] += P_n V_n (M=128 N=hd K=128, A = P in TMEM)
      // once the softmax has released P_n and V tile n is there; the first PV
      // of an item overwrites O[k & 1], which the epilogue must have read
      // (item k - 2)
      constexpr uint32_t id_o = idesc_bf16_f32(kBQ, HD);
      int g = 0;
      int k = 0;
      for (int it = blockIdx.x; it < n_items; it += gridDim.x, ++k) {
        const int nkv = items[it].n_kv;
        const int ob = k & 1;
        bool ok = k < 2 || mbar_wait(&o_empty[ob], ((k - 2) >> 1) & 1, abort_flag, err);
        for (int j = 0; ok && j < nkv; ++j, ++g) {
          const int st = g % NV;
          const int sb = g & 1;  // TMEM buffer holding P
          ok = mbar_wait(p_full, g & 1, abort_flag, err) && mbar_wait(&v_full[st], (g / NV) & 1, abort_flag, err);
          if (!ok) break;
          tc_fence_after();
          const uint32_t va = smem_u32(sV + st * C::V_BYTES);
          // A = P in TMEM (the S buffer it was computed in: 16 keys = 8 columns per MMA)
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)
            tc_mma_bf16_ta(tmem_base + C::O_COL + ob * HD, tmem_base + sb * kBK + 8 * kk,
                           sw128_kmajor_desc(va + (kk >> 2) * (HD * 128)) + 2u * (kk & 3), id_o,
                           (j > 0 || kk > 0) ? 1u : 0u);
          tc_commit(pv_done);
          tc_commit(&pv_free[sb]);
          tc_commit(&v_empty[st]);                   // PV_n has read its V tile
          if (j == nkv - 1) tc_commit(&o_full[ob]);  // the item's O is complete
        }
        if (!ok) break;
      }
    }
  } else if (warp >= 4 && warp < kEpiWarp0) {
    // softmax warps 4 .. 4 + 4 kParts - 1: kParts per TMEM lane quarter (a
    // warp reaches lanes 32 * (warp % 4) ..); thread = one query row x one
    // part of the tile's 128 keys (part p: warps 4 + 4p .. 7 + 4p).  The
    // threads of a row exchange their partial maxima, so all scale P by the
    // same m, and keep their own parts of the row sum.
    const int quarter = warp & 3;
    const int part = (warp - 4) >> 2;
    const int r = quarter * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const float sl2 = rsqrtf((float)HD) * kLog2e;
    constexpr int KH = kBK / kParts;  // keys of a tile per thread
    // Exchange with the row's other threads (named barrier 1 + quarter, the
    // 32 kParts threads of the quarter's warps): the row max over all parts.
    // A failed bounded wait travels with the value; all threads of every row
    // then leave together, so that no thread waits at a barrier a partner
    // has left.  good is kept uniform over the warp (the tcgen05 loads and
    // stores are warp-wide).
    auto exchange = [&](float mine, bool& good) -> float {
      tc_fence_before();
      m_xchg[part * kBQ + r] = make_float2(mine, good ? 1.f : 0.f);
      asm volatile("bar.sync %0, %1;" ::"r"(1 + quarter), "r"(32 * kParts) : "memory");
      tc_fence_after();
      float m = mine;
      bool all_ok = good;
#pragma unroll
      for (int q = 0; q < kParts; ++q) {
        const float2 other = m_xchg[q * kBQ + r];
        m = fmaxf(m, other.x);
        all_ok = all_ok && other.y != 0.f;
      }
      asm volatile("bar.sync %0, %1;" ::"r"(1 + quarter), "r"(32 * kParts) : "memory");  // all have read before any writes again
      good = __all_sync(0xffffffffu, all_ok);
      return m;
    };
    int g = 0;  // key tiles of this CTA
    int k = 0;  // items of this CTA
    bool good = true;
    for (int it = blockIdx.x; it < n_items; it += gridDim.x, ++k) {
      const TcAttnItem w = items[it];
      const int ob = k & 1;         // O buffer of this item
      const int qp = w.q_pos0 + r;  // position of this row in its sequence
      float m_used = -INFINITY, l = 0.f;
      bool stop = false;
      for (int j = 0; j < w.n_kv; ++j, ++g) {
        const int sb = g & 1;
        if (good) good = mbar_wait(&s_full[sb], (g >> 1) & 1, abort_flag, err);
        good = __all_sync(0xffffffffu, good);
        const uint32_t s_addr = tmem_base + lane_off + static_cast<uint32_t>(sb * kBK);
        const bool diag = j == w.n_kv - 1;
        const int key0 = kBK * j + KH * part;
        uint32_t v[KH];
        float mx = -INFINITY;
        if (good) {
          tc_fence_after();
          // this part of the row's scores into registers: KH / 32 loads, one wait
#pragma unroll
          for (int c = 0; c < KH / 32; ++c) tmem_ld_32x32b_x32(s_addr + KH * part + 32 * c, v + 32 * c);
          tmem_ld_wait();
          // row max on the raw scores (the scale is positive); the causal
          // mask only applies on the diagonal tile (key > query position).
          // Independent partial maxima: one chain of dependent max operations
          // would sit in front of every exponential of the tile.
          if (diag) {
#pragma unroll
            for (int e = 0; e < KH; ++e)
              if (key0 + e > qp) v[e] = __float_as_uint(-INFINITY);
          }
          float mp[kMaxLanes];
#pragma unroll
          for (int i = 0; i < kMaxLanes; ++i) mp[i] = __uint_as_float(v[i]);
#pragma unroll
          for (int e = kMaxLanes; e < KH; e += kMaxLanes)
#pragma unroll
            for (int i = 0; i < kMaxLanes; ++i) mp[i] = fmaxf(mp[i], __uint_as_float(v[e + i]));
#pragma unroll
          for (int w2 = kMaxLanes / 2; w2 > 0; w2 >>= 1)
#pragma unroll
            for (int i = 0; i < w2; ++i) mp[i] = fmaxf(mp[i], mp[i + w2]);
          mx = mp[0];
        }
        // the row max over all parts; every part has read its scores before
        // any writes P over them below
        const float mo = exchange(mx, good);
        if (!good) {
          stop = true;
          break;
        }
        const float mrow = mo * sl2;  // in the log2 domain of the exponentials
        float alpha = 1.f;
        bool resc = false;
        if (mrow > m_used + kRescaleLog2) {
          alpha = (m_used == -INFINITY) ? 0.f : ex2_approx(m_used - mrow);
          l *= alpha;
          m_used = mrow;
          resc = j > 0;
        }
        // P = exp2(s - m) as bf16 pairs, this part's KH / 2 columns of the
        // first 64 of the buffer.  The row sum adds the f32 values before rounding:
        // the bf16 weights the PV product uses then sum to l within a relative
        // 2^-9 / sqrt(keys), below the bf16 rounding of the output.
        uint32_t pk[KH / 2];
        float psum[4] = {0.f, 0.f, 0.f, 0.f};  // partial sums, for the same reason as the maxima
#pragma unroll
        for (int e = 0; e < KH; e += 2) {
          const float p0 = ex2_approx(fmaf(__uint_as_float(v[e]), sl2, -m_used));
          const float p1 = ex2_approx(fmaf(__uint_as_float(v[e + 1]), sl2, -m_used));
          pk[e >> 1] = pack_bf16x2(p0, p1);
          psum[(e >> 1) & 3] += p0 + p1;
        }
        const float ps = (psum[0] + psum[1]) + (psum[2] + psum[3]);
        if constexpr (KH / 2 == 32) {
          tmem_st_32x32b_x32(s_addr + (KH / 2) * part, pk);
        } else {
          tmem_st_32x32b_x16(s_addr + (KH / 2) * part, pk);
        }
        // The previous PV (of this item, or the last of the previous one) must
        // be complete before this tile's P is released, and before O is
        // rescaled.  Every release waits for it, the first tile of an item
        // too: no thread's arrival for tile g can then reach the P barrier
        // before every thread's arrival for tile g - 1 (which the PV of g - 1
        // needs), and the PV barrier never runs two phases ahead of a thread.
        if (g > 0) good = __all_sync(0xffffffffu, mbar_wait(pv_done, (g - 1) & 1, abort_flag, err));
        if (good) {
          tc_fence_after();
          if (__any_sync(0xffffffffu, resc)) {
            // rare: this part's hd / kParts columns of O (whole 32-column
            // chunks, over the parts in turn)
            const float a = resc ? alpha : 1.f;
#pragma unroll 1
            for (int c = part; c < HD / 32; c += kParts) {
              uint32_t o[32];
              const uint32_t o_addr = tmem_base + lane_off + C::O_COL + ob * HD + 32 * c;
              tmem_ld_32x32b_x32(o_addr, o);
              tmem_ld_wait();
#pragma unroll
              for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * a);
              tmem_st_32x32b_x32(o_addr, o);
            }
          }
          tmem_st_wait();
          l += ps;
          tc_fence_before();
          mbar_arrive(p_full);
        }
      }
      if (stop) break;  // both halves, at the same exchange
      // end of the item: this part's row sum goes to the epilogue warps once
      // they have taken item k - 2's from this buffer (a failed wait reaches
      // the partner with the next item's first exchange)
      if (good && k >= 2) good = __all_sync(0xffffffffu, mbar_wait(&o_empty[ob], ((k - 2) >> 1) & 1, abort_flag, err));
      if (good) {
        l_buf[(ob * kParts + part) * kBQ + r] = l;
        mbar_arrive(&l_full[ob]);
      }
    }
  } else if (warp >= kEpiWarp0) {
    // epilogue warps (the last 4): O[k & 1] / l (x gate) as bf16, one query
    // row per thread, while the softmax warps run the next item
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    constexpr int CP = kParts > 2 ? 32 : (HD < 64 ? HD : 64);  // columns per pass (registers)
    int k = 0;
    for (int it = blockIdx.x; it < n_items; it += gridDim.x, ++k) {
      const int ob = k & 1;
      bool good = mbar_wait(&o_full[ob], (k >> 1) & 1, abort_flag, err);
      good = good && mbar_wait(&l_full[ob], (k >> 1) & 1, abort_flag, err);
      if (!__all_sync(0xffffffffu, good)) break;
      tc_fence_after();
      const TcAttnItem w = items[it];
      float lsum = 0.f;
#pragma unroll
      for (int q = 0; q < kParts; ++q) lsum += l_buf[(ob * kParts + q) * kBQ + r];
      const float inv = 1.f / lsum;
      bf16* orow = out + (long long)(w.q_start + r) * H * HD + w.head * HD;
      const bf16* grow = gate ? gate + (long long)(w.q_start + r) * H * HD + w.head * HD : nullptr;
#pragma unroll 1
      for (int c0 = 0; c0 < HD; c0 += CP) {
        uint32_t ov[CP];
#pragma unroll
        for (int c = 0; c < CP / 32; ++c)
          tmem_ld_32x32b_x32(tmem_base + lane_off + C::O_COL + ob * HD + c0 + 32 * c, ov + 32 * c);
        tmem_ld_wait();
        if (c0 + CP == HD) {  // all of O (and l) read: the buffer is free
          tc_fence_before();
          mbar_arrive(&o_empty[ob]);
        }
        if (r < w.q_len) {
#pragma unroll
          for (int c = 0; c < CP / 8; ++c) {
            const uint32_t* v = ov + 8 * c;
            float f[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) f[e] = __uint_as_float(v[e]) * inv;
            if (grow) {
              const uint4 gq = *reinterpret_cast<const uint4*>(grow + c0 + 8 * c);
              const __nv_bfloat162* gh = reinterpret_cast<const __nv_bfloat162*>(&gq);
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float2 gf = __bfloat1622float2(gh[e]);
                f[2 * e] *= gf.x;
                f[2 * e + 1] *= gf.y;
              }
            }
            *reinterpret_cast<uint4*>(orow + c0 + 8 * c) =
                make_uint4(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3]), pack_bf16x2(f[4], f[5]),
                           pack_bf16x2(f[6], f[7]));
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, 512);
  }
}

// V^T [KVH * hd, vt_ld] from head-major V [KVH, kv_ld, hd]: token t of sequence
// b goes to column v_start[b] + (t - cu[b]).  One CTA = 64 tokens of one kv head,
// staged in shared memory so that both the reads and the writes are coalesced.
template <int HD>
__global__ void __launch_bounds__(256) k_v_transpose(const bf16* __restrict__ vh, const int* __restrict__ cu,
                                                     const int* __restrict__ v_start, int B, int T, int kv_ld,
                                                     bf16* __restrict__ vt, long long vt_ld) {
  pdl_trigger();
  pdl_wait();
  constexpr int LDW = HD / 2 + 1;  // words per staged token (odd: conflict-free column reads)
  __shared__ uint32_t tile[64 * LDW];
  __shared__ int col[64];
  const int t0 = blockIdx.x * 64;
  const int g = blockIdx.y;
  if (threadIdx.x < 64) {
    const int t = t0 + threadIdx.x;
    int c = -1;
    if (t < T) {
      int lo = 0, hi = B;
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (cu[mid] <= t) lo = mid;
        else hi = mid;
      }
      c = v_start[lo] + (t - cu[lo]);
    }
    col[threadIdx.x] = c;
  }
  for (int idx = threadIdx.x; idx < 64 * (HD / 8); idx += blockDim.x) {
    const int tok = idx / (HD / 8);
    const int c8 = idx - tok * (HD / 8);
    uint4 v = make_uint4(0, 0, 0, 0);
    if (t0 + tok < T) v = *reinterpret_cast<const uint4*>(vh + ((long long)g * kv_ld + t0 + tok) * HD + c8 * 8);
    uint32_t* dst = tile + tok * LDW + c8 * 4;
    dst[0] = v.x;
    dst[1] = v.y;
    dst[2] = v.z;
    dst[3] = v.w;
  }
  __syncthreads();
  const uint16_t* t16 = reinterpret_cast<const uint16_t*>(tile);
  for (int idx = threadIdx.x; idx < HD * 64; idx += blockDim.x) {
    const int d = idx >> 6;
    const int tok = idx & 63;
    const int c = col[tok];
    if (c >= 0) {
      const uint16_t bits = t16[tok * (2 * LDW) + d];
      reinterpret_cast<uint16_t*>(vt)[((long long)g * HD + d) * vt_ld + c] = bits;
    }
  }
}

template <int HD>
cudaError_t launch_tc(const CUtensorMap& q_map, const CUtensorMap& k_map, const CUtensorMap& vt_map,
                      const TcAttnItem* items, int n_items, int kv_ld, int H, int KVH, void* out, const void* gate,
                      int* err, int num_sms, cudaStream_t stream) {
  using C = TcAttnCfg<HD>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_attn_prefill_tc<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int grid = n_items < num_sms ? n_items : num_sms;
  OUTLETS_TRY_LAUNCH(launch_k(k_attn_prefill_tc<HD>, dim3(grid), dim3(kThreads), C::SMEM, stream, q_map, k_map, vt_map,
                              items, n_items, kv_ld, H, KVH, reinterpret_cast<bf16*>(out),
                              reinterpret_cast<const bf16*>(gate), err));
  return cudaGetLastError();
}

}  // namespace

cudaError_t v_transpose_launch(const void* vh, const int* cu, const int* v_start, int B, int T, int kv_ld, int KVH,
                               int hd, void* vt, long long vt_ld, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  const dim3 grid((T + 63) / 64, KVH);
  if (hd == 128) {
    OUTLETS_TRY_LAUNCH(launch_k(k_v_transpose<128>, grid, dim3(256), 0, stream, reinterpret_cast<const bf16*>(vh), cu,
                                v_start, B, T, kv_ld, reinterpret_cast<bf16*>(vt), vt_ld));
  } else if (hd == 64) {
    OUTLETS_TRY_LAUNCH(launch_k(k_v_transpose<64>, grid, dim3(256), 0, stream, reinterpret_cast<const bf16*>(vh), cu,
                                v_start, B, T, kv_ld, reinterpret_cast<bf16*>(vt), vt_ld));
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t attn_prefill_tc_launch(const CUtensorMap& q_map, const CUtensorMap& k_map, const CUtensorMap& vt_map,
                                   const TcAttnItem* items, int n_items, int kv_ld, int H, int KVH, int hd, void* out,
                                   const void* gate, int* err, int num_sms, cudaStream_t stream) {
  if (n_items == 0) return cudaSuccess;
  if (hd == 128) return launch_tc<128>(q_map, k_map, vt_map, items, n_items, kv_ld, H, KVH, out, gate, err, num_sms, stream);
  if (hd == 64) return launch_tc<64>(q_map, k_map, vt_map, items, n_items, kv_ld, H, KVH, out, gate, err, num_sms, stream);
  return cudaErrorInvalidValue;
}

}  // namespace outlets
