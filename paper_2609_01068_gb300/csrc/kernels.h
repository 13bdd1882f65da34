// Internal launch interface between the C-ABI runtime (outlets.cu) and the
// kernels.  Nothing here is part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace outlets {

typedef __nv_bfloat16 bf16;

// Error bits written by kernels into the context's device error word.
enum : int {
  ERR_TIMEOUT = 1,    // a bounded wait ran out (an mbarrier phase never completed)
  ERR_BAD_INDEX = 2,  // a kernel met an index it refused to use
};

// Every prediction kernel is launched with programmatic stream serialization:
// it signals its dependents at once and runs its prologue (barrier init, TMEM
// allocation, L2 prefetch of weights) before waiting (griddepcontrol.wait) for
// the previous kernel's memory, so launch latency and prologues overlap the
// previous kernel's tail.  OUTLETS_PDL=0 in the environment turns this off.
bool pdl_enabled();

#define OUTLETS_TRY_LAUNCH(...)                \
  do {                                         \
    const cudaError_t e_launch_ = (__VA_ARGS__); \
    if (e_launch_ != cudaSuccess) return e_launch_; \
  } while (0)

template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                     Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// GEMM: C[M, N] = A[M, K] * B[N, K]^T, A optionally split along K across up to
// three separately addressed row-major matrices (the three taps of Eq. 1).
enum Epi : int {
  EPI_F32 = 0,        // out f32 = acc (+ residual f32)
  EPI_ACT = 1,        // out act (bf16 on the tensor-core path, f32 on the CUDA-core path) = acc
  EPI_SWIGLU = 2,     // B rows interleaved in blocks of 32 [gate | up]; out act = silu(g) * u
  EPI_BIAS_RELU = 3,  // out f32 = max(acc + bias, 0)
  EPI_SLICES = 6,     // small M: split-K, K split s writes its f32 partial to slice s (summed by the consumer)
  EPI_LM1 = 7,        // draft LM head (Eq. 2): per (row, N tile) softmax statistics and best column
  EPI_LM8 = 8,        // same with the 8 best columns
};

// Draft LM head partials, one entry per (row, partial tile), row-major
// [rows][tiles]; the tensor-core epilogue splits every N tile into two column
// halves, each its own partial tile (partial tile 2t + h: half h of N tile t):
//   stats: (max logit m_t, sum over the tile's columns of exp(logit - m_t))
//   top:   the tile's best (logit bits, token id) pairs, best first, up to KT
//          of them (order: larger logit, then smaller id; empty places hold
//          (-inf, INT_MAX)).  A tile may keep fewer than KT pairs: it drops
//          pairs below a lower bound of the row's KT-th best logit over the
//          whole vocabulary, which no pair of the row's top-KT falls below.
// Row bounds: kLmBoundSlots int keys per row (floats mapped so that int order
// is float order; kLmBoundInit is below every finite logit); the merge kernel
// puts its rows back to kLmBoundInit.
constexpr int kLmBoundSlots = 8;
constexpr int kLmBoundInit = (int)0x80808080;  // byte pattern 0x80: cudaMemset can write it

// B operands (weights) live in a k-block-major, pre-swizzled layout owned by the
// library: element (n, k) of a [N, K] weight is stored at
//   ((k / 64) * b_np + n) * 64 + (((k % 64) / 8) ^ (n % 8)) * 8 + k % 8
// with b_np >= every tile's last row (zero rows beyond N).  A tile of BN rows of
// one 64-wide K block is then one contiguous run of BN * 128 bytes, already in
// the 128-byte-swizzled order the tensor-core descriptors expect, loaded by one
// bulk copy.
struct GemmArgs {
  int M, N, K;
  const void* b;          // weights, layout above
  long long b_np;         // padded rows per K block
  int k_per_map;          // K extent of each A piece (multiple of 64 when pieces > 1)
  int splits;             // split-K factor (small-M kernel); 1 for the persistent kernel
  int group_m;            // tile raster: M blocks per group
  int prefetch;           // K blocks of B to prefetch into L2 ahead of the smem ring (0 = off)
  long long group_stride; // small-M split-K: elements between the f32 slices of consecutive K splits
  void* out;
  long long ldo;          // elements
  const float* residual;  // EPI_F32 only, may be null
  long long ldr;
  const float* bias;      // EPI_BIAS_RELU
  int* err;
  float* lm_logits;       // EPI_LM*: optional f32 logits [M, N] with row stride ldo (null: not stored)
  float2* lm_stats;       // EPI_LM*: partials [M][tiles], layout above
  int2* lm_top;           // EPI_LM*: partials [M][tiles][KT]
  // RMSNorm folded into the GEMMs (large-M path): a producer (EPI_F32) also
  // writes its output rows as bf16 (nrm_out, row stride ldo) and each row's
  // sum of squares per 64-column group (nrm_ss [M][nrm_tiles]); a consumer (EPI_ACT,
  // EPI_SWIGLU) whose A operand is such a bf16 copy and whose weights carry
  // the norm gain scales row r by rsqrt(sum_t row_ss[r][t] / nrm_d + nrm_eps).
  bf16* nrm_out;
  float* nrm_ss;
  const float* row_ss;
  int nrm_tiles, nrm_d;
  float nrm_eps;
  int* lm_bound;          // EPI_LM8: [M][kLmBoundSlots] per-row slots bounding the row's 8th best logit (int keys)
};

// tcgen05 path (bf16 operands).  a_maps: 3 tensor maps over the A pieces (box
// 64 x 128).  mt: 128-row sub-tiles per tile (1 or 2).  grid = min(tiles, num_sms).
cudaError_t gemm_tc_launch(const CUtensorMap a_maps[3], int bn, int epi, int mt, const GemmArgs& args, int num_sms,
                           cudaStream_t stream);

// Small-M GEMM (M <= 128 * mt): one output tile and one K split per CTA.
//   epi == EPI_SWIGLU: args.splits == 1, fused SwiGLU epilogue (bf16 out).
//   epi == EPI_SLICES: args.splits balanced K splits per tile; split s writes
//     its f32 partial [M, N] to out + s * group_stride (N % 4 == 0).
cudaError_t gemm_small_launch(const CUtensorMap a_maps[3], int bn, int epi, int mt, const GemmArgs& args,
                              cudaStream_t stream);

// Draft LM head, CUDA-core path: partials of tiles of tile_w columns from f32
// logits [rows, V] (row stride ld); kt is 1 or 8.
cudaError_t lm_tile_stats_f32_launch(const float* logits, long long ld, int rows, int V, int tile_w, int kt,
                                     float2* stats, int2* top, cudaStream_t stream);

// Draft LM head: combines the n_tiles partials of each row into the row's
// logsumexp and its k (<= kt) best tokens with their log-probabilities
// (ids, logprob: [rows, k]; lse: [rows] or null) and resets the rows' bound
// slots to kLmBoundInit (bound may be null).  n_tiles <= 4096.
cudaError_t lm_merge_launch(const float2* stats, const int2* top, int n_tiles, int kt, int rows, int k, int* ids,
                            float* logprob, float* lse, int* bound, cudaStream_t stream);

// CUDA-core path of the f32 configuration.  a[0..2]: A pieces with row stride k_per_map.
cudaError_t gemm_simt_f32_launch(const float* const a[3], const float* b, int epi, const GemmArgs& args,
                                 cudaStream_t stream);

// ---------------------------------------------------------------- elementwise
// y[r] = x[r] * g * rsqrt(mean(x[r]^2) + eps); optionally copy x[r] into copy_out[r].
template <typename Act>
cudaError_t rmsnorm_launch(const float* x, const float* g, Act* y, float* copy_out, int rows, int d, float eps,
                           cudaStream_t stream);

// y[i] = norm(x[row_index[i]]).
template <typename Act>
cudaError_t rmsnorm_gather_launch(const float* x, const int* row_index, const float* g, Act* y, int rows, int d,
                                  float eps, cudaStream_t stream);

// v[i] = residual[src] + sum_s x[s * split_stride + src], src = row_index ? row_index[i] : i;
// y[i] = norm(v[i]) * g; copy_out[i] = v[i] when copy_out is given.
template <typename Act>
cudaError_t rmsnorm_reduce_launch(const float* x, int n_split, long long split_stride, const float* residual,
                                  const int* row_index, const float* g, Act* y, float* copy_out, int rows, int d,
                                  float eps, cudaStream_t stream, bool discard = false);

// Input-embedding branch: y[r] = RMSNorm(table[tokens[r]]) * g (table [vocab, d],
// row-major, act dtype); an id outside [0, vocab) sets ERR_BAD_INDEX in *err.
template <typename Act>
cudaError_t embed_rmsnorm_launch(const int* tokens, const Act* table, int vocab, const float* g, Act* y, int rows,
                                 int d, float eps, int* err, cudaStream_t stream);

struct RopeArgs {
  int T;                 // rows of this launch (rows row0 .. row0 + T - 1 of the call)
  int row0;              // first row (a prefill call may run its rows in chunks)
  int H, KVH, hd;
  const int* cu;         // prefill: sequence offsets [B+1] (position = row - cu[b]); else null
  int B;
  const int* pos;        // step: position of each row; else null
  const float* cos_tab;  // [max_pos, hd/2]
  const float* sin_tab;
  int max_pos;
  void* q_out;           // [T, H, hd], or null: q heads are skipped (keys/values only)
  void* k_out;           // head-major [KVH, kv_ld_rows, hd] or null
  void* v_out;
  long long kv_ld_rows;
  void* k_pool;          // paged cache [pages][KVH][page_tokens][hd] or null
  void* v_pool;
  const int* page_list;  // pages of each sequence/request, concatenated
  const int* page_off;   // [B+1] (prefill: per sequence; step: per row)
  int page_tokens;
  int n_split;           // qkv holds n_split slices (split-K partial sums) to add up
  long long split_stride;
  int qkv_ld;            // elements per qkv row: (H + 2 KVH) hd, + H hd gate columns when gated
  void* gate_out;        // gated attention: [T, H*hd] sigmoid of the gate columns, else null
  int* err;
  bool discard;          // f32 slices: drop each row's slice lines from L2 after reading them
};
template <typename In, typename Act>
cudaError_t rope_scatter_launch(const In* qkv, const RopeArgs& a, cudaStream_t stream);

// u[r, j] = silu(gu[r, gate(j)]) * gu[r, up(j)], gu interleaved in blocks of 32.
template <typename Act>
cudaError_t swiglu_launch(const float* gu, Act* u, int rows, int f_pad, cudaStream_t stream);

// h[r] = sum_s h_pre[s * split_stride + r]; z[r] = w_last . a(h[r]) + b_last with
// a(x) = relu(x + b_prev) (identity if b_prev is null); len[r] = max(0, expm1(z[r])).
cudaError_t head_tail_launch(const float* h_pre, int n_split, long long split_stride, const float* b_prev,
                             const float* w_last, const float* b_last, int rows, int width, float* z, float* len,
                             cudaStream_t stream, bool discard = false);

// dst[r] = src[idx[r]] for r < rows: rows of row_bytes bytes (a multiple of 16,
// 16-byte aligned rows).
cudaError_t gather_rows_launch(const void* src, const int* idx, void* dst, int rows, long long row_bytes,
                               cudaStream_t stream);

// dst row map(row_base + r) <- src row r (f32 -> Act); map: row_mode 0 identity,
// 1 gate rows, 2 up rows of the [gate 32 | up 32] interleave.  kb_np == 0:
// row-major with row stride dst_ld; kb_np > 0: the k-block-major swizzled
// weight layout of GemmArgs with b_np = kb_np.
template <typename Act>
cudaError_t convert_rows_launch(const float* src, Act* dst, int rows, int cols, long long dst_ld, int row_mode,
                                int row_base, long long kb_np, const float* col_scale, cudaStream_t stream);

// One CTA whose bounded mbarrier wait can never complete: raises ERR_TIMEOUT in err.
cudaError_t wait_selftest_launch(int* err, unsigned long long timeout_ns, cudaStream_t stream);

// ---------------------------------------------------------------- attention
// k/v head-major [KVH, kv_ld, hd]; q/out [n_rows, H, hd]; gate (or null) [n_rows, H*hd]
// multiplies the output elementwise (gated attention).
template <typename Act>
cudaError_t attn_prefill_simt_launch(const Act* q, const Act* k, const Act* v, const int* cu, int B, int n_rows,
                                     int kv_ld, int H, int KVH, int hd, Act* out, const Act* gate,
                                     cudaStream_t stream);

// tcgen05 flash attention of the static pass.  A work item: one 128-row query
// tile (rows q_start .. q_start + q_len - 1 of the pack, q_len <= 128) of the
// sequence [seq_start, seq_start + seq_len) for one query head; n_kv = number
// of 128-key tiles it attends to (the last one is the diagonal tile);
// v_start = the sequence's first column in V^T (a multiple of 8).
// One work item: q_len query rows from row q_start of q (positions q_pos0 ..
// q_pos0 + q_len - 1 of their sequence) against keys 0 .. 128 n_kv - 1 of the
// sequence at rows seq_start.. of K; keys past a row's position are masked,
// which the kernel does on the last key tile only.
struct TcAttnItem {
  int q_start, q_len, seq_start, seq_len, v_start, head, n_kv, q_pos0;
};
// q_map over q [rows, H*hd] (box 64 x 128), k_map over head-major K
// [KVH * kv_ld, hd] (box 64 x 128), vt_map over V^T [KVH * hd, vt_ld] (box
// 64 x hd).  Persistent: min(n_items, num_sms) CTAs.  hd in {64, 128}.
cudaError_t attn_prefill_tc_launch(const CUtensorMap& q_map, const CUtensorMap& k_map, const CUtensorMap& vt_map,
                                   const TcAttnItem* items, int n_items, int kv_ld, int H, int KVH, int hd, void* out,
                                   const void* gate, int* err, int num_sms, cudaStream_t stream);
// V^T [KVH * hd, vt_ld] from head-major V [KVH, kv_ld, hd]; token t of sequence b
// (cu[b] <= t < cu[b+1]) goes to column v_start[b] + t - cu[b].
cudaError_t v_transpose_launch(const void* vh, const int* cu, const int* v_start, int B, int T, int kv_ld, int KVH,
                               int hd, void* vt, long long vt_ld, cudaStream_t stream);

struct DecodeArgs {
  int B, H, KVH, hd;
  const void* q;          // [B, H, hd]
  const void* k_pool;     // [pages][KVH][page_tokens][hd]
  const void* v_pool;
  int page_tokens;
  const int* page_list;   // concatenated page ids of every request
  const int* page_off;    // [B+1] offsets into page_list
  // first K/V row of page p for kv head g: p * page_stride + g * head_stride
  // (cache pools: KVH * 64 and 64; head-major [KVH, kv_ld, hd] buffers, with
  // page ids that are row offsets: 1 and kv_ld)
  long long page_stride;
  int head_stride;
  const int* seq_len;     // [B] keys per request (cached + the new token)
  const int* work;        // [n_work] pairs (request, split), grouped by request
  const int* work_off;    // [B+1] first work item of each request
  const int* order;       // [n_work] launch order of the work items (longest first), or null
  int n_work;
  int split_len;          // keys per split (multiple of page_tokens)
  int max_splits;         // most splits of one request
  float* part_o;          // [n_work, H, hd] normalized partial outputs
  float* part_ml;         // [n_work, H, 2] (max in log2 units, sum)
  int* combine_count;     // [B, KVH] split completion counters, zero between calls
  void* out;              // [B, H, hd]
  const void* gate;       // [B, H*hd] elementwise output gate (gated attention) or null
  int* err;
};
cudaError_t attn_decode_bf16_launch(const CUtensorMap& k_map, const CUtensorMap& v_map, const DecodeArgs& a,
                                    cudaStream_t stream);
template <typename Act>
cudaError_t attn_decode_simt_launch(const DecodeArgs& a, cudaStream_t stream);

}  // namespace outlets
