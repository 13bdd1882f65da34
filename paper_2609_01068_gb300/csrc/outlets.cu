// Host runtime behind the C ABI of include/outlets.h: argument validation,
// weight upload and re-layout, the paged draft KV cache, per-call metadata
// staging and the launch sequences of static (prefill) and dynamic (step)
// prediction (Sec. 3.2).
//
// Launch sequence of one prediction call, on the caller's stream:
//   FC (Eq. 1, tcgen05 GEMM over the three taps) -> RMSNorm ->
//   QKV GEMM -> RoPE + K/V scatter (workspace and/or paged cache) ->
//   attention (varlen causal flash attention, or paged split-KV decode) ->
//   O GEMM + residual -> RMSNorm -> gate/up GEMM with fused SwiGLU ->
//   down GEMM + residual -> final RMSNorm of the predicted rows (h^draft) ->
//   head Linear+ReLU (GEMM) ... -> head output row + expm1 (Sec. 4.2).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <numeric>
#include <cstdlib>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <unordered_map>
#include <vector>

#include "kernels.h"
#include "outlets.h"

using namespace outlets;

namespace {

constexpr int kPageTokens = 64;
constexpr int kMaxTapChunks = 16;     // row chunks of host taps copied while earlier chunks compute
constexpr int kMinTapChunkRows = 1024;
constexpr int kSplitLen = 512;        // shortest split-KV work item (keys)
constexpr int kDecodeCtasPerSm = 3;   // resident decode-attention CTAs per SM
constexpr int kRing = 4;
constexpr int kMaxVocab = 262144;     // draft head: at most 2048 tiles of 128 columns per row
constexpr int kLmRowsPerPass = 256;   // draft head rows per GEMM + merge pass (one 256-row tile)
constexpr int kLmTileF32 = 256;       // draft head tile width of the f32 path

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// 2D bf16 tensor map: rows x cols (cols contiguous, row stride ld elements),
// box box_rows x 64 columns, 128-byte swizzle, zero fill outside the tensor.
bool make_map(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint64_t ld, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || rows == 0 || cols == 0) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Memo of encoded tensor maps: weights and workspace buffers are re-used by
// every call with the same shapes, so their maps are encoded once.
struct MapKey {
  const void* base;
  uint64_t cols, rows, ld;
  uint32_t box_rows;
  bool operator==(const MapKey& o) const {
    return base == o.base && cols == o.cols && rows == o.rows && ld == o.ld && box_rows == o.box_rows;
  }
};
struct MapKeyHash {
  size_t operator()(const MapKey& k) const {
    size_t h = std::hash<const void*>()(k.base);
    h ^= std::hash<uint64_t>()(k.cols * 1000003ull + k.rows * 7919ull + k.ld * 131ull + k.box_rows) + 0x9e3779b9 +
         (h << 6) + (h >> 2);
    return h;
  }
};

bool is_device_ptr(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

inline long long cdiv(long long a, long long b) { return (a + b - 1) / b; }

// K blocks of weights each small-M GEMM CTA keeps in flight toward L2 ahead of
// its shared-memory ring (OUTLETS_PREFETCH overrides; default 8).
int prefetch_blocks() {
  static const int n = [] {
    const char* v = getenv("OUTLETS_PREFETCH");
    return v ? atoi(v) : 8;
  }();
  return n;
}

// Whether the kernels that add up split-K slices drop the slices' lines from
// L2 after reading them (no write-back of scratch; OUTLETS_L2_DISCARD=0 keeps
// them, for comparison).
bool discard_slices() {
  static const bool on = [] {
    const char* v = getenv("OUTLETS_L2_DISCARD");
    return !v || atoi(v) != 0;
  }();
  return on;
}

}  // namespace

struct outlets_ctx {
  outlets_config cfg{};
  std::string err;
  int num_sms = 0;
  bool bf16 = true;
  size_t esz = 2;
  int d = 0, H = 0, KVH = 0, hd = 0, F = 0, Fp = 0, qkv_n = 0, attn_w = 0, max_rows = 0;
  bool gated = false;        // gated attention: QKV carries H*hd gate columns after q, k, v
  // input-embedding branch: table [EV, d] (act dtype, row-major), its gain, the
  // normalized embedding of each row; the QKV GEMM then has K = 2d (qkv_k)
  int EV = 0, qkv_k = 0;
  // RMSNorm folded into the GEMMs (bf16 path): g_in / g_post are folded into
  // the QKV / gate-up weights at upload, so explicit norms of f and a use unit
  // gains; on the large-M path the FC and O GEMMs also write bf16 copies and
  // per-tile sums of squares, and QKV / gate-up scale their rows
  bool fold = false;
  float* ones = nullptr;
  float *ss_f = nullptr, *ss_a = nullptr;  // [max_rows][ss_stride]
  int ss_stride = 0;
  bool xin_raw = false;          // xhat holds bf16(f), not the normalized x_hat (last call)
  int fold_tiles_f = 0;          // 64-column groups of the FC output in ss_f (its consumer needs the count)
  void* xin_scratch = nullptr;   // x_hat on request (outlets_get_intermediate)
  void* w_embed = nullptr;
  float* g_emb = nullptr;
  void* ehat = nullptr;
  // draft LM head (Eq. 2): weights, per (row, tile) partials, outputs of host callers
  int V = 0;
  void* w_lm = nullptr;
  long long np_lm = 0;
  int lm_rows_cap = 0;       // rows per GEMM + merge pass
  float2* lm_stats = nullptr;
  int2* lm_top = nullptr;
  int* lm_bound = nullptr;   // per-row slots bounding the 8th best logit (reset by the merge kernel)
  bool lm_bound_dirty = true;  // a pass may have stopped before its merge: reset before the next GEMM
  int* lm_ids = nullptr;
  float *lm_lp = nullptr, *lm_lse = nullptr;
  float* lm_logits_ws = nullptr;  // f32 path: logits of one pass
  float* lm_logits_stage = nullptr;  // host `logits` callers: one pass, copied out (allocated on first use)
  void* vt = nullptr;        // V^T [KVH * hd, vt_ld] for the tcgen05 prefill attention (bf16)
  long long vt_ld = 0;
  void* gate_act = nullptr;  // [max_rows, H*hd] sigmoid(gate), act dtype
  // static prediction of the last rows only (bf16): x_hat, the embedding
  // half of the layer input and f of each sequence's last row, [max_batch, d]
  void *last_x = nullptr, *last_e = nullptr;
  float* last_f = nullptr;
  // split-KV partials of the last rows' attention (decode attention over the
  // head-major K/V of the call): [last_part_items, H, hd] and [.., H, 2]
  float *last_part_o = nullptr, *last_part_ml = nullptr;
  size_t last_part_items = 0;
  std::vector<int> head_dims;  // d, hidden..., 1
  std::vector<void*> allocs;
  size_t dev_bytes = 0;

  void *w_proj = nullptr, *w_qkv = nullptr, *w_o = nullptr, *w_gu = nullptr, *w_down = nullptr,
       *head_w0 = nullptr;
  // padded rows per K block of each weight in the k-block-major layout (bf16 path; 0 = row-major)
  long long np_proj = 0, np_qkv = 0, np_o = 0, np_gu = 0, np_down = 0, np_h0 = 0;
  float *g_in = nullptr, *g_post = nullptr, *g_final = nullptr;
  std::vector<float*> head_wf, head_b;
  float *rope_cos = nullptr, *rope_sin = nullptr;

  float *f = nullptr, *a = nullptr, *y = nullptr, *h1a = nullptr, *h1b = nullptr, *z = nullptr, *len = nullptr,
        *gu32 = nullptr;
  void *xhat = nullptr, *ahat = nullptr, *qkv = nullptr, *q = nullptr, *kh = nullptr, *vh = nullptr,
       *attn = nullptr, *u = nullptr, *hn = nullptr;
  void* taps_stage[3] = {nullptr, nullptr, nullptr};
  int* err_dev = nullptr;
  int* dec_count = nullptr;  // [max_batch, KVH] split-KV completion counters of decode attention
  float* part = nullptr;  // f32 split-K slices of the small-M path
  size_t part_floats = 0;
  int* meta_dev = nullptr;  // device metadata of the current call (a ring slot's buffer)

  // Ring of metadata slots: pinned host staging + device buffer.  A slot is
  // reused only after the call that last used it has finished on the GPU
  // (`done`), so the upload of one call overlaps the kernels of the previous.
  struct Pin {
    int* h = nullptr;
    size_t cap = 0;
    int* dev = nullptr;
    size_t dev_cap = 0;
    cudaEvent_t ev = nullptr;    // upload complete (copy stream)
    cudaEvent_t done = nullptr;  // the call that used the slot is complete (its stream)
    bool used = false;
  } ring[kRing];
  int ring_i = 0;
  int cur_slot = -1;
  bool meta_waited = false;
  cudaEvent_t done_ev = nullptr;
  // copies of host taps in row chunks, overlapped with the prefill front
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t copy_start = nullptr;
  cudaEvent_t chunk_ev[kMaxTapChunks] = {};
  bool have_prev = false;

  int last_rows = 0, last_out_rows = 0;
  int last_tail_rows = 0;         // rows of q / attention / a / y of the last call (all rows, or the predicted ones)
  int last_kind = 0;              // 0: none, 1: prefill, 2: step or draft step (its y rows feed a draft step)
  std::vector<int> last_slots;    // slots of the last step, in row order
  bool oom = false;
  std::unordered_map<MapKey, CUtensorMap, MapKeyHash> map_cache;  // library-owned buffers only

  // stage timing and launch accounting
  struct ProfRec {
    int stage;
    cudaEvent_t a, b;
  };
  unsigned prof = 0;  // bit mask of timed stages
  int cur_stage = -1;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  std::vector<ProfRec> recs;
  unsigned long long launches = 0;
  cudaStream_t cur_stream = nullptr;

  cudaEvent_t next_event() {
    if (ev_used == ev_pool.size()) {
      cudaEvent_t e = nullptr;
      if (cudaEventCreate(&e) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
      }
      ev_pool.push_back(e);
    }
    return ev_pool[ev_used++];
  }
  void stage_begin(int stage) {
    cur_stage = -1;
    if (!((prof >> stage) & 1u)) return;
    ProfRec r{stage, next_event(), next_event()};
    if (!r.a || !r.b) return;
    cudaEventRecord(r.a, cur_stream);
    recs.push_back(r);
    cur_stage = stage;
  }
  void stage_end(int n_kernels) {
    launches += (unsigned long long)n_kernels;
    if (cur_stage < 0 || recs.empty()) return;
    cudaEventRecord(recs.back().b, cur_stream);
    cur_stage = -1;
  }

  outlets_status fail(outlets_status st, const std::string& msg) {
    err = msg;
    return st;
  }
  outlets_status cuda_fail(cudaError_t e, const char* what) {
    err = std::string(what) + ": " + cudaGetErrorString(e);
    return OUTLETS_ECUDA;
  }
  void* alloc(size_t bytes) {
    if (bytes == 0) bytes = 16;
    void* p = nullptr;
    if (cudaMalloc(&p, bytes) != cudaSuccess) {
      cudaGetLastError();
      oom = true;
      return nullptr;
    }
    cudaMemset(p, 0, bytes);
    allocs.push_back(p);
    dev_bytes += bytes;
    return p;
  }
};

struct outlets_kv {
  outlets_ctx* ctx = nullptr;
  int device = 0;
  int max_slots = 0, num_pages = 0, max_pages_per_slot = 0;
  void *k_pool = nullptr, *v_pool = nullptr;
  float *part_o = nullptr, *part_ml = nullptr;
  size_t part_items = 0;
  std::vector<int> len;
  std::vector<std::vector<int>> pages;
  std::vector<int> free_list;
  std::vector<void*> allocs;
};

#define OUT_CK(ctx, ...)                                         \
  do {                                                            \
    cudaError_t e_ = (__VA_ARGS__);                               \
    if (e_ != cudaSuccess) return (ctx)->cuda_fail(e_, #__VA_ARGS__); \
  } while (0)

namespace {

// True for buffers the context allocated itself (their tensor maps may be memoized).
bool owned_by(const outlets_ctx* c, const void* p) {
  for (void* q : c->allocs)
    if (q == p) return true;
  for (int i = 0; i < 3; ++i)
    if (c->taps_stage[i] == p) return true;
  return false;
}

// Uploads a host f32 matrix [rows, cols] through a device staging buffer and
// converts it (f32 -> act) into dst with the given row mapping and layout
// (kb_np > 0: k-block-major swizzled weight layout, else row-major, stride dst_ld).
outlets_status upload_rows(outlets_ctx* c, const float* src, int rows, int cols, void* dst, long long dst_ld,
                           int row_mode, int row_base, long long kb_np, float* stage, size_t stage_floats,
                           const float* col_scale = nullptr) {
  const int chunk = (int)std::max<size_t>(1, stage_floats / (size_t)cols);
  for (int r0 = 0; r0 < rows; r0 += chunk) {
    const int n = std::min(chunk, rows - r0);
    OUT_CK(c, cudaMemcpy(stage, src + (size_t)r0 * cols, (size_t)n * cols * 4, cudaMemcpyHostToDevice));
    const cudaError_t e =
        c->bf16 ? convert_rows_launch<bf16>(stage, (bf16*)dst, n, cols, dst_ld, row_mode, row_base + r0, kb_np,
                                            col_scale, 0)
                : convert_rows_launch<float>(stage, (float*)dst, n, cols, dst_ld, row_mode, row_base + r0, kb_np,
                                             col_scale, 0);
    OUT_CK(c, e);
    OUT_CK(c, cudaDeviceSynchronize());
  }
  return OUTLETS_OK;
}

outlets_status validate_config(const outlets_config* cfg, std::string& why) {
  auto bad = [&](const char* m) {
    why = m;
    return OUTLETS_EINVAL;
  };
  if (cfg->dtype != OUTLETS_F32 && cfg->dtype != OUTLETS_BF16) return bad("dtype must be OUTLETS_F32 or OUTLETS_BF16");
  if (cfg->d_model <= 0 || cfg->d_model % 64) return bad("d_model must be a positive multiple of 64");
  if (cfg->n_heads <= 0 || cfg->n_kv_heads <= 0 || cfg->n_heads % cfg->n_kv_heads)
    return bad("n_heads must be a positive multiple of n_kv_heads");
  if (cfg->head_dim <= 0 || cfg->head_dim % 16) return bad("head_dim must be a positive multiple of 16");
  if ((cfg->n_heads * cfg->head_dim) % 64) return bad("n_heads * head_dim must be a multiple of 64");
  if (cfg->ffn_dim <= 0) return bad("ffn_dim must be positive");
  if (cfg->vocab != 0 && (cfg->vocab < 8 || cfg->vocab > kMaxVocab)) return bad("vocab must be 0 or in 8..262144");
  if (cfg->embed_vocab < 0) return bad("embed_vocab must be >= 0");
  if (cfg->n_head_hidden < 1 || cfg->n_head_hidden > OUTLETS_MAX_HEAD_HIDDEN)
    return bad("n_head_hidden must be in 1..OUTLETS_MAX_HEAD_HIDDEN");
  for (int i = 0; i < cfg->n_head_hidden; ++i)
    if (cfg->head_hidden[i] <= 0 || cfg->head_hidden[i] % 4) return bad("head widths must be positive multiples of 4");
  if (!(cfg->rope_theta > 1.0f)) return bad("rope_theta must be > 1");
  if (!(cfg->rms_eps >= 0.0f)) return bad("rms_eps must be >= 0");
  if (cfg->max_tokens <= 0 || cfg->max_batch <= 0 || cfg->max_position <= 0)
    return bad("max_tokens, max_batch and max_position must be positive");
  if (cfg->dtype == OUTLETS_BF16) {
    if (cfg->head_dim != 64 && cfg->head_dim != 128) return bad("bf16 path supports head_dim 64 or 128");
    if (cfg->n_heads / cfg->n_kv_heads > 16) return bad("bf16 path supports at most 16 query heads per kv head");
  } else {
    if (cfg->head_dim > 256) return bad("f32 path supports head_dim <= 256");
  }
  return OUTLETS_OK;
}

#define OUT_TRY(expr)                      \
  do {                                     \
    outlets_status st_ = (expr);           \
    if (st_ != OUTLETS_OK) return st_;     \
  } while (0)

outlets_status ensure_copy_stream(outlets_ctx* c) {
  if (c->copy_stream) return OUTLETS_OK;
  OUT_CK(c, cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking));
  OUT_CK(c, cudaEventCreateWithFlags(&c->copy_start, cudaEventDisableTiming));
  for (auto& e : c->chunk_ev) OUT_CK(c, cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
  return OUTLETS_OK;
}

// One call's index metadata: pinned staging, one H2D copy on the copy stream
// into the slot's device buffer.  Sets c->meta_dev; kernels that read it are
// enqueued after wait_meta (the FC, norm and QKV kernels before them keep
// their programmatic launch chain).  The slot is released when the call's
// stream passes the slot's `done` event (recorded by CallSlot on every exit).
outlets_status upload_meta(outlets_ctx* c, const std::vector<int>& meta, cudaStream_t s) {
  if (meta.empty()) return OUTLETS_OK;
  OUT_TRY(ensure_copy_stream(c));
  const int slot = c->ring_i;
  outlets_ctx::Pin& p = c->ring[slot];
  c->ring_i = (c->ring_i + 1) % kRing;
  if (p.used) OUT_CK(c, cudaEventSynchronize(p.done));
  const size_t cap = std::max<size_t>(meta.size() * 2, 1 << 16);
  if (meta.size() > p.cap) {
    if (p.h) cudaFreeHost(p.h);
    p.h = nullptr;
    p.cap = 0;
    if (cudaMallocHost(&p.h, cap * sizeof(int)) != cudaSuccess) {
      cudaGetLastError();
      return c->fail(OUTLETS_ENOMEM, "pinned metadata buffer allocation failed");
    }
    p.cap = cap;
  }
  if (meta.size() > p.dev_cap) {
    if (p.dev) cudaFree(p.dev);
    p.dev = nullptr;
    p.dev_cap = 0;
    if (cudaMalloc(&p.dev, cap * sizeof(int)) != cudaSuccess) {
      cudaGetLastError();
      return c->fail(OUTLETS_ENOMEM, "metadata buffer allocation failed");
    }
    p.dev_cap = cap;
  }
  std::memcpy(p.h, meta.data(), meta.size() * sizeof(int));
  OUT_CK(c, cudaMemcpyAsync(p.dev, p.h, meta.size() * sizeof(int), cudaMemcpyHostToDevice, c->copy_stream));
  OUT_CK(c, cudaEventRecord(p.ev, c->copy_stream));
  p.used = true;
  c->cur_slot = slot;
  c->meta_waited = false;
  c->meta_dev = p.dev;
  return OUTLETS_OK;
}

// Makes stream s wait for the current call's metadata upload (once).
outlets_status wait_meta(outlets_ctx* c, cudaStream_t s) {
  if (c->cur_slot < 0 || c->meta_waited) return OUTLETS_OK;
  OUT_CK(c, cudaStreamWaitEvent(s, c->ring[c->cur_slot].ev, 0));
  c->meta_waited = true;
  return OUTLETS_OK;
}

// Releases the call's metadata slot on every exit from a prediction call:
// records the slot's `done` event after everything the call enqueued.
struct CallSlot {
  outlets_ctx* c;
  cudaStream_t s;
  ~CallSlot() {
    if (c->cur_slot >= 0) {
      if (!c->meta_waited) cudaStreamWaitEvent(s, c->ring[c->cur_slot].ev, 0);  // done implies uploaded
      cudaEventRecord(c->ring[c->cur_slot].done, s);
      c->cur_slot = -1;
    }
  }
};

struct MetaBuilder {
  std::vector<int> v;
  size_t put(const int* src, size_t n) {
    while (v.size() % 4) v.push_back(0);
    size_t off = v.size();
    v.insert(v.end(), src, src + n);
    return off;
  }
  size_t put(const std::vector<int>& x) { return put(x.data(), x.size()); }
};

// Tensor map of a library-owned buffer (weights, workspace): encoded once.
bool cached_map(outlets_ctx* c, CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint64_t ld,
                uint32_t box_rows) {
  const MapKey k{base, cols, rows, ld, box_rows};
  auto it = c->map_cache.find(k);
  if (it != c->map_cache.end()) {
    *m = it->second;
    return true;
  }
  if (!make_map(m, base, cols, rows, ld, box_rows)) return false;
  if (c->map_cache.size() > 4096) c->map_cache.clear();
  c->map_cache.emplace(k, *m);
  return true;
}

bool owned_by(const outlets_ctx* c, const void* p);

// Tensor maps of the (up to three) A pieces of a GEMM.
outlets_status a_maps(outlets_ctx* c, const void* const* a, int n_pieces, int k_piece, long long lda, int M,
                      CUtensorMap* am) {
  for (int i = 0; i < 3; ++i) {
    const void* base = a[i < n_pieces ? i : 0];
    if (i > 0 && n_pieces == 1) {
      am[i] = am[0];
      continue;
    }
    const bool ok = owned_by(c, base) ? cached_map(c, &am[i], base, (uint64_t)k_piece, (uint64_t)M, (uint64_t)lda, 128)
                                      : make_map(&am[i], base, (uint64_t)k_piece, (uint64_t)M, (uint64_t)lda, 128);
    if (!ok) return c->fail(OUTLETS_ECUDA, "cuTensorMapEncodeTiled failed for a GEMM A operand");
  }
  return OUTLETS_OK;
}

// bf16 GEMM through tcgen05 with an explicit tile plan.  A pieces: row-major
// [M, k_piece] with row stride lda.
// RMSNorm folded into a large-M GEMM pair (see GemmArgs): a producer writes
// out_bf16 and ss (row stride ss_stride; tiles = its 64-column groups, set
// here); a consumer reads row_ss with the producer's group count.
struct NormFold {
  bf16* out_bf16 = nullptr;
  float* ss = nullptr;
  const float* row_ss = nullptr;
  int tiles = 0;
};

outlets_status gemm_tc_ex(outlets_ctx* c, const void* const* a, int n_pieces, int k_piece, long long lda, int M,
                          const void* b, long long b_np, int N, int K, int epi, int bn, int mt, int splits, void* out,
                          long long ldo, const float* residual, long long ldr, const float* bias, cudaStream_t s,
                          NormFold* nf = nullptr) {
  if (M == 0) return OUTLETS_OK;
  CUtensorMap am[3];
  OUT_TRY(a_maps(c, a, n_pieces, k_piece, lda, M, am));
  GemmArgs g{};
  g.M = M;
  g.N = N;
  g.K = K;
  g.b = b;
  g.b_np = b_np;
  g.k_per_map = k_piece;
  g.splits = splits;
  g.prefetch = M <= 256 ? prefetch_blocks() : 0;  // small M streams every weight tile once
  // Tile raster: groups of M blocks (tm rows each), N-major inside a group.
  // A group's activation panel fills about 48 MB of L2, so its weight tiles
  // are fetched once per group; and it is never narrower than a square wave
  // (about sqrt(SMs * bn / tm) blocks), since the panels one wave of tiles
  // touches are what it reads from DRAM when the panels do not stay in L2
  // across waves (long K).
  const long long tm = 128LL * mt;
  const long long sq = (long long)std::lround(std::sqrt((double)c->num_sms * bn / (double)tm));
  g.group_m = (int)std::max<long long>(std::max<long long>(1, sq),
                                       std::min<long long>(cdiv(M, tm), (48ll << 20) / (tm * K * 2)));
  g.out = out;
  g.ldo = ldo;
  g.residual = residual;
  g.ldr = ldr;
  g.bias = bias;
  g.err = c->err_dev;
  if (nf) {
    g.nrm_d = c->d;
    g.nrm_eps = c->cfg.rms_eps;
    if (nf->out_bf16) {  // producer
      nf->tiles = (int)cdiv(N, 64);  // sums of squares per 64-column group
      if (nf->tiles > c->ss_stride) return c->fail(OUTLETS_ECAPACITY, "folded-norm tile count");
      g.nrm_out = nf->out_bf16;
      g.nrm_ss = nf->ss;
    } else {  // consumer
      g.row_ss = nf->row_ss;
    }
    g.nrm_tiles = nf->tiles;
  }
  OUT_CK(c, gemm_tc_launch(am, bn, epi, mt, g, c->num_sms, s));
  return OUTLETS_OK;
}

// Large-M GEMM (prefill): 128-row tiles, tile width chosen to fill the SMs.
outlets_status gemm_tc(outlets_ctx* c, const void* const* a, int n_pieces, int k_piece, long long lda, int M,
                       const void* b, long long b_np, int N, int K, int epi, void* out, long long ldo,
                       const float* residual, long long ldr, const float* bias, cudaStream_t s,
                       NormFold* nf = nullptr) {
  int bn = 256;
  if (epi == EPI_BIAS_RELU) {
    bn = 64;  // the head's first layer (N <= a few thousand): the only width built for this epilogue
  } else if (epi != EPI_SWIGLU) {
    auto tiles = [&](int bnv) { return cdiv(M, 128) * cdiv(N, bnv); };
    if (tiles(256) >= c->num_sms) bn = 256;
    else if (tiles(128) >= c->num_sms) bn = 128;
    else bn = 64;
  }
  // 256 x 256 tiles (two 128-row MMAs per staged weight tile, one TMEM
  // accumulator) where a wave of them fills the SMs: a third fewer operand
  // bytes per MMA and more of them in flight per ring stage, at the price of
  // an epilogue that no longer overlaps the next tile's main loop.  That
  // price outweighs the gain only for the f32 + residual epilogue after a
  // short K loop (the O projection at K = 4096).
  const bool wide_epi = !(epi == EPI_F32 && residual && K < 8192);
  const int mt = (wide_epi && bn == 256 && cdiv(M, 256) * cdiv(N, 256) >= c->num_sms) ? 2 : 1;
  return gemm_tc_ex(c, a, n_pieces, k_piece, lda, M, b, b_np, N, K, epi, bn, mt, 1, out, ldo, residual, ldr, bias, s,
                    nf);
}

// Small-M GEMM (M <= 256): every weight tile is streamed once.  K is split so
// that enough CTAs stream the weights, but every split adds an f32 slice
// part[s][M][N] that is written and read back through L2 by the consuming
// kernel.  Tile width and split count minimise an estimate of both costs:
// operand streaming per CTA (A and B tiles, ~85 GB/s per CTA) plus the slice
// traffic (~6 TB/s), rates measured on GB300.  Returns the slice count in
// *slices.
outlets_status gemm_split(outlets_ctx* c, const void* const* a, int n_pieces, int k_piece, long long lda, int M,
                          const void* b, long long b_np, int N, int K, float* part, int* slices, cudaStream_t s) {
  if (M == 0) return OUTLETS_OK;
  const int mt = M <= 128 ? 1 : 2;
  const long long tm = 128LL * mt;
  const long long kb = cdiv(K, 64);
  const long long max_s = std::min<long long>(kb, (long long)(c->part_floats / ((size_t)M * N)));
  if (max_s < 1 || N % 4) return c->fail(OUTLETS_ECAPACITY, "split-K workspace too small");
  int best_bn = 256, best_s = 1;
  double best_t = -1.0;
  for (int bn : {256, 128}) {
    const long long tiles = cdiv(N, bn) * cdiv(M, tm);
    for (long long sp = 1; sp <= max_s && (sp == 1 || tiles * sp <= c->num_sms); ++sp) {
      const double waves = (double)cdiv(tiles * sp, c->num_sms);
      const double per_cta = (double)(bn + tm) * 64.0 * 2.0 * (double)cdiv(kb, sp);
      const double t = waves * per_cta / 85e3 + 2.0 * sp * M * N * 4.0 / 6e6;
      if (best_t < 0 || t < best_t) {
        best_t = t;
        best_bn = bn;
        best_s = (int)sp;
      }
    }
  }
  const int bn = best_bn;
  CUtensorMap am[3];
  OUT_TRY(a_maps(c, a, n_pieces, k_piece, lda, M, am));
  GemmArgs g{};
  g.M = M;
  g.N = N;
  g.K = K;
  g.b = b;
  g.b_np = b_np;
  g.k_per_map = k_piece;
  g.splits = best_s;
  g.group_stride = (long long)M * N;
  g.group_m = 1;
  g.out = part;
  g.ldo = N;
  g.err = c->err_dev;
  OUT_CK(c, gemm_small_launch(am, bn, EPI_SLICES, mt, g, s));
  *slices = best_s;
  return OUTLETS_OK;
}

inline bool small_path(const outlets_ctx* c, int M) { return c->bf16 && M <= 256; }

outlets_status gemm_f32(outlets_ctx* c, const void* const* a, int k_piece, int M, const void* b, int N, int K,
                        int epi, void* out, long long ldo, const float* residual, long long ldr, const float* bias,
                        cudaStream_t s) {
  const float* ap[3] = {(const float*)a[0], (const float*)a[1], (const float*)a[2]};
  GemmArgs g{};
  g.M = M;
  g.N = N;
  g.K = K;
  g.k_per_map = k_piece;
  g.splits = 1;
  g.group_m = 1;
  g.out = out;
  g.ldo = ldo;
  g.residual = residual;
  g.ldr = ldr;
  g.bias = bias;
  g.err = c->err_dev;
  OUT_CK(c, gemm_simt_f32_launch(ap, (const float*)b, epi, g, s));
  return OUTLETS_OK;
}


// Everything after attention: O projection + residual, post-attention norm,
// SwiGLU MLP + residual, final norm of the predicted rows, length head.
// resid: the rows of f (the layer input's residual stream) that go with the
// rows of c->attn.
outlets_status run_tail(outlets_ctx* c, int rows, int out_rows, const int* out_row_idx_dev, float* z_dev,
                        float* len_dev, cudaStream_t s, const float* resid) {
  const int d = c->d;
  const float eps = c->cfg.rms_eps;
  const bool small = small_path(c, rows);
  int sl = 1;
  NormFold nf_a;  // large-M bf16: the O GEMM leaves bf16(a) and its sums of squares for gate/up
  nf_a.out_bf16 = (bf16*)c->ahat;
  nf_a.ss = c->ss_a;
  // O projection + residual: a = f + attn W_o^T; post-attention RMSNorm
  c->stage_begin(OUTLETS_S_O);
  {
    const void* a1[3] = {c->attn, c->attn, c->attn};
    if (small)
      OUT_TRY(gemm_split(c, a1, 1, c->attn_w, c->attn_w, rows, c->w_o, c->np_o, d, c->attn_w, c->part, &sl, s));
    else if (c->bf16)  // a = f + attn W_o^T, its bf16 copy and per-tile sums of squares (norm folded)
      OUT_TRY(gemm_tc(c, a1, 1, c->attn_w, c->attn_w, rows, c->w_o, c->np_o, d, c->attn_w, EPI_F32, c->a, d, resid, d,
                      nullptr, s, &nf_a));
    else
      OUT_TRY(gemm_f32(c, a1, c->attn_w, rows, c->w_o, d, c->attn_w, EPI_F32, c->a, d, resid, d, nullptr, s));
  }
  c->stage_end(1);
  if (small) {
    c->stage_begin(OUTLETS_S_NORM_POST);
    OUT_CK(c, rmsnorm_reduce_launch<bf16>(c->part, sl, (long long)rows * d, resid, nullptr, c->ones, (bf16*)c->ahat,
                                          c->a, rows, d, eps, s, discard_slices()));
    c->stage_end(1);
  } else if (!c->bf16) {
    c->stage_begin(OUTLETS_S_NORM_POST);
    OUT_CK(c, rmsnorm_launch<float>(c->a, c->g_post, (float*)c->ahat, nullptr, rows, d, eps, s));
    c->stage_end(1);
  }
  // gate/up + SwiGLU
  c->stage_begin(OUTLETS_S_GATEUP);
  {
    const void* a1[3] = {c->ahat, c->ahat, c->ahat};
    if (small) {
      // one wave of tiles: the width (multiple of 64) that minimizes waves x width
      int best_bn = 256;
      long long best = -1;
      for (int bnv : {256, 192, 128}) {
        const long long cost = cdiv(cdiv(2 * c->Fp, bnv), c->num_sms) * bnv;
        if (best < 0 || cost < best) {
          best = cost;
          best_bn = bnv;
        }
      }
      CUtensorMap am[3];
      OUT_TRY(a_maps(c, a1, 1, d, d, rows, am));
      GemmArgs g{};
      g.M = rows;
      g.N = 2 * c->Fp;
      g.K = d;
      g.b = c->w_gu;
      g.b_np = c->np_gu;
      g.k_per_map = d;
      g.splits = 1;
      g.group_m = 1;
      g.out = c->u;
      g.ldo = c->Fp;
      g.err = c->err_dev;
      OUT_CK(c, gemm_small_launch(am, best_bn, EPI_SWIGLU, rows <= 128 ? 1 : 2, g, s));
    } else if (c->bf16) {  // A = bf16(a); the rows are scaled by their RMSNorm factor before SwiGLU
      NormFold use{nullptr, nullptr, c->ss_a, nf_a.tiles};
      OUT_TRY(gemm_tc(c, a1, 1, d, d, rows, c->w_gu, c->np_gu, 2 * c->Fp, d, EPI_SWIGLU, c->u, c->Fp, nullptr, 0, nullptr,
                      s, &use));
    } else {
      OUT_TRY(gemm_f32(c, a1, d, rows, c->w_gu, 2 * c->Fp, d, EPI_F32, c->gu32, 2 * c->Fp, nullptr, 0, nullptr, s));
      OUT_CK(c, swiglu_launch<float>(c->gu32, (float*)c->u, rows, c->Fp, s));
      c->launches += 1;
    }
  }
  c->stage_end(1);
  // down + residual: y = a + u W_down^T
  c->stage_begin(OUTLETS_S_DOWN);
  {
    const void* a1[3] = {c->u, c->u, c->u};
    if (small)
      OUT_TRY(gemm_split(c, a1, 1, c->Fp, c->Fp, rows, c->w_down, c->np_down, d, c->Fp, c->part, &sl, s));
    else if (c->bf16)
      OUT_TRY(gemm_tc(c, a1, 1, c->Fp, c->Fp, rows, c->w_down, c->np_down, d, c->Fp, EPI_F32, c->y, d, c->a, d, nullptr, s));
    else
      OUT_TRY(gemm_f32(c, a1, c->Fp, rows, c->w_down, d, c->Fp, EPI_F32, c->y, d, c->a, d, nullptr, s));
  }
  c->stage_end(1);
  // final RMSNorm of the predicted rows -> h^draft
  c->stage_begin(OUTLETS_S_FINAL_NORM);
  int n_final = 1;
  if (small && !out_row_idx_dev) {
    // every row is predicted: add the slices and the residual, normalize, in one pass
    OUT_CK(c, rmsnorm_reduce_launch<bf16>(c->part, sl, (long long)rows * d, c->a, nullptr, c->g_final, (bf16*)c->hn,
                                          c->y, rows, d, eps, s, discard_slices()));
  } else {
    if (small) {
      // y for every row (the normed copy goes to a dead buffer), then the predicted rows
      OUT_CK(c, rmsnorm_reduce_launch<bf16>(c->part, sl, (long long)rows * d, c->a, nullptr, c->g_final,
                                            (bf16*)c->ahat, c->y, rows, d, eps, s, discard_slices()));
      n_final = 2;
    }
    if (c->bf16)
      OUT_CK(c, rmsnorm_gather_launch<bf16>(c->y, out_row_idx_dev, c->g_final, (bf16*)c->hn, out_rows, d, eps, s));
    else
      OUT_CK(c, rmsnorm_gather_launch<float>(c->y, out_row_idx_dev, c->g_final, (float*)c->hn, out_rows, d, eps, s));
  }
  c->stage_end(n_final);
  // length head: Linear+ReLU layers, then the output row
  c->stage_begin(OUTLETS_S_HEAD);
  const int nl = (int)c->head_dims.size() - 1;
  const int w1 = c->head_dims[1];
  const void* ah[3] = {c->hn, c->hn, c->hn};
  if (small_path(c, out_rows) && nl == 2) {
    int hs = 1;
    OUT_TRY(gemm_split(c, ah, 1, d, d, out_rows, c->head_w0, c->np_h0, w1, d, c->part, &hs, s));
    OUT_CK(c, head_tail_launch(c->part, hs, (long long)out_rows * w1, c->head_b[0], c->head_wf[1], c->head_b[1],
                               out_rows, w1, z_dev, len_dev, s, discard_slices()));
    c->stage_end(2);
    return OUTLETS_OK;
  }
  float* cur = c->h1a;
  if (c->bf16)
    OUT_TRY(gemm_tc(c, ah, 1, d, d, out_rows, c->head_w0, c->np_h0, w1, d, EPI_BIAS_RELU, cur, w1, nullptr, 0, c->head_b[0], s));
  else
    OUT_TRY(gemm_f32(c, ah, d, out_rows, c->head_w0, w1, d, EPI_BIAS_RELU, cur, w1, nullptr, 0, c->head_b[0], s));
  for (int i = 1; i < nl - 1; ++i) {
    float* nxt = (cur == c->h1a) ? c->h1b : c->h1a;
    const void* a1[3] = {cur, cur, cur};
    OUT_TRY(gemm_f32(c, a1, c->head_dims[i], out_rows, c->head_wf[i], c->head_dims[i + 1], c->head_dims[i],
                     EPI_BIAS_RELU, nxt, c->head_dims[i + 1], nullptr, 0, c->head_b[i], s));
    cur = nxt;
  }
  OUT_CK(c, head_tail_launch(cur, 1, 0, nullptr, c->head_wf[nl - 1], c->head_b[nl - 1], out_rows,
                             c->head_dims[nl - 1], z_dev, len_dev, s));
  c->stage_end(nl);
  return OUTLETS_OK;
}

// Draft LM head tile width (tensor-core path): the one of 256, 224, 128 with
// the smallest estimated time, waves x per-tile time.  A tile streams K/64
// blocks of A and W_lm tiles (about 90 GB/s per SM) or is bound by its MMAs
// (about 11.5 TFLOP/s per SM), whichever is slower, and then reduces its
// logits on chip (the epilogue, about 45 ps per logit).  Narrower tiles fill
// the last wave better (V = 128256 on 152 SMs: 224 gives 3.8 waves).
int lm_tile_width(const outlets_ctx* c, int rows) {
  const double tm = rows <= 128 ? 128.0 : 256.0;
  const double kb = (double)cdiv(c->d, 64);
  int best = 256;
  double best_t = -1.0;
  for (int bn : {256, 224, 128}) {
    const double waves = (double)cdiv(cdiv(c->V, bn), c->num_sms);
    const double ingest = (tm + bn) * 128.0 / 90e3;
    const double mma = 2.0 * tm * bn * 64.0 / 11.5e6;
    const double t = waves * (kb * std::max(ingest, mma) + tm * bn * 4.5e-5);
    if (best_t < 0 || t < best_t) {
      best_t = t;
      best = bn;
    }
  }
  return best;
}

outlets_status check_draft(outlets_ctx* c, const outlets_draft_out* o) {
  if (!o) return c->fail(OUTLETS_EINVAL, "draft outputs must not be NULL");
  if (c->V == 0) return c->fail(OUTLETS_EUNSUPPORTED, "the context has no draft head (vocab == 0)");
  if (o->k < 1 || o->k > OUTLETS_MAX_TOPK || o->k > c->V)
    return c->fail(OUTLETS_EINVAL, "draft k must be in 1 .. min(OUTLETS_MAX_TOPK, vocab)");
  if (!o->topk_ids || !o->topk_logprob) return c->fail(OUTLETS_EINVAL, "topk_ids and topk_logprob must not be NULL");
  return OUTLETS_OK;
}

// Draft LM head (Sec. 4.2, Eq. 2) on rows states h [rows, d] (act dtype, on the
// device), in passes of lm_rows_cap rows: GEMM with the on-chip softmax/top-k
// epilogue (CUDA-core path: logits, then tile statistics), then the merge.
// Device outputs are written in place; host outputs go through the context's
// buffers and are copied on the stream.
outlets_status run_draft(outlets_ctx* c, const void* h, int rows, const outlets_draft_out& o, cudaStream_t s) {
  if (rows == 0) return OUTLETS_OK;
  const int V = c->V, d = c->d, k = o.k, kt = k == 1 ? 1 : 8;
  int* ids = is_device_ptr(o.topk_ids) ? o.topk_ids : c->lm_ids;
  float* lp = is_device_ptr(o.topk_logprob) ? o.topk_logprob : c->lm_lp;
  float* lse = o.logsumexp ? (is_device_ptr(o.logsumexp) ? o.logsumexp : c->lm_lse) : nullptr;
  const bool host_logits = o.logits && !is_device_ptr(o.logits);
  if ((ids == c->lm_ids || lp == c->lm_lp || lse == c->lm_lse) && rows > c->max_rows)
    return c->fail(OUTLETS_ECAPACITY, "rows exceed the context's output buffers (max_tokens / max_batch)");
  if (host_logits && !c->lm_logits_stage) {
    c->lm_logits_stage = (float*)c->alloc((size_t)c->lm_rows_cap * V * 4);
    if (!c->lm_logits_stage) return c->fail(OUTLETS_ENOMEM, "draft logits staging allocation failed");
  }
  c->stage_begin(OUTLETS_S_DRAFT);
  int n_launch = 0;
  if (c->lm_bound_dirty) {
    OUT_CK(c, cudaMemsetAsync(c->lm_bound, kLmBoundInit & 0xFF, (size_t)c->lm_rows_cap * kLmBoundSlots * sizeof(int),
                              s));
    c->lm_bound_dirty = false;
  }
  for (int g0 = 0; g0 < rows; g0 += c->lm_rows_cap) {
    const int gr = std::min(c->lm_rows_cap, rows - g0);
    const void* hg = static_cast<const char*>(h) + (size_t)g0 * d * c->esz;
    float* lg = o.logits ? (host_logits ? c->lm_logits_stage : o.logits + (size_t)g0 * V) : nullptr;
    const void* a1[3] = {hg, hg, hg};
    int n_tiles = 0;
    if (c->bf16) {
      const int bn = lm_tile_width(c, gr);
      n_tiles = 2 * (int)cdiv(V, bn);  // two column halves per tile
      CUtensorMap am[3];
      OUT_TRY(a_maps(c, a1, 1, d, d, gr, am));
      GemmArgs g{};
      g.M = gr;
      g.N = V;
      g.K = d;
      g.b = c->w_lm;
      g.b_np = c->np_lm;
      g.k_per_map = d;
      g.splits = 1;
      g.group_m = 1;
      g.ldo = V;
      g.err = c->err_dev;
      g.lm_logits = lg;
      g.lm_stats = c->lm_stats;
      g.lm_top = c->lm_top;
      g.lm_bound = c->lm_bound;
      c->lm_bound_dirty = true;  // until its merge is enqueued
      OUT_CK(c, gemm_small_launch(am, bn, kt == 1 ? EPI_LM1 : EPI_LM8, gr <= 128 ? 1 : 2, g, s));
      n_launch += 1;
    } else {
      float* lw = lg ? lg : c->lm_logits_ws;
      OUT_TRY(gemm_f32(c, a1, d, gr, c->w_lm, V, d, EPI_F32, lw, V, nullptr, 0, nullptr, s));
      n_tiles = (int)cdiv(V, kLmTileF32);
      OUT_CK(c, lm_tile_stats_f32_launch(lw, V, gr, V, kLmTileF32, kt, c->lm_stats, c->lm_top, s));
      n_launch += 2;
    }
    OUT_CK(c, lm_merge_launch(c->lm_stats, c->lm_top, n_tiles, kt, gr, k, ids + (size_t)g0 * k,
                              lp + (size_t)g0 * k, lse ? lse + g0 : nullptr, c->lm_bound, s));
    c->lm_bound_dirty = false;
    n_launch += 1;
    if (host_logits)
      OUT_CK(c, cudaMemcpyAsync(o.logits + (size_t)g0 * V, lg, (size_t)gr * V * 4, cudaMemcpyDeviceToHost, s));
  }
  c->stage_end(n_launch);
  if (ids != o.topk_ids)
    OUT_CK(c, cudaMemcpyAsync(o.topk_ids, ids, (size_t)rows * k * sizeof(int), cudaMemcpyDeviceToHost, s));
  if (lp != o.topk_logprob)
    OUT_CK(c, cudaMemcpyAsync(o.topk_logprob, lp, (size_t)rows * k * 4, cudaMemcpyDeviceToHost, s));
  if (lse && lse != o.logsumexp)
    OUT_CK(c, cudaMemcpyAsync(o.logsumexp, lse, (size_t)rows * 4, cudaMemcpyDeviceToHost, s));
  return OUTLETS_OK;
}

// FC (Eq. 1) -> input RMSNorm -> QKV projection.  Fills the input side of the
// RoPE arguments (fused qkv rows, or split slices on the small-M path).
struct QkvSrc {
  const void* p;
  bool f32;
  int n_split;
  long long stride;
};

// FC (Eq. 1) -> input RMSNorm -> QKV for rows row0 .. row0 + rows - 1 (tp
// points at row row0 of each tap; row0 > 0 only on the large-M path).
outlets_status run_qkv(outlets_ctx* c, int rows, QkvSrc* q, cudaStream_t s, int row0, const int* tok_dev, int sl,
                       int n_norm, bool kv_only);

// kv_only: the large-M QKV GEMM computes only the key and value columns (the
// static prediction of the last rows computes their queries separately).
outlets_status run_front(outlets_ctx* c, const void* const tp[3], int rows, QkvSrc* q, cudaStream_t s,
                         int row0, const int* tok_dev, bool kv_only = false) {
  const int d = c->d;
  const float eps = c->cfg.rms_eps;
  const bool small = small_path(c, rows);
  int sl = 1;
  if (!tp) {
    c->xin_raw = false;
    // draft rollout step: the feature input is the draft layer's own output
    // state y of the previous step (same rows), in place of Eq. 1's fused taps
    c->stage_begin(OUTLETS_S_NORM_IN);
    OUT_CK(c, cudaMemcpyAsync(c->f, c->y, (size_t)rows * d * 4, cudaMemcpyDeviceToDevice, s));
    if (c->bf16) OUT_CK(c, rmsnorm_launch<bf16>(c->f, c->ones, (bf16*)c->xhat, nullptr, rows, d, eps, s));
    else OUT_CK(c, rmsnorm_launch<float>(c->f, c->g_in, (float*)c->xhat, nullptr, rows, d, eps, s));
    return run_qkv(c, rows, q, s, row0, tok_dev, sl, 1, false);
  }
  // large-M bf16 without the embedding branch: the input RMSNorm is folded
  // into the FC (bf16 copy + sums of squares) and QKV (row scale) GEMMs
  const bool fold_in = !small && c->bf16 && c->EV == 0;
  c->xin_raw = fold_in;
  c->stage_begin(OUTLETS_S_FC);
  if (small) {
    OUT_TRY(gemm_split(c, tp, 3, d, d, rows, c->w_proj, c->np_proj, d, 3 * d, c->part, &sl, s));
  } else if (c->bf16) {
    NormFold nf;
    nf.out_bf16 = (bf16*)c->xhat + (size_t)row0 * d;
    nf.ss = c->ss_f + (size_t)row0 * c->ss_stride;
    OUT_TRY(gemm_tc(c, tp, 3, d, d, rows, c->w_proj, c->np_proj, d, 3 * d, EPI_F32, c->f + (size_t)row0 * d, d, nullptr,
                    0, nullptr, s, fold_in ? &nf : nullptr));
    c->fold_tiles_f = nf.tiles;
  } else {
    OUT_TRY(gemm_f32(c, tp, d, rows, c->w_proj, d, 3 * d, EPI_F32, c->f, d, nullptr, 0, nullptr, s));
  }
  c->stage_end(1);
  if (fold_in) return run_qkv(c, rows, q, s, row0, tok_dev, sl, 0, kv_only);
  c->stage_begin(OUTLETS_S_NORM_IN);
  if (small)
    OUT_CK(c, rmsnorm_reduce_launch<bf16>(c->part, sl, (long long)rows * d, nullptr, nullptr, c->ones, (bf16*)c->xhat,
                                          c->f, rows, d, eps, s, discard_slices()));
  else if (c->bf16)
    OUT_CK(c, rmsnorm_launch<bf16>(c->f + (size_t)row0 * d, c->ones, (bf16*)c->xhat + (size_t)row0 * d, nullptr, rows,
                                   d, eps, s));
  else
    OUT_CK(c, rmsnorm_launch<float>(c->f, c->g_in, (float*)c->xhat, nullptr, rows, d, eps, s));
  return run_qkv(c, rows, q, s, row0, tok_dev, sl, 1, kv_only);
}

// Input-embedding branch (if any) and the QKV projection; the input-norm stage
// (n_norm kernels so far) is still open.
outlets_status run_qkv(outlets_ctx* c, int rows, QkvSrc* q, cudaStream_t s, int row0, const int* tok_dev, int sl,
                       int n_norm, bool kv_only) {
  const int d = c->d;
  const float eps = c->cfg.rms_eps;
  const bool small = small_path(c, rows);
  const void* xr = (const char*)c->xhat + (size_t)row0 * d * c->esz;
  const void* a1[3] = {xr, xr, xr};
  int pieces = 1;
  if (c->EV > 0) {
    // input-embedding branch: the normalized embeddings are the first d input
    // columns of the QKV GEMM (a second A piece; nothing is concatenated)
    OUT_TRY(wait_meta(c, s));  // host token ids travel with the call's metadata
    void* er = (char*)c->ehat + (size_t)row0 * d * c->esz;
    if (c->bf16)
      OUT_CK(c, embed_rmsnorm_launch<bf16>(tok_dev + row0, (const bf16*)c->w_embed, c->EV, c->g_emb, (bf16*)er, rows,
                                           d, eps, c->err_dev, s));
    else
      OUT_CK(c, embed_rmsnorm_launch<float>(tok_dev + row0, (const float*)c->w_embed, c->EV, c->g_emb, (float*)er,
                                            rows, d, eps, c->err_dev, s));
    a1[0] = er;
    a1[1] = xr;
    pieces = 2;
    n_norm = 2;
  }
  c->stage_end(n_norm);
  c->stage_begin(OUTLETS_S_QKV);
  const int K = c->qkv_k;
  if (small) {
    OUT_TRY(gemm_split(c, a1, pieces, d, d, rows, c->w_qkv, c->np_qkv, c->qkv_n, K, c->part, &sl, s));
    *q = {c->part, true, sl, (long long)rows * c->qkv_n};
  } else if (c->bf16) {
    NormFold use;  // folded input norm: scale the rows by the FC's sums of squares
    use.row_ss = c->ss_f + (size_t)row0 * c->ss_stride;
    use.tiles = c->fold_tiles_f;
    // keys and values only: output columns H*hd .. (H + 2 KVH)*hd, i.e. the
    // weight rows from H*hd on in the k-block-major layout (row offset n0:
    // n0 * 64 elements; n0 is a multiple of 8, so the swizzle phase holds)
    const long long n0 = kv_only ? (long long)c->H * c->hd : 0;
    const int n_cols = kv_only ? 2 * c->KVH * c->hd : c->qkv_n;
    OUT_TRY(gemm_tc(c, a1, pieces, d, d, rows, (const char*)c->w_qkv + (size_t)n0 * 64 * c->esz, c->np_qkv, n_cols,
                    K, EPI_ACT, (char*)c->qkv + ((size_t)row0 * c->qkv_n + n0) * c->esz, c->qkv_n, nullptr, 0,
                    nullptr, s, c->xin_raw ? &use : nullptr));
    *q = {c->qkv, false, 1, 0};
  } else {
    OUT_TRY(gemm_f32(c, a1, d, rows, c->w_qkv, c->qkv_n, K, EPI_F32, c->qkv, c->qkv_n, nullptr, 0, nullptr, s));
    *q = {c->qkv, true, 1, 0};
  }
  c->stage_end(1);
  return OUTLETS_OK;
}

outlets_status launch_rope(outlets_ctx* c, const QkvSrc& q, RopeArgs& ra, cudaStream_t s) {
  ra.n_split = q.n_split;
  ra.split_stride = q.stride;
  ra.discard = q.f32 && q.p == c->part && discard_slices();
  if (c->bf16) {
    if (q.f32) OUT_CK(c, rope_scatter_launch<float, bf16>((const float*)q.p, ra, s));
    else OUT_CK(c, rope_scatter_launch<bf16, bf16>((const bf16*)q.p, ra, s));
  } else {
    OUT_CK(c, rope_scatter_launch<float, float>((const float*)q.p, ra, s));
  }
  return OUTLETS_OK;
}

// Stages host taps (or passes device taps through); checks alignment.
outlets_status prepare_taps(outlets_ctx* c, const void* const taps[3], int rows, const void* out[3],
                            cudaStream_t s) {
  for (int i = 0; i < 3; ++i) {
    if (!taps[i]) return c->fail(OUTLETS_EINVAL, "taps[i] is NULL");
    if (is_device_ptr(taps[i])) {
      if (reinterpret_cast<uintptr_t>(taps[i]) % 16) return c->fail(OUTLETS_EINVAL, "device taps must be 16-byte aligned");
      out[i] = taps[i];
    } else {
      if (!c->taps_stage[i]) {
        c->taps_stage[i] = c->alloc((size_t)c->max_rows * c->d * c->esz);
        if (!c->taps_stage[i]) return c->fail(OUTLETS_ENOMEM, "tap staging allocation failed");
      }
      OUT_CK(c, cudaMemcpyAsync(c->taps_stage[i], taps[i], (size_t)rows * c->d * c->esz, cudaMemcpyHostToDevice, s));
      out[i] = c->taps_stage[i];
    }
  }
  return OUTLETS_OK;
}

// Host taps of a large call: copied in n row chunks on the context's copy
// stream (after the work already queued on s, which may still read the
// staging buffers); chunk i's completion is recorded in chunk_ev[i] so the
// front of the pipeline can start on rows that have landed while later rows
// are still in transit.  tp receives the staging buffers.
outlets_status stage_taps_chunked(outlets_ctx* c, const void* const taps[3], int rows, int n, int chunk_rows,
                                  const void* tp[3], cudaStream_t s) {
  OUT_TRY(ensure_copy_stream(c));
  const size_t row_bytes = (size_t)c->d * c->esz;
  for (int i = 0; i < 3; ++i) {
    if (!taps[i]) return c->fail(OUTLETS_EINVAL, "taps[i] is NULL");
    if (!c->taps_stage[i]) {
      c->taps_stage[i] = c->alloc((size_t)c->max_rows * row_bytes);
      if (!c->taps_stage[i]) return c->fail(OUTLETS_ENOMEM, "tap staging allocation failed");
    }
    tp[i] = c->taps_stage[i];
  }
  OUT_CK(c, cudaEventRecord(c->copy_start, s));
  OUT_CK(c, cudaStreamWaitEvent(c->copy_stream, c->copy_start, 0));
  for (int k = 0; k < n; ++k) {
    const int r0 = k * chunk_rows, r1 = std::min(rows, r0 + chunk_rows);
    for (int i = 0; i < 3; ++i)
      OUT_CK(c, cudaMemcpyAsync((char*)c->taps_stage[i] + (size_t)r0 * row_bytes,
                                (const char*)taps[i] + (size_t)r0 * row_bytes, (size_t)(r1 - r0) * row_bytes,
                                cudaMemcpyHostToDevice, c->copy_stream));
    OUT_CK(c, cudaEventRecord(c->chunk_ev[k], c->copy_stream));
  }
  return OUTLETS_OK;
}

outlets_status begin_call(outlets_ctx* c, cudaStream_t s) {
  OUT_CK(c, cudaSetDevice(c->cfg.device));
  c->cur_stream = s;
  if (c->have_prev) OUT_CK(c, cudaStreamWaitEvent(s, c->done_ev, 0));
  return OUTLETS_OK;
}

// Where the head writes z_hat and the length: straight into the caller's
// buffers when they are device memory (no copy after the head, so the next
// call's first kernel can start under this call's last one), else into the
// context's buffers, copied out by end_call.
struct OutDst {
  float* z;
  float* len;
};
OutDst out_dst(outlets_ctx* c, float* z_out, float* len_out) {
  return {is_device_ptr(z_out) ? z_out : c->z, (len_out && is_device_ptr(len_out)) ? len_out : c->len};
}

outlets_status end_call(outlets_ctx* c, int out_rows, float* z_out, float* len_out, const OutDst& od,
                        cudaStream_t s) {
  if (z_out != od.z) OUT_CK(c, cudaMemcpyAsync(z_out, od.z, (size_t)out_rows * 4, cudaMemcpyDefault, s));
  if (len_out && len_out != od.len)
    OUT_CK(c, cudaMemcpyAsync(len_out, od.len, (size_t)out_rows * 4, cudaMemcpyDefault, s));
  OUT_CK(c, cudaEventRecord(c->done_ev, s));
  c->have_prev = true;
  return OUTLETS_OK;
}

// Device address of outlets_length_head_noalloc's static scratch array
// (defined with that entry point at the end of this file).
cudaError_t head_scratch_ptr(int device, float** out);
outlets_status head_noalloc_run(outlets_ctx* c, const void* h_draft, int rows, float* z_out, float* len_out,
                                cudaStream_t s);
constexpr int kMaxDevices = 64;

}  // namespace

extern "C" {

outlets_status outlets_create(const outlets_config* cfg, const outlets_weights* w, outlets_ctx** out) {
  if (!out) return OUTLETS_EINVAL;
  *out = nullptr;
  if (!cfg || !w) return OUTLETS_EINVAL;
  std::string why;
  if (validate_config(cfg, why) != OUTLETS_OK) {
    std::fprintf(stderr, "outlets_create: %s\n", why.c_str());
    return OUTLETS_EINVAL;
  }
  const float* req[] = {w->w_proj, w->w_q, w->w_k, w->w_v, w->w_o, w->g_in, w->g_post, w->g_final,
                        w->w_gate, w->w_up, w->w_down};
  for (const float* p : req)
    if (!p) return OUTLETS_EINVAL;
  for (int i = 0; i <= cfg->n_head_hidden; ++i)
    if (!w->head_w[i] || !w->head_b[i]) return OUTLETS_EINVAL;
  if (cfg->vocab > 0 && !w->w_lm) return OUTLETS_EINVAL;
  if (cfg->embed_vocab > 0 && (!w->w_embed || !w->g_emb)) return OUTLETS_EINVAL;
  if (cudaSetDevice(cfg->device) != cudaSuccess) {
    cudaGetLastError();
    return OUTLETS_ECUDA;
  }
  int major = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, cfg->device);
  if (cfg->dtype == OUTLETS_BF16 && (major < 10 || !encode_fn())) return OUTLETS_EUNSUPPORTED;

  outlets_ctx* c = new outlets_ctx();
  c->cfg = *cfg;
  c->bf16 = cfg->dtype == OUTLETS_BF16;
  c->esz = c->bf16 ? 2 : 4;
  c->d = cfg->d_model;
  c->H = cfg->n_heads;
  c->KVH = cfg->n_kv_heads;
  c->hd = cfg->head_dim;
  c->F = cfg->ffn_dim;
  c->Fp = (int)cdiv(c->F, 128) * 128;
  c->attn_w = c->H * c->hd;
  c->gated = w->w_attn_gate != nullptr;
  c->qkv_n = (c->H + 2 * c->KVH) * c->hd + (c->gated ? c->attn_w : 0);
  c->EV = cfg->embed_vocab;
  c->qkv_k = c->EV > 0 ? 2 * cfg->d_model : cfg->d_model;
  c->max_rows = std::max(cfg->max_tokens, cfg->max_batch);
  c->V = cfg->vocab;
  c->head_dims.push_back(c->d);
  for (int i = 0; i < cfg->n_head_hidden; ++i) c->head_dims.push_back(cfg->head_hidden[i]);
  c->head_dims.push_back(1);
  cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, cfg->device);

  auto cleanup_fail = [&](outlets_status st) {
    outlets_destroy(c);
    return st;
  };
  // Resolve the no-allocation head's scratch array here, where allocating is
  // allowed: the lookup loads the module that holds the array, which commits
  // its device memory, so that outlets_length_head_noalloc itself never does.
  if (cfg->device < kMaxDevices) {
    float* scratch = nullptr;
    if (head_scratch_ptr(cfg->device, &scratch) != cudaSuccess) {
      cudaGetLastError();
      return cleanup_fail(OUTLETS_ECUDA);
    }
  }
  const int d = c->d;
  const size_t es = c->esz;
  // ---- weights (bf16: k-block-major swizzled, rows padded to a multiple of 768 =
  // lcm of the tile widths 64..256, so every tile's bulk copy stays in bounds)
  auto np_of = [&](int n) -> long long { return c->bf16 ? cdiv(n, 768) * 768 : 0; };
  c->np_proj = np_of(d);
  c->np_qkv = np_of(c->qkv_n);
  c->np_o = np_of(d);
  c->np_gu = np_of(2 * c->Fp);
  c->np_down = np_of(d);
  c->np_h0 = np_of(c->head_dims[1]);
  // draft LM head: rows padded so that a tile of any of its widths (256, 224, 128) stays in bounds
  if (c->V > 0 && c->bf16)
    c->np_lm = std::max({cdiv(c->V, 256) * 256, cdiv(c->V, 224) * 224, cdiv(c->V, 128) * 128});
  auto rows_of = [&](long long np, int n) -> size_t { return (size_t)(np ? np : n); };
  c->w_proj = c->alloc(rows_of(c->np_proj, d) * 3 * d * es);
  c->w_qkv = c->alloc(rows_of(c->np_qkv, c->qkv_n) * c->qkv_k * es);
  c->w_o = c->alloc(rows_of(c->np_o, d) * c->attn_w * es);
  c->w_gu = c->alloc(rows_of(c->np_gu, 2 * c->Fp) * d * es);
  c->w_down = c->alloc(rows_of(c->np_down, d) * c->Fp * es);
  c->g_in = (float*)c->alloc((size_t)d * 4);
  c->g_post = (float*)c->alloc((size_t)d * 4);
  c->g_final = (float*)c->alloc((size_t)d * 4);
  const int nl = (int)c->head_dims.size() - 1;
  c->head_wf.assign(nl, nullptr);
  c->head_b.assign(nl, nullptr);
  c->head_w0 = c->alloc(rows_of(c->np_h0, c->head_dims[1]) * d * es);
  for (int i = 1; i < nl; ++i) c->head_wf[i] = (float*)c->alloc((size_t)c->head_dims[i + 1] * c->head_dims[i] * 4);
  for (int i = 0; i < nl; ++i) c->head_b[i] = (float*)c->alloc((size_t)c->head_dims[i + 1] * 4);
  if (c->EV > 0) {
    c->w_embed = c->alloc((size_t)c->EV * d * es);
    c->g_emb = (float*)c->alloc((size_t)d * 4);
  }
  if (c->V > 0) {
    c->w_lm = c->alloc(rows_of(c->np_lm, c->V) * d * es);
    c->lm_rows_cap = std::min(c->max_rows, kLmRowsPerPass);
    // partial tiles per row: two column halves of every 128-wide tile (tensor-core path)
    const size_t tiles = c->bf16 ? 2 * (size_t)cdiv(c->V, 128) : (size_t)cdiv(c->V, kLmTileF32);
    c->lm_stats = (float2*)c->alloc((size_t)c->lm_rows_cap * tiles * sizeof(float2));
    c->lm_top = (int2*)c->alloc((size_t)c->lm_rows_cap * tiles * OUTLETS_MAX_TOPK * sizeof(int2));
    c->lm_bound = (int*)c->alloc((size_t)c->lm_rows_cap * kLmBoundSlots * sizeof(int));
    c->lm_ids = (int*)c->alloc((size_t)c->max_rows * OUTLETS_MAX_TOPK * sizeof(int));
    c->lm_lp = (float*)c->alloc((size_t)c->max_rows * OUTLETS_MAX_TOPK * 4);
    c->lm_lse = (float*)c->alloc((size_t)c->max_rows * 4);
    if (!c->bf16) c->lm_logits_ws = (float*)c->alloc((size_t)c->lm_rows_cap * c->V * 4);
  }
  c->rope_cos = (float*)c->alloc((size_t)cfg->max_position * (c->hd / 2) * 4);
  c->rope_sin = (float*)c->alloc((size_t)cfg->max_position * (c->hd / 2) * 4);
  // ---- workspace
  const size_t R = (size_t)c->max_rows;
  c->f = (float*)c->alloc(R * d * 4);
  c->a = (float*)c->alloc(R * d * 4);
  c->y = (float*)c->alloc(R * d * 4);
  c->xhat = c->alloc(R * d * es);
  c->ahat = c->alloc(R * d * es);
  c->hn = c->alloc(R * d * es);
  if (c->EV > 0) c->ehat = c->alloc(R * d * es);
  if (c->bf16) {  // RMSNorm gains folded into the consuming weights
    c->fold = true;
    c->ones = (float*)c->alloc((size_t)d * 4);
    c->ss_stride = (int)cdiv(d, 64);
    c->ss_f = (float*)c->alloc(R * c->ss_stride * 4);
    c->ss_a = (float*)c->alloc(R * c->ss_stride * 4);
  }
  c->qkv = c->alloc(R * c->qkv_n * es);
  c->q = c->alloc(R * c->attn_w * es);
  if (c->gated) c->gate_act = c->alloc(R * c->attn_w * es);
  c->attn = c->alloc(R * c->attn_w * es);
  c->kh = c->alloc((size_t)c->KVH * cfg->max_tokens * c->hd * es);
  c->vh = c->alloc((size_t)c->KVH * cfg->max_tokens * c->hd * es);
  if (c->bf16) {  // every sequence starts at a column that is a multiple of 8
    c->vt_ld = (long long)cdiv((long long)cfg->max_tokens + 8LL * cfg->max_batch, 64) * 64;
    c->vt = c->alloc((size_t)c->KVH * c->hd * c->vt_ld * es);
  }
  c->u = c->alloc(R * c->Fp * es);
  if (!c->bf16) c->gu32 = (float*)c->alloc(R * 2 * c->Fp * 4);
  if (c->bf16) {
    c->last_x = c->alloc((size_t)cfg->max_batch * d * es);
    if (c->EV > 0) c->last_e = c->alloc((size_t)cfg->max_batch * d * es);
    c->last_f = (float*)c->alloc((size_t)cfg->max_batch * d * 4);
    c->last_part_items = (size_t)cfg->max_batch + (size_t)cdiv(cfg->max_tokens, kSplitLen);
    c->last_part_o = (float*)c->alloc(c->last_part_items * c->H * c->hd * 4);
    c->last_part_ml = (float*)c->alloc(c->last_part_items * c->H * 2 * 4);
  }
  int hmax = 1;
  for (size_t i = 1; i < c->head_dims.size(); ++i) hmax = std::max(hmax, c->head_dims[i]);
  c->h1a = (float*)c->alloc(R * hmax * 4);
  c->h1b = (float*)c->alloc(R * hmax * 4);
  c->z = (float*)c->alloc(R * 4);
  c->len = (float*)c->alloc(R * 4);
  c->err_dev = (int*)c->alloc(16);
  c->dec_count = (int*)c->alloc((size_t)cfg->max_batch * c->KVH * sizeof(int));
  if (c->bf16) {  // f32 split-K slices of the small-M path (up to 12 of the widest GEMM)
    const size_t widest = (size_t)std::max(std::max(d, c->qkv_n), c->head_dims[1]);
    c->part_floats = (size_t)12 * std::min<size_t>(R, 256) * widest;
    c->part = (float*)c->alloc(c->part_floats * 4);
  }
  if (c->oom) return cleanup_fail(OUTLETS_ENOMEM);
  // metadata slots sized for the largest call up front (growing one later
  // allocates and synchronizes): prefill attention items (8 ints per 128-row
  // tile and head), per-sequence arrays, page lists
  const size_t meta_ints = (size_t)8 * c->H * (cdiv(cfg->max_tokens, 128) + cfg->max_batch) +
                           (size_t)8 * (cfg->max_batch + 1) + (size_t)2 * (cdiv(cfg->max_tokens, 64) + cfg->max_batch) +
                           (c->EV > 0 ? R : 0) + (1u << 16);
  for (auto& p : c->ring) {
    if (cudaEventCreateWithFlags(&p.ev, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&p.done, cudaEventDisableTiming) != cudaSuccess)
      return cleanup_fail(OUTLETS_ECUDA);
    if (cudaMallocHost(&p.h, meta_ints * sizeof(int)) != cudaSuccess) {
      cudaGetLastError();
      return cleanup_fail(OUTLETS_ENOMEM);
    }
    p.cap = meta_ints;
    if (cudaMalloc(&p.dev, meta_ints * sizeof(int)) != cudaSuccess) {
      cudaGetLastError();
      return cleanup_fail(OUTLETS_ENOMEM);
    }
    p.dev_cap = meta_ints;
  }
  if (cudaEventCreateWithFlags(&c->done_ev, cudaEventDisableTiming) != cudaSuccess) return cleanup_fail(OUTLETS_ECUDA);

  // ---- upload
  size_t stage_floats = (size_t)16 << 20;  // 64 MB staging
  float* stage = nullptr;
  if (cudaMalloc(&stage, stage_floats * 4) != cudaSuccess) {
    cudaGetLastError();
    return cleanup_fail(OUTLETS_ENOMEM);
  }
  // keep interleaved uploads chunked on 128-row boundaries
  const size_t il_floats = std::max<size_t>((stage_floats / d) / 128 * 128, 128) * d;
  outlets_status st = OUTLETS_OK;
  auto up = [&](const float* src, int rows, int cols, void* dst, long long ld, int mode, int base, long long np,
                const float* col_scale = nullptr) {
    if (st == OUTLETS_OK)
      st = upload_rows(c, src, rows, cols, dst, ld, mode, base, np, stage, mode == 0 ? stage_floats : il_floats,
                       col_scale);
  };
  // column scales folding the RMSNorm gains into the weights that read the
  // normalized rows (bf16 path): QKV columns of the fused feature by g_in,
  // gate/up columns by g_post (the embedding columns keep g_emb in their norm)
  float *qkv_scale = nullptr, *gu_scale = nullptr;
  if (c->fold) {
    std::vector<float> one(d, 1.0f), qs((size_t)c->qkv_k, 1.0f);
    std::memcpy(qs.data() + (c->qkv_k - d), w->g_in, (size_t)d * 4);
    if (cudaMalloc(&qkv_scale, qs.size() * 4) != cudaSuccess || cudaMalloc(&gu_scale, (size_t)d * 4) != cudaSuccess) {
      cudaGetLastError();
      cudaFree(stage);
      cudaFree(qkv_scale);
      return cleanup_fail(OUTLETS_ENOMEM);
    }
    if (cudaMemcpy(qkv_scale, qs.data(), qs.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(gu_scale, w->g_post, (size_t)d * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(c->ones, one.data(), (size_t)d * 4, cudaMemcpyHostToDevice) != cudaSuccess)
      st = OUTLETS_ECUDA;
  }
  up(w->w_proj, d, 3 * d, c->w_proj, 3 * d, 0, 0, c->np_proj);
  const int qk = c->qkv_k;
  up(w->w_q, c->H * c->hd, qk, c->w_qkv, qk, 0, 0, c->np_qkv, qkv_scale);
  up(w->w_k, c->KVH * c->hd, qk, c->w_qkv, qk, 0, c->H * c->hd, c->np_qkv, qkv_scale);
  up(w->w_v, c->KVH * c->hd, qk, c->w_qkv, qk, 0, (c->H + c->KVH) * c->hd, c->np_qkv, qkv_scale);
  if (c->gated)
    up(w->w_attn_gate, c->attn_w, qk, c->w_qkv, qk, 0, (c->H + 2 * c->KVH) * c->hd, c->np_qkv, qkv_scale);
  if (c->EV > 0) up(w->w_embed, c->EV, d, c->w_embed, d, 0, 0, 0);
  up(w->w_o, d, c->attn_w, c->w_o, c->attn_w, 0, 0, c->np_o);
  up(w->w_gate, c->F, d, c->w_gu, d, 1, 0, c->np_gu, gu_scale);
  up(w->w_up, c->F, d, c->w_gu, d, 2, 0, c->np_gu, gu_scale);
  up(w->w_down, d, c->F, c->w_down, c->Fp, 0, 0, c->np_down);
  up(w->head_w[0], c->head_dims[1], d, c->head_w0, d, 0, 0, c->np_h0);
  if (c->V > 0) up(w->w_lm, c->V, d, c->w_lm, d, 0, 0, c->np_lm);
  cudaFree(stage);
  cudaFree(qkv_scale);
  cudaFree(gu_scale);
  if (st != OUTLETS_OK) return cleanup_fail(st);
  auto h2d = [&](void* dst, const void* src, size_t bytes) {
    if (st == OUTLETS_OK && cudaMemcpy(dst, src, bytes, cudaMemcpyHostToDevice) != cudaSuccess) st = OUTLETS_ECUDA;
  };
  h2d(c->g_in, w->g_in, (size_t)d * 4);
  h2d(c->g_post, w->g_post, (size_t)d * 4);
  h2d(c->g_final, w->g_final, (size_t)d * 4);
  if (c->EV > 0) h2d(c->g_emb, w->g_emb, (size_t)d * 4);
  for (int i = 1; i < nl; ++i) h2d(c->head_wf[i], w->head_w[i], (size_t)c->head_dims[i + 1] * c->head_dims[i] * 4);
  for (int i = 0; i < nl; ++i) h2d(c->head_b[i], w->head_b[i], (size_t)c->head_dims[i + 1] * 4);
  // RoPE table, angles in fp64: pos * theta^(-2i/hd)
  {
    const int half = c->hd / 2;
    std::vector<float> cs((size_t)cfg->max_position * half), sn((size_t)cfg->max_position * half);
    for (int i = 0; i < half; ++i) {
      const double inv = std::pow((double)cfg->rope_theta, -2.0 * i / c->hd);
      for (int p = 0; p < cfg->max_position; ++p) {
        const double ang = (double)p * inv;
        cs[(size_t)p * half + i] = (float)std::cos(ang);
        sn[(size_t)p * half + i] = (float)std::sin(ang);
      }
    }
    h2d(c->rope_cos, cs.data(), cs.size() * 4);
    h2d(c->rope_sin, sn.data(), sn.size() * 4);
  }
  if (st != OUTLETS_OK) return cleanup_fail(st);
  // One no-allocation head call on a zero row: under lazy module loading this
  // loads every kernel that entry point launches (loading commits device
  // memory), so that its later calls allocate nothing.
  if (cfg->device < kMaxDevices) {
    if (cudaMemset(c->hn, 0, (size_t)d * es) != cudaSuccess) return cleanup_fail(OUTLETS_ECUDA);
    st = head_noalloc_run(c, c->hn, 1, c->h1a, c->h1b, nullptr);
    if (st != OUTLETS_OK) return cleanup_fail(st);
  }
  if (cudaDeviceSynchronize() != cudaSuccess) {
    cudaGetLastError();
    return cleanup_fail(OUTLETS_ECUDA);
  }
  *out = c;
  return OUTLETS_OK;
}

void outlets_destroy(outlets_ctx* c) {
  if (!c) return;
  cudaSetDevice(c->cfg.device);
  cudaDeviceSynchronize();
  for (void* p : c->allocs)
    if (p) cudaFree(p);
  for (auto& p : c->ring) {
    if (p.h) cudaFreeHost(p.h);
    if (p.dev) cudaFree(p.dev);
    if (p.ev) cudaEventDestroy(p.ev);
    if (p.done) cudaEventDestroy(p.done);
  }
  if (c->done_ev) cudaEventDestroy(c->done_ev);
  for (cudaEvent_t e : c->ev_pool) cudaEventDestroy(e);
  if (c->copy_start) cudaEventDestroy(c->copy_start);
  for (cudaEvent_t e : c->chunk_ev)
    if (e) cudaEventDestroy(e);
  if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
  delete c;
}

outlets_status outlets_selftest_bounded_wait(outlets_ctx* c, uint64_t timeout_ns, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  if (timeout_ns < 1000 || timeout_ns > 1000000000ull)
    return c->fail(OUTLETS_EINVAL, "timeout_ns must be in [1 us, 1 s]");
  OUT_CK(c, cudaSetDevice(c->cfg.device));
  OUT_CK(c, wait_selftest_launch(c->err_dev, timeout_ns, (cudaStream_t)stream));
  return OUTLETS_OK;
}

outlets_status outlets_profile_enable(outlets_ctx* c, int32_t enable) {
  if (!c) return OUTLETS_EINVAL;
  OUT_CK(c, cudaSetDevice(c->cfg.device));
  OUT_CK(c, cudaDeviceSynchronize());
  c->prof = static_cast<unsigned>(enable) & ((1u << OUTLETS_N_STAGES) - 1u);
  c->recs.clear();
  c->ev_used = 0;
  return OUTLETS_OK;
}

outlets_status outlets_profile_read(outlets_ctx* c, double* ms, int32_t* count) {
  if (!c || !ms) return OUTLETS_EINVAL;
  OUT_CK(c, cudaSetDevice(c->cfg.device));
  for (int i = 0; i < OUTLETS_N_STAGES; ++i) {
    ms[i] = 0.0;
    if (count) count[i] = 0;
  }
  for (const auto& r : c->recs) {
    OUT_CK(c, cudaEventSynchronize(r.b));
    float t = 0.f;
    OUT_CK(c, cudaEventElapsedTime(&t, r.a, r.b));
    ms[r.stage] += t;
    if (count) count[r.stage] += 1;
  }
  c->recs.clear();
  c->ev_used = 0;
  return OUTLETS_OK;
}

const char* outlets_stage_name(int32_t s) {
  static const char* names[OUTLETS_N_STAGES] = {"fc_gemm",      "rmsnorm_in",     "qkv_gemm",    "rope_scatter",
                                                "attention",    "o_gemm",         "rmsnorm_post", "gateup_swiglu_gemm",
                                                "down_gemm",    "final_rmsnorm",  "length_head",
                                                "draft_head"};
  return (s >= 0 && s < OUTLETS_N_STAGES) ? names[s] : "";
}

uint64_t outlets_launch_count(const outlets_ctx* c) { return c ? (uint64_t)c->launches : 0; }

const char* outlets_last_error(const outlets_ctx* c) { return c ? c->err.c_str() : "null context"; }

size_t outlets_device_bytes(const outlets_ctx* c) { return c ? c->dev_bytes : 0; }

outlets_status outlets_kv_create(outlets_ctx* c, int32_t max_slots, int32_t max_tokens_total, outlets_kv** out) {
  if (!out) return OUTLETS_EINVAL;
  *out = nullptr;
  if (!c) return OUTLETS_EINVAL;
  if (max_slots <= 0 || max_tokens_total <= 0) return c->fail(OUTLETS_EINVAL, "max_slots and max_tokens_total must be positive");
  OUT_CK(c, cudaSetDevice(c->cfg.device));
  outlets_kv* kv = new outlets_kv();
  kv->ctx = c;
  kv->device = c->cfg.device;
  kv->max_slots = max_slots;
  kv->num_pages = (int)cdiv(max_tokens_total, kPageTokens) + max_slots;
  kv->max_pages_per_slot = (int)cdiv(c->cfg.max_position, kPageTokens);
  const size_t pool = (size_t)kv->num_pages * c->KVH * kPageTokens * c->hd * c->esz;
  kv->part_items = (size_t)c->cfg.max_batch + kv->num_pages;
  auto a = [&](size_t bytes) -> void* {
    void* p = nullptr;
    if (cudaMalloc(&p, bytes) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    cudaMemset(p, 0, bytes);
    kv->allocs.push_back(p);
    return p;
  };
  kv->k_pool = a(pool);
  kv->v_pool = a(pool);
  kv->part_o = (float*)a(kv->part_items * c->H * c->hd * 4);
  kv->part_ml = (float*)a(kv->part_items * c->H * 2 * 4);
  if (!kv->k_pool || !kv->v_pool || !kv->part_o || !kv->part_ml) {
    outlets_kv_destroy(kv);
    return c->fail(OUTLETS_ENOMEM, "KV pool allocation failed");
  }
  kv->len.assign(max_slots, 0);
  kv->pages.assign(max_slots, {});
  kv->free_list.reserve(kv->num_pages);
  for (int p = kv->num_pages - 1; p >= 0; --p) kv->free_list.push_back(p);
  *out = kv;
  return OUTLETS_OK;
}

void outlets_kv_destroy(outlets_kv* kv) {
  if (!kv) return;
  cudaSetDevice(kv->device);
  cudaDeviceSynchronize();
  for (void* p : kv->allocs) cudaFree(p);
  delete kv;
}

outlets_status outlets_kv_truncate(outlets_kv* kv, int32_t slot, int32_t length) {
  if (!kv || slot < 0 || slot >= kv->max_slots || length < 0 || length > kv->len[slot]) return OUTLETS_EINVAL;
  const size_t keep = (size_t)cdiv(length, kPageTokens);
  while (kv->pages[slot].size() > keep) {
    kv->free_list.push_back(kv->pages[slot].back());
    kv->pages[slot].pop_back();
  }
  kv->len[slot] = length;
  return OUTLETS_OK;
}

outlets_status outlets_kv_reset_slot(outlets_kv* kv, int32_t slot) {
  if (!kv || slot < 0 || slot >= kv->max_slots) return OUTLETS_EINVAL;
  for (int p : kv->pages[slot]) kv->free_list.push_back(p);
  kv->pages[slot].clear();
  kv->len[slot] = 0;
  return OUTLETS_OK;
}

int32_t outlets_kv_slot_length(const outlets_kv* kv, int32_t slot) {
  if (!kv || slot < 0 || slot >= kv->max_slots) return -1;
  return kv->len[slot];
}

int32_t outlets_kv_free_pages(const outlets_kv* kv) { return kv ? (int32_t)kv->free_list.size() : -1; }

outlets_status outlets_check(outlets_ctx* c, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  OUT_CK(c, cudaSetDevice(c->cfg.device));
  OUT_CK(c, cudaStreamSynchronize((cudaStream_t)stream));
  int e = 0;
  OUT_CK(c, cudaMemcpy(&e, c->err_dev, sizeof(int), cudaMemcpyDeviceToHost));
  if (e) {
    OUT_CK(c, cudaMemset(c->err_dev, 0, sizeof(int)));
    // a CTA that gave up may have left a split counter mid-count
    OUT_CK(c, cudaMemset(c->dec_count, 0, (size_t)c->cfg.max_batch * c->KVH * sizeof(int)));
    if (e & ERR_TIMEOUT) return c->fail(OUTLETS_ETIMEOUT, "a kernel's bounded wait ran out");
    return c->fail(OUTLETS_EDEVICE, "a kernel refused an out-of-range index");
  }
  return OUTLETS_OK;
}

}  // extern "C"

namespace {

// Token ids of the input-embedding branch: required exactly when the context
// has the branch; host ids are range-checked here (device ids by the kernel).
outlets_status check_tokens(outlets_ctx* c, const int32_t* tokens, long long n) {
  if (c->EV == 0) {
    if (tokens) return c->fail(OUTLETS_EINVAL, "token ids given, but the context has no input-embedding branch");
    return OUTLETS_OK;
  }
  if (!tokens)
    return c->fail(OUTLETS_EINVAL, "the context has the input-embedding branch: pass token ids (the *_ex calls)");
  if (!is_device_ptr(tokens))
    for (long long i = 0; i < n; ++i)
      if (tokens[i] < 0 || tokens[i] >= c->EV) return c->fail(OUTLETS_EINVAL, "token id outside 0 .. embed_vocab-1");
  return OUTLETS_OK;
}

// Split-KV work of decode attention over requests with seq_len[b] keys each.
// Keys per work item: about a third of one resident CTA's share of all keys
// (never below 512), so most requests need no split (and no merge) while the
// longest items still fit several times into the whole pass.  Launch order:
// longest items first (the short ones fill the tail).
struct DecodeWork {
  int split_len = 0, max_splits = 1, n_work = 0;
  std::vector<int> work, work_off, order;  // (request, split) pairs, [B+1] offsets, launch order
};
DecodeWork decode_work(const outlets_ctx* c, const std::vector<int>& seq_len) {
  DecodeWork w;
  const int B = (int)seq_len.size();
  long long total_keys = 0;
  for (int b = 0; b < B; ++b) total_keys += seq_len[b];
  const long long share = cdiv(total_keys * c->KVH, 3LL * kDecodeCtasPerSm * c->num_sms);
  w.split_len = (int)std::max<long long>(kSplitLen, cdiv(share, kPageTokens) * kPageTokens);
  w.work_off.assign(B + 1, 0);
  for (int b = 0; b < B; ++b) {
    const int ns = (int)cdiv(seq_len[b], w.split_len);
    w.max_splits = std::max(w.max_splits, ns);
    for (int sp = 0; sp < ns; ++sp) {
      w.work.push_back(b);
      w.work.push_back(sp);
    }
    w.work_off[b + 1] = (int)(w.work.size() / 2);
  }
  w.n_work = w.work_off[B];
  std::vector<int> item_keys(w.n_work);
  w.order.resize(w.n_work);
  for (int i = 0; i < w.n_work; ++i) {
    w.order[i] = i;
    item_keys[i] = std::min(w.split_len, seq_len[w.work[2 * i]] - w.work[2 * i + 1] * w.split_len);
  }
  std::stable_sort(w.order.begin(), w.order.end(), [&](int x, int y) { return item_keys[x] > item_keys[y]; });
  return w;
}

// Static prediction of the last rows only: x_hat (and the embedding half of
// the layer input) of each sequence's last row, its q / k / v projection, and
// RoPE of q at position L - 1 into rows 0 .. B-1 of c->q (the gate of gated
// attention into rows 0 .. B-1 of c->gate_act).  The keys and values of
// every row were written by the front.
outlets_status run_last_q(outlets_ctx* c, int B, const int* last_dev, const int* pos_dev, cudaStream_t s) {
  const int d = c->d;
  c->stage_begin(OUTLETS_S_QKV);
  // g_in is folded into W_qkv: the norm has unit gains
  OUT_CK(c, rmsnorm_gather_launch<bf16>(c->f, last_dev, c->ones, (bf16*)c->last_x, B, d, c->cfg.rms_eps, s));
  int n = 2;
  const void* a1[3] = {c->last_x, c->last_x, c->last_x};
  int pieces = 1;
  if (c->EV > 0) {
    OUT_CK(c, gather_rows_launch(c->ehat, last_dev, c->last_e, B, (long long)d * c->esz, s));
    a1[0] = c->last_e;
    a1[1] = c->last_x;
    pieces = 2;
    ++n;
  }
  QkvSrc q;
  if (small_path(c, B)) {
    int sl = 1;
    OUT_TRY(gemm_split(c, a1, pieces, d, d, B, c->w_qkv, c->np_qkv, c->qkv_n, c->qkv_k, c->part, &sl, s));
    q = {c->part, true, sl, (long long)B * c->qkv_n};
  } else {
    OUT_TRY(gemm_tc(c, a1, pieces, d, d, B, c->w_qkv, c->np_qkv, c->qkv_n, c->qkv_k, EPI_ACT, c->qkv, c->qkv_n, nullptr,
                    0, nullptr, s));
    q = {c->qkv, false, 1, 0};
  }
  c->stage_end(n);
  c->stage_begin(OUTLETS_S_ROPE);
  RopeArgs ra{};
  ra.T = B;
  ra.H = c->H;
  ra.KVH = c->KVH;
  ra.hd = c->hd;
  ra.B = B;
  ra.pos = pos_dev;
  ra.cos_tab = c->rope_cos;
  ra.sin_tab = c->rope_sin;
  ra.max_pos = c->cfg.max_position;
  ra.q_out = c->q;
  ra.kv_ld_rows = c->cfg.max_tokens;
  ra.qkv_ld = c->qkv_n;
  ra.gate_out = c->gated ? c->gate_act : nullptr;
  ra.err = c->err_dev;
  OUT_TRY(launch_rope(c, q, ra, s));
  c->stage_end(1);
  return OUTLETS_OK;
}

outlets_status predict_prefill(outlets_ctx* c, const void* const taps[3], const int32_t* tokens, const int32_t* cu,
                               int32_t B, int32_t T, outlets_kv* kv, const int32_t* slots, uint32_t flags,
                               float* z_out, float* len_out, const outlets_draft_out* draft, void* stream) {
  cudaStream_t s = (cudaStream_t)stream;
  if (!taps || !cu || !z_out) return c->fail(OUTLETS_EINVAL, "taps, cu_seqlens and z_out must not be NULL");
  if (flags & ~(OUTLETS_ALL_TOKENS | OUTLETS_KEEP_ROWS)) return c->fail(OUTLETS_EINVAL, "unknown flag");
  if (B < 0 || T < 0) return c->fail(OUTLETS_EINVAL, "B and T must be >= 0");
  if ((kv == nullptr) != (slots == nullptr)) return c->fail(OUTLETS_EINVAL, "kv and slots go together");
  if (kv && kv->ctx != c) return c->fail(OUTLETS_EINVAL, "kv belongs to another context");
  if (B == 0) {
    if (T != 0) return c->fail(OUTLETS_EINVAL, "T must be 0 when B is 0");
    return OUTLETS_OK;
  }
  if (cu[0] != 0) return c->fail(OUTLETS_EINVAL, "cu_seqlens[0] must be 0");
  int max_len = 0;
  for (int b = 0; b < B; ++b) {
    if (cu[b + 1] <= cu[b]) return c->fail(OUTLETS_EINVAL, "cu_seqlens must be strictly increasing (every sequence non-empty)");
    max_len = std::max(max_len, cu[b + 1] - cu[b]);
  }
  if (cu[B] != T) return c->fail(OUTLETS_EINVAL, "cu_seqlens[B] must equal T");
  if (T > c->cfg.max_tokens) return c->fail(OUTLETS_ECAPACITY, "T exceeds max_tokens");
  OUT_TRY(check_tokens(c, tokens, T));
  if (B > c->cfg.max_batch) return c->fail(OUTLETS_ECAPACITY, "B exceeds max_batch");
  if (max_len > c->cfg.max_position) return c->fail(OUTLETS_ECAPACITY, "a sequence is longer than max_position");
  if (kv) {
    std::vector<char> seen(kv->max_slots, 0);
    long long need = 0, freed = 0;
    for (int b = 0; b < B; ++b) {
      const int sl = slots[b];
      if (sl < 0 || sl >= kv->max_slots) return c->fail(OUTLETS_EINVAL, "slot out of range");
      if (seen[sl]) return c->fail(OUTLETS_EINVAL, "slots must be distinct");
      seen[sl] = 1;
      need += cdiv(cu[b + 1] - cu[b], kPageTokens);
      freed += (long long)kv->pages[sl].size();
    }
    if (need > (long long)kv->free_list.size() + freed) return c->fail(OUTLETS_ECAPACITY, "not enough free KV pages");
  }
  const bool all_tokens = flags & OUTLETS_ALL_TOKENS;
  const int out_rows = all_tokens ? T : B;
  // Only each sequence's last row is predicted, and the layer's output at a
  // row feeds nothing but that row's prediction: every row needs its keys and
  // values (attention of the last rows, the cache), only the last rows need
  // queries, attention, O, the MLP, the final norm and the head.
  const bool prune = c->bf16 && !all_tokens && !(flags & OUTLETS_KEEP_ROWS) && !small_path(c, T);

  OUT_TRY(begin_call(c, s));
  CallSlot slot_guard{c, s};
  c->last_kind = 0;
  // Large calls with host taps overlap the copy with the front of the pipeline
  // (FC, input norm, QKV, RoPE are row-wise): rows run in chunks of whole
  // 128-row tiles as their taps land.
  // A chunk's FC tiles (256 x 256; d / 256 of them per 256 rows) are a whole
  // number of waves over the SMs where such a chunk is small enough (at most
  // kMaxTapChunks of them); else the chunks are equal, in whole 128-row tiles.
  int n_chunks = 1, chunk_rows = T;
  if (c->bf16 && !small_path(c, T) && !is_device_ptr(taps[0]) && !is_device_ptr(taps[1]) && !is_device_ptr(taps[2])) {
    const long long ntn = cdiv(c->d, 256);
    const long long unit = 256LL * (c->num_sms / std::gcd((long long)c->num_sms, ntn));  // rows of whole waves
    const long long per = cdiv(T, kMaxTapChunks);
    const long long aligned = cdiv(per, unit) * unit;
    if (aligned * 2 <= T) {
      chunk_rows = (int)aligned;
    } else {
      const int n = std::max(1, std::min(8, T / kMinTapChunkRows));
      chunk_rows = (int)(cdiv(cdiv(T, n), 128) * 128);
    }
    n_chunks = (int)cdiv(T, chunk_rows);
    if (n_chunks < 2) {
      n_chunks = 1;
      chunk_rows = T;
    }
  }

  // ---- host metadata
  MetaBuilder mb;
  const size_t off_cu = mb.put(cu, B + 1);
  const bool tok_host = tokens && !is_device_ptr(tokens);
  const size_t off_tok = tok_host ? mb.put(tokens, T) : 0;
  std::vector<int> last(B);
  for (int b = 0; b < B; ++b) last[b] = cu[b + 1] - 1;
  const size_t off_last = mb.put(last);
  std::vector<int> pos_last(B);
  for (int b = 0; b < B; ++b) pos_last[b] = cu[b + 1] - cu[b] - 1;
  const size_t off_pos_last = prune ? mb.put(pos_last) : 0;
  size_t off_items = 0, off_vstart = 0;
  int n_items = 0;
  DecodeWork lw;  // pruned: decode attention of each prompt's last row over its head-major keys
  size_t off_lsl = 0, off_lpl = 0, off_lpo = 0, off_lw = 0, off_lwo = 0, off_lord = 0;
  if (prune) {
    std::vector<int> lsl(B), lpl, lpo(B + 1, 0);
    for (int b = 0; b < B; ++b) {
      lsl[b] = cu[b + 1] - cu[b];
      for (int p0 = 0; p0 < lsl[b]; p0 += kPageTokens) lpl.push_back(cu[b] + p0);  // page id = first row
      lpo[b + 1] = (int)lpl.size();
    }
    lw = decode_work(c, lsl);
    if ((size_t)lw.n_work > c->last_part_items) return c->fail(OUTLETS_ECAPACITY, "split-KV partial buffer too small");
    off_lsl = mb.put(lsl);
    off_lpl = mb.put(lpl);
    off_lpo = mb.put(lpo);
    off_lw = mb.put(lw.work);
    off_lwo = mb.put(lw.work_off);
    off_lord = mb.put(lw.order);
  } else if (c->bf16) {
    // tcgen05 attention work items: 128-row query tiles x query heads, the
    // ones with the most key tiles first; V^T columns of each sequence start
    // at a multiple of 8
    std::vector<int> vstart(B);
    long long col = 0;
    for (int b = 0; b < B; ++b) {
      vstart[b] = (int)col;
      col += cdiv(cu[b + 1] - cu[b], 8) * 8;
    }
    if (col > c->vt_ld) return c->fail(OUTLETS_ECAPACITY, "V^T workspace too small");
    off_vstart = mb.put(vstart);
    std::vector<std::pair<int, int>> tiles;  // (n_kv, tile id)
    std::vector<int> tq;                    // per tile: b, tile index
    for (int b = 0; b < B; ++b) {
      const int L = cu[b + 1] - cu[b];
      for (int i = 0; i * 128 < L; ++i) {
        tiles.push_back({i + 1, (int)(tq.size() / 2)});
        tq.push_back(b);
        tq.push_back(i);
      }
    }
    std::stable_sort(tiles.begin(), tiles.end(), [](const auto& x, const auto& y) { return x.first > y.first; });
    std::vector<int> items;
    items.reserve(tiles.size() * c->H * 8);
    for (auto& t : tiles) {
      const int b = tq[2 * t.second], i = tq[2 * t.second + 1];
      const int L = cu[b + 1] - cu[b];
      for (int h = 0; h < c->H; ++h) {
        const int v[8] = {cu[b] + 128 * i, std::min(128, L - 128 * i), cu[b], L, vstart[b], h, i + 1, 128 * i};
        items.insert(items.end(), v, v + 8);
      }
    }
    n_items = (int)(items.size() / 8);
    off_items = mb.put(items);
  }
  size_t off_pl = 0, off_po = 0;
  if (kv) {
    // commit the cache change: reset every slot of the batch, then allocate its pages
    for (int b = 0; b < B; ++b) outlets_kv_reset_slot(kv, slots[b]);
    std::vector<int> pl, po(B + 1, 0);
    for (int b = 0; b < B; ++b) {
      const int L = cu[b + 1] - cu[b];
      const int np = (int)cdiv(L, kPageTokens);
      for (int i = 0; i < np; ++i) {
        const int p = kv->free_list.back();
        kv->free_list.pop_back();
        kv->pages[slots[b]].push_back(p);
        pl.push_back(p);
      }
      kv->len[slots[b]] = L;
      po[b + 1] = (int)pl.size();
    }
    off_pl = mb.put(pl);
    off_po = mb.put(po);
  }
  OUT_TRY(upload_meta(c, mb.v, s));
  // taps after the metadata: both go through the copy stream, and the call's
  // stream waits for the metadata before its first kernel
  const void* tp[3];
  if (n_chunks > 1) OUT_TRY(stage_taps_chunked(c, taps, T, n_chunks, chunk_rows, tp, s));
  else OUT_TRY(prepare_taps(c, taps, T, tp, s));
  const int* m = c->meta_dev;
  const int* cu_dev = m + off_cu;
  const int* tok_dev = tok_host ? m + off_tok : tokens;

  // ---- per row chunk: FC (Eq. 1) -> input RMSNorm -> QKV -> RoPE (q,
  // head-major k/v, cache)
  {
    RopeArgs ra{};
    ra.T = T;
    ra.H = c->H;
    ra.KVH = c->KVH;
    ra.hd = c->hd;
    ra.cu = cu_dev;
    ra.B = B;
    ra.cos_tab = c->rope_cos;
    ra.sin_tab = c->rope_sin;
    ra.max_pos = c->cfg.max_position;
    ra.q_out = c->q;
    ra.k_out = c->kh;
    ra.v_out = c->vh;
    ra.kv_ld_rows = c->cfg.max_tokens;
    if (kv) {
      ra.k_pool = kv->k_pool;
      ra.v_pool = kv->v_pool;
      ra.page_list = m + off_pl;
      ra.page_off = m + off_po;
      ra.page_tokens = kPageTokens;
    }
    ra.qkv_ld = c->qkv_n;
    ra.gate_out = c->gated && !prune ? c->gate_act : nullptr;
    ra.err = c->err_dev;
    if (prune) ra.q_out = nullptr;  // keys and values of every row; queries of the last rows below
    for (int k = 0; k < n_chunks; ++k) {
      const int r0 = k * chunk_rows, rows = std::min(T, r0 + chunk_rows) - r0;
      if (n_chunks > 1) OUT_CK(c, cudaStreamWaitEvent(s, c->chunk_ev[k], 0));
      const size_t off = (size_t)r0 * c->d * c->esz;
      const void* tpc[3] = {(const char*)tp[0] + off, (const char*)tp[1] + off, (const char*)tp[2] + off};
      QkvSrc qsrc;
      OUT_TRY(run_front(c, tpc, rows, &qsrc, s, r0, tok_dev, prune));
      OUT_TRY(wait_meta(c, s));
      c->stage_begin(OUTLETS_S_ROPE);
      ra.row0 = r0;
      ra.T = rows;
      OUT_TRY(launch_rope(c, qsrc, ra, s));
      c->stage_end(1);
    }
  }
  if (prune) OUT_TRY(run_last_q(c, B, m + off_last, m + off_pos_last, s));
  // ---- attention
  c->stage_begin(OUTLETS_S_ATTN);
  if (prune) {
    // each prompt's last row against all its keys: the decode-attention
    // kernels on the head-major K/V ("pages" of 64 rows from the prompt's first)
    DecodeArgs da{};
    da.B = B;
    da.H = c->H;
    da.KVH = c->KVH;
    da.hd = c->hd;
    da.q = c->q;
    da.k_pool = c->kh;
    da.v_pool = c->vh;
    da.page_tokens = kPageTokens;
    da.page_list = m + off_lpl;
    da.page_off = m + off_lpo;
    da.page_stride = 1;
    da.head_stride = c->cfg.max_tokens;
    da.seq_len = m + off_lsl;
    da.work = m + off_lw;
    da.work_off = m + off_lwo;
    da.n_work = lw.n_work;
    da.split_len = lw.split_len;
    da.order = m + off_lord;
    da.max_splits = lw.max_splits;
    da.part_o = c->last_part_o;
    da.part_ml = c->last_part_ml;
    da.combine_count = c->dec_count;
    da.out = c->attn;
    da.gate = c->gate_act;  // null unless gated
    da.err = c->err_dev;
    CUtensorMap km, vm;
    const uint64_t kv_rows = (uint64_t)c->KVH * c->cfg.max_tokens;
    if (!cached_map(c, &km, c->kh, c->hd, kv_rows, c->hd, 64) || !cached_map(c, &vm, c->vh, c->hd, kv_rows, c->hd, 64))
      return c->fail(OUTLETS_ECUDA, "cuTensorMapEncodeTiled failed for the head-major K/V");
    OUT_CK(c, attn_decode_bf16_launch(km, vm, da, s));
  } else if (c->bf16) {
    // V^T for the tcgen05 attention (keys contiguous), then the attention
    OUT_CK(c, v_transpose_launch(c->vh, cu_dev, m + off_vstart, B, T, c->cfg.max_tokens, c->KVH, c->hd, c->vt,
                                 c->vt_ld, s));
    CUtensorMap qm, km, vm;
    const uint64_t kv_rows = (uint64_t)c->KVH * c->cfg.max_tokens;
    if (!cached_map(c, &qm, c->q, c->attn_w, T, c->attn_w, 128) ||
        !cached_map(c, &km, c->kh, c->hd, kv_rows, c->hd, 128) ||
        !cached_map(c, &vm, c->vt, c->vt_ld, (uint64_t)c->KVH * c->hd, c->vt_ld, c->hd))
      return c->fail(OUTLETS_ECUDA, "cuTensorMapEncodeTiled failed for attention");
    OUT_CK(c, attn_prefill_tc_launch(qm, km, vm, reinterpret_cast<const TcAttnItem*>(m + off_items), n_items,
                                     c->cfg.max_tokens, c->H, c->KVH, c->hd, c->attn, c->gate_act, c->err_dev,
                                     c->num_sms, s));
    c->launches += 1;  // the transpose
  } else {
    OUT_CK(c, attn_prefill_simt_launch<float>((const float*)c->q, (const float*)c->kh, (const float*)c->vh, cu_dev,
                                              B, T, c->cfg.max_tokens, c->H, c->KVH, c->hd, (float*)c->attn,
                                              (const float*)c->gate_act, s));
  }
  c->stage_end(1);
  const OutDst od = out_dst(c, z_out, len_out);
  if (prune) {
    // the residual f of the last rows, then O, the MLP, the norm and the head on those rows
    c->stage_begin(OUTLETS_S_O);
    OUT_CK(c, gather_rows_launch(c->f, m + off_last, c->last_f, B, (long long)c->d * 4, s));
    c->stage_end(1);
    OUT_TRY(run_tail(c, B, B, nullptr, od.z, od.len, s, c->last_f));
  } else {
    OUT_TRY(run_tail(c, T, out_rows, all_tokens ? nullptr : m + off_last, od.z, od.len, s, c->f));
  }
  if (draft) OUT_TRY(run_draft(c, c->hn, out_rows, *draft, s));
  c->last_tail_rows = prune ? B : T;
  c->last_rows = T;
  c->last_out_rows = out_rows;
  c->last_kind = 1;
  c->last_slots.clear();
  return end_call(c, out_rows, z_out, len_out, od, s);
}

outlets_status predict_step(outlets_ctx* c, const void* const taps[3], const int32_t* tokens, int32_t B,
                            outlets_kv* kv, const int32_t* slots, float* z_out, float* len_out,
                            const outlets_draft_out* draft, void* stream, bool self_feed = false) {
  cudaStream_t s = (cudaStream_t)stream;
  if ((!taps && !self_feed) || !kv || !slots || !z_out)
    return c->fail(OUTLETS_EINVAL, "taps, kv, slots and z_out must not be NULL");
  if (self_feed) {
    bool same = c->last_kind == 2 && (int)c->last_slots.size() == B;
    for (int b = 0; same && b < B; ++b) same = c->last_slots[b] == slots[b];
    if (!same)
      return c->fail(OUTLETS_EINVAL,
                     "a draft step follows a step or draft step of this context over the same slots, in the same order");
  }
  if (kv->ctx != c) return c->fail(OUTLETS_EINVAL, "kv belongs to another context");
  if (B < 0) return c->fail(OUTLETS_EINVAL, "B must be >= 0");
  if (B == 0) return OUTLETS_OK;
  if (B > c->cfg.max_batch) return c->fail(OUTLETS_ECAPACITY, "B exceeds max_batch");
  OUT_TRY(check_tokens(c, tokens, B));
  std::vector<char> seen(kv->max_slots, 0);
  int need = 0;
  for (int b = 0; b < B; ++b) {
    const int sl = slots[b];
    if (sl < 0 || sl >= kv->max_slots) return c->fail(OUTLETS_EINVAL, "slot out of range");
    if (seen[sl]) return c->fail(OUTLETS_EINVAL, "slots must be distinct");
    seen[sl] = 1;
    if (kv->len[sl] >= c->cfg.max_position) return c->fail(OUTLETS_ECAPACITY, "slot reached max_position");
    if (kv->len[sl] % kPageTokens == 0) ++need;
  }
  if (need > (int)kv->free_list.size()) return c->fail(OUTLETS_ECAPACITY, "not enough free KV pages");

  OUT_TRY(begin_call(c, s));
  CallSlot slot_guard{c, s};
  c->last_kind = 0;  // y is rewritten from here on: a later draft step needs this call to complete
  const void* tp[3] = {nullptr, nullptr, nullptr};
  if (!self_feed) OUT_TRY(prepare_taps(c, taps, B, tp, s));

  // ---- commit the append and build metadata
  std::vector<int> pos(B), seq_len(B), po(B + 1, 0), pl;
  for (int b = 0; b < B; ++b) {
    const int sl = slots[b];
    if (kv->len[sl] % kPageTokens == 0) {
      kv->pages[sl].push_back(kv->free_list.back());
      kv->free_list.pop_back();
    }
    pos[b] = kv->len[sl];
    kv->len[sl] += 1;
    seq_len[b] = kv->len[sl];
    pl.insert(pl.end(), kv->pages[sl].begin(), kv->pages[sl].end());
    po[b + 1] = (int)pl.size();
  }
  const DecodeWork dw = decode_work(c, seq_len);
  const int n_work = dw.n_work, split_len = dw.split_len, max_splits = dw.max_splits;
  MetaBuilder mb;
  const size_t off_pos = mb.put(pos);
  const size_t off_sl = mb.put(seq_len);
  const size_t off_po = mb.put(po);
  const size_t off_pl = mb.put(pl);
  const size_t off_w = mb.put(dw.work);
  const size_t off_wo = mb.put(dw.work_off);
  const size_t off_ord = mb.put(dw.order);
  const bool tok_host = tokens && !is_device_ptr(tokens);
  const size_t off_tok = tok_host ? mb.put(tokens, B) : 0;
  OUT_TRY(upload_meta(c, mb.v, s));
  const int* m = c->meta_dev;

  QkvSrc qsrc;
  OUT_TRY(run_front(c, self_feed ? nullptr : tp, B, &qsrc, s, 0, tok_host ? m + off_tok : tokens));
  OUT_TRY(wait_meta(c, s));  // RoPE is the first kernel that reads the metadata
  c->stage_begin(OUTLETS_S_ROPE);
  {
    RopeArgs ra{};
    ra.T = B;
    ra.H = c->H;
    ra.KVH = c->KVH;
    ra.hd = c->hd;
    ra.B = B;
    ra.pos = m + off_pos;
    ra.cos_tab = c->rope_cos;
    ra.sin_tab = c->rope_sin;
    ra.max_pos = c->cfg.max_position;
    ra.q_out = c->q;
    ra.k_pool = kv->k_pool;
    ra.v_pool = kv->v_pool;
    ra.page_list = m + off_pl;
    ra.page_off = m + off_po;
    ra.page_tokens = kPageTokens;
    ra.qkv_ld = c->qkv_n;
    ra.gate_out = c->gated ? c->gate_act : nullptr;
    ra.err = c->err_dev;
    OUT_TRY(launch_rope(c, qsrc, ra, s));
  }
  c->stage_end(1);
  c->stage_begin(OUTLETS_S_ATTN);
  {
    DecodeArgs da{};
    da.B = B;
    da.H = c->H;
    da.KVH = c->KVH;
    da.hd = c->hd;
    da.q = c->q;
    da.k_pool = kv->k_pool;
    da.v_pool = kv->v_pool;
    da.page_tokens = kPageTokens;
    da.page_list = m + off_pl;
    da.page_off = m + off_po;
    da.page_stride = (long long)c->KVH * kPageTokens;
    da.head_stride = kPageTokens;
    da.seq_len = m + off_sl;
    da.work = m + off_w;
    da.work_off = m + off_wo;
    da.n_work = n_work;
    da.split_len = split_len;
    da.order = m + off_ord;
    da.max_splits = max_splits;
    da.part_o = kv->part_o;
    da.part_ml = kv->part_ml;
    da.combine_count = c->dec_count;
    da.out = c->attn;
    da.gate = c->gate_act;  // null unless gated
    da.err = c->err_dev;
    if ((size_t)n_work > kv->part_items) return c->fail(OUTLETS_ECAPACITY, "split-KV partial buffer too small");
    if (c->bf16) {
      CUtensorMap km, vm;
      const uint64_t rows = (uint64_t)kv->num_pages * c->KVH * kPageTokens;
      if (!cached_map(c, &km, kv->k_pool, c->hd, rows, c->hd, 64) || !cached_map(c, &vm, kv->v_pool, c->hd, rows, c->hd, 64))
        return c->fail(OUTLETS_ECUDA, "cuTensorMapEncodeTiled failed for the KV pools");
      OUT_CK(c, attn_decode_bf16_launch(km, vm, da, s));
      c->stage_end(1);
    } else {
      OUT_CK(c, attn_decode_simt_launch<float>(da, s));
      c->stage_end(1);
    }
  }
  const OutDst od = out_dst(c, z_out, len_out);
  OUT_TRY(run_tail(c, B, B, nullptr, od.z, od.len, s, c->f));
  if (draft) OUT_TRY(run_draft(c, c->hn, B, *draft, s));
  c->last_rows = B;
  c->last_out_rows = B;
  c->last_tail_rows = B;
  c->last_kind = 2;
  c->last_slots.assign(slots, slots + B);
  return end_call(c, B, z_out, len_out, od, s);
}

}  // namespace

extern "C" {

outlets_status outlets_predict_prefill(outlets_ctx* c, const void* const taps[3], const int32_t* cu, int32_t B,
                                       int32_t T, outlets_kv* kv, const int32_t* slots, uint32_t flags,
                                       float* z_out, float* len_out, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  return predict_prefill(c, taps, nullptr, cu, B, T, kv, slots, flags, z_out, len_out, nullptr, stream);
}

outlets_status outlets_predict_prefill_dual(outlets_ctx* c, const void* const taps[3], const int32_t* cu,
                                            int32_t B, int32_t T, outlets_kv* kv, const int32_t* slots,
                                            uint32_t flags, float* z_out, float* len_out,
                                            const outlets_draft_out* draft, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  OUT_TRY(check_draft(c, draft));
  return predict_prefill(c, taps, nullptr, cu, B, T, kv, slots, flags, z_out, len_out, draft, stream);
}

outlets_status outlets_predict_prefill_ex(outlets_ctx* c, const void* const taps[3], const int32_t* tokens,
                                          const int32_t* cu, int32_t B, int32_t T, outlets_kv* kv,
                                          const int32_t* slots, uint32_t flags, float* z_out, float* len_out,
                                          const outlets_draft_out* draft, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  if (draft) OUT_TRY(check_draft(c, draft));
  return predict_prefill(c, taps, tokens, cu, B, T, kv, slots, flags, z_out, len_out, draft, stream);
}

outlets_status outlets_predict_step(outlets_ctx* c, const void* const taps[3], int32_t B, outlets_kv* kv,
                                    const int32_t* slots, float* z_out, float* len_out, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  return predict_step(c, taps, nullptr, B, kv, slots, z_out, len_out, nullptr, stream);
}

outlets_status outlets_predict_step_dual(outlets_ctx* c, const void* const taps[3], int32_t B, outlets_kv* kv,
                                         const int32_t* slots, float* z_out, float* len_out,
                                         const outlets_draft_out* draft, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  OUT_TRY(check_draft(c, draft));
  return predict_step(c, taps, nullptr, B, kv, slots, z_out, len_out, draft, stream);
}

outlets_status outlets_predict_step_ex(outlets_ctx* c, const void* const taps[3], const int32_t* tokens, int32_t B,
                                       outlets_kv* kv, const int32_t* slots, float* z_out, float* len_out,
                                       const outlets_draft_out* draft, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  if (draft) OUT_TRY(check_draft(c, draft));
  return predict_step(c, taps, tokens, B, kv, slots, z_out, len_out, draft, stream);
}

outlets_status outlets_predict_draft_step(outlets_ctx* c, const int32_t* tokens, int32_t B, outlets_kv* kv,
                                          const int32_t* slots, float* z_out, float* len_out,
                                          const outlets_draft_out* draft, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  if (draft) OUT_TRY(check_draft(c, draft));
  return predict_step(c, nullptr, tokens, B, kv, slots, z_out, len_out, draft, stream, true);
}

outlets_status outlets_draft_head(outlets_ctx* c, const void* h_draft, int32_t rows, const outlets_draft_out* draft,
                                  void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  OUT_TRY(check_draft(c, draft));
  if (rows < 0) return c->fail(OUTLETS_EINVAL, "rows must be >= 0");
  if (rows == 0) return OUTLETS_OK;
  if (!h_draft || !is_device_ptr(h_draft) || reinterpret_cast<uintptr_t>(h_draft) % 16)
    return c->fail(OUTLETS_EINVAL, "h_draft must be 16-byte aligned device memory");
  cudaStream_t s = (cudaStream_t)stream;
  OUT_TRY(begin_call(c, s));
  OUT_TRY(run_draft(c, h_draft, rows, *draft, s));
  OUT_CK(c, cudaEventRecord(c->done_ev, s));
  c->have_prev = true;
  return OUTLETS_OK;
}

outlets_status outlets_get_intermediate(outlets_ctx* c, int32_t which, void* dst, size_t dst_bytes,
                                        outlets_tensor_info* info, void* stream) {
  if (!c || !info) return OUTLETS_EINVAL;
  const int act = c->bf16 ? OUTLETS_BF16 : OUTLETS_F32;
  const void* src = nullptr;
  outlets_tensor_info ti{};
  switch (which) {
    case OUTLETS_T_FCTX: ti = {OUTLETS_F32, c->last_rows, c->d}; src = c->f; break;
    case OUTLETS_T_XIN: ti = {act, c->last_rows, c->d}; src = c->xhat; break;  // bf16: recomputed below
    case OUTLETS_T_Q: ti = {act, c->last_tail_rows, c->attn_w}; src = c->q; break;
    case OUTLETS_T_ATTN: ti = {act, c->last_tail_rows, c->attn_w}; src = c->attn; break;
    case OUTLETS_T_A: ti = {OUTLETS_F32, c->last_tail_rows, c->d}; src = c->a; break;
    case OUTLETS_T_Y: ti = {OUTLETS_F32, c->last_tail_rows, c->d}; src = c->y; break;
    case OUTLETS_T_HDRAFT: ti = {act, c->last_out_rows, c->d}; src = c->hn; break;
    default: return c->fail(OUTLETS_EINVAL, "unknown intermediate");
  }
  *info = ti;
  if (!dst) return OUTLETS_OK;
  const size_t bytes = (size_t)ti.rows * ti.cols * (ti.dtype == OUTLETS_BF16 ? 2 : 4);
  if (dst_bytes < bytes) return c->fail(OUTLETS_EINVAL, "dst too small");
  OUT_CK(c, cudaSetDevice(c->cfg.device));
  if (which == OUTLETS_T_XIN && c->fold) {
    // the bf16 path keeps g_in in the QKV weights and never materializes
    // x_hat = RMSNorm(f; g_in) itself: normalize f on request
    if (!c->xin_scratch) {
      c->xin_scratch = c->alloc((size_t)c->max_rows * c->d * c->esz);
      if (!c->xin_scratch) return c->fail(OUTLETS_ENOMEM, "x_hat scratch allocation failed");
    }
    OUT_CK(c, rmsnorm_launch<bf16>(c->f, c->g_in, (bf16*)c->xin_scratch, nullptr, c->last_rows, c->d,
                                   c->cfg.rms_eps, (cudaStream_t)stream));
    src = c->xin_scratch;
  }
  OUT_CK(c, cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDefault, (cudaStream_t)stream));
  return OUTLETS_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Length head without device allocation.
//
// Some callers cannot call cudaMalloc while they serve: a serving process that
// hands all spare device memory to its KV-cache pool at start-up and treats any
// later allocation as a failure, or a caller on a latency-critical path where
// cudaMalloc's implicit device-wide synchronization is not acceptable.  For
// them, outlets_length_head_noalloc runs the length head (Linear+ReLU layers
// and the output row) with its hidden activations in the file-scope array
// below instead of in memory it allocates.  The array is part of the library
// image.  Under lazy module loading its 16 MiB are committed on a device when
// the module holding it is first used there; outlets_create looks up the
// array's address, so the memory is reserved when the first context is
// created on that device and stays until the process exits.  All calls on a
// device share it, so calls that overlap on the GPU race; nothing in it has
// to start at zero (every value read was written earlier in the same call).
namespace {

constexpr size_t kHeadScratchFloats = (size_t)4 << 20;  // 16 MiB
static __device__ __align__(256) float g_head_scratch[kHeadScratchFloats];

std::mutex g_head_scratch_mu;
float* g_head_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once
// per device; host code must not use the symbol itself as an address).
cudaError_t head_scratch_ptr(int device, float** out) {
  std::lock_guard<std::mutex> lock(g_head_scratch_mu);
  if (!g_head_scratch_ptr[device]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_head_scratch);
    if (e != cudaSuccess) return e;
    g_head_scratch_ptr[device] = static_cast<float*>(p);
  }
  *out = g_head_scratch_ptr[device];
  return cudaSuccess;
}

}  // namespace

extern "C" outlets_status outlets_length_head_noalloc(outlets_ctx* c, const void* h_draft, int32_t rows,
                                                      float* z_out, float* len_out, void* stream) {
  if (!c) return OUTLETS_EINVAL;
  c->err.clear();
  if (!h_draft || !z_out) return c->fail(OUTLETS_EINVAL, "h_draft and z_out must not be NULL");
  if (rows < 0) return c->fail(OUTLETS_EINVAL, "rows must be >= 0");
  if (rows == 0) return OUTLETS_OK;
  if (c->cfg.device < 0 || c->cfg.device >= kMaxDevices) return c->fail(OUTLETS_EUNSUPPORTED, "device ordinal too large");
  if (!is_device_ptr(h_draft) || !is_device_ptr(z_out) || (len_out && !is_device_ptr(len_out)))
    return c->fail(OUTLETS_EINVAL, "h_draft, z_out and len_out must be device memory");
  if (reinterpret_cast<uintptr_t>(h_draft) % 16) return c->fail(OUTLETS_EINVAL, "h_draft must be 16-byte aligned");
  const int nl = (int)c->head_dims.size() - 1;
  int wmax = 1;
  for (int i = 1; i < nl; ++i) wmax = std::max(wmax, c->head_dims[i]);
  const size_t need = (size_t)rows * (nl > 2 ? 2 * (size_t)wmax : (size_t)c->head_dims[1]);
  if (need > kHeadScratchFloats)
    return c->fail(OUTLETS_ECAPACITY, "rows x head width exceeds the 16 MiB scratch of outlets_length_head_noalloc (" +
                                          std::to_string(need) + " > " + std::to_string(kHeadScratchFloats) +
                                          " floats)");
  OUT_CK(c, cudaSetDevice(c->cfg.device));
  return head_noalloc_run(c, h_draft, rows, z_out, len_out, (cudaStream_t)stream);
}

namespace {

// The head on rows of draft states with its hidden activations in the static
// scratch array (argument checks are the caller's).
outlets_status head_noalloc_run(outlets_ctx* c, const void* h_draft, int rows, float* z_out, float* len_out,
                                cudaStream_t s) {
  float* scratch = nullptr;
  OUT_CK(c, head_scratch_ptr(c->cfg.device, &scratch));
  const int nl = (int)c->head_dims.size() - 1;
  int wmax = 1;
  for (int i = 1; i < nl; ++i) wmax = std::max(wmax, c->head_dims[i]);
  const int d = c->d;
  float* buf[2] = {scratch, scratch + (size_t)rows * wmax};
  float* cur = buf[0];
  const void* a1[3] = {h_draft, h_draft, h_draft};
  const int w1 = c->head_dims[1];
  if (c->bf16)
    OUT_TRY(gemm_tc(c, a1, 1, d, d, rows, c->head_w0, c->np_h0, w1, d, EPI_BIAS_RELU, cur, w1, nullptr, 0, c->head_b[0], s));
  else
    OUT_TRY(gemm_f32(c, a1, d, rows, c->head_w0, w1, d, EPI_BIAS_RELU, cur, w1, nullptr, 0, c->head_b[0], s));
  for (int i = 1; i < nl - 1; ++i) {
    float* nxt = (cur == buf[0]) ? buf[1] : buf[0];
    const void* ai[3] = {cur, cur, cur};
    OUT_TRY(gemm_f32(c, ai, c->head_dims[i], rows, c->head_wf[i], c->head_dims[i + 1], c->head_dims[i],
                     EPI_BIAS_RELU, nxt, c->head_dims[i + 1], nullptr, 0, c->head_b[i], s));
    cur = nxt;
  }
  OUT_CK(c, head_tail_launch(cur, 1, 0, nullptr, c->head_wf[nl - 1], c->head_b[nl - 1], rows, c->head_dims[nl - 1],
                             z_out, len_out, s));
  return OUTLETS_OK;
}

}  // namespace
