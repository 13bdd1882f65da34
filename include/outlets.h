/*
 * OUTLETS length prediction on one GB300 (sm_103a): the C ABI.
 *
 * The library computes the batched length-prediction forward of OUTLETS
 * ("Output-Length Prediction from Speculative Decoding Backbones"):
 *
 *   Eq. 1, Sec. 4.1    f_ctx = W_proj . Concat(h^(2), h^(floor(N/2)), h^(N-2))
 *   Sec. 4.1           one draft decoder layer (pre-norm: RMSNorm, RoPE causal
 *                      GQA self-attention, residual, RMSNorm, SwiGLU MLP, residual)
 *   Sec. 4.2           final RMSNorm -> h^draft; z_hat = MLP_len(h^draft)
 *                      (Linear/ReLU/.../Linear); z = log(1 + length), so the
 *                      returned length is max(0, exp(z_hat) - 1)
 *   Sec. 3.2           static prediction r_hat_0 after prefill (last prompt
 *                      position); dynamic prediction r_hat_t at decode step t,
 *                      one new token per request against the draft KV cache.
 *   Sec. 4.2, Eq. 2    dual head: the same h^draft also feeds the draft LM
 *                      head, P_draft = softmax(W_lm h^draft) over the
 *                      vocabulary (the *_dual calls and outlets_draft_head).
 *
 * The returned length is the REMAINING length r_hat_t (Sec. 3.1); a scheduler
 * forms the projected total t + r_hat_t itself.
 *
 * Conventions
 *  - Every entry point returns an outlets_status.  Argument errors are found
 *    on the host before anything is launched; the context's last-error string
 *    (outlets_last_error) then says what was wrong.  No C++ exception crosses
 *    the ABI.
 *  - Prediction calls are asynchronous on the caller's CUDA stream (a
 *    cudaStream_t passed as void*, NULL = legacy default stream).  Calls on
 *    one context are ordered: a call on a different stream waits for the
 *    previous call of the same context.
 *  - Tensors: "device or host" arguments may be device memory or host memory
 *    (pageable or pinned); the library detects which.  Host inputs are copied
 *    to the device inside the call; host outputs are written by an
 *    asynchronous copy, so synchronize the stream before reading them.
 *    Small index arrays (cu_seqlens, slots) are always host memory.
 *  - The library owns its device copy of the weights, its workspace and the
 *    KV pools; inputs and outputs stay owned by the caller and are only
 *    borrowed for the duration of the call's work on the stream.
 *  - Kernels never trap.  Bounded waits that run out, or indices a kernel
 *    refuses, set a device error word; outlets_check() synchronizes and
 *    reports it (OUTLETS_ETIMEOUT / OUTLETS_EDEVICE).
 */
#ifndef OUTLETS_H_
#define OUTLETS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum outlets_status {
  OUTLETS_OK = 0,
  OUTLETS_EINVAL = 1,        /* invalid argument; nothing was launched or changed */
  OUTLETS_ENOMEM = 2,        /* device or pinned-host allocation failed */
  OUTLETS_ECUDA = 3,         /* a CUDA runtime/driver call failed */
  OUTLETS_EUNSUPPORTED = 4,  /* shape or feature the library does not implement */
  OUTLETS_ECAPACITY = 5,     /* KV cache or workspace too small; nothing changed */
  OUTLETS_ETIMEOUT = 6,      /* a kernel's bounded wait ran out (from outlets_check) */
  OUTLETS_EDEVICE = 7        /* a kernel refused an index (from outlets_check) */
} outlets_status;

typedef enum outlets_dtype {
  OUTLETS_F32 = 0,   /* f32 weights/activations, CUDA-core kernels */
  OUTLETS_BF16 = 1   /* bf16 weights/activations, f32 accumulation, tensor cores */
} outlets_dtype;

#define OUTLETS_MAX_HEAD_HIDDEN 7

/* Shape of the draft backbone and of the length head, plus workspace limits. */
typedef struct outlets_config {
  int32_t d_model;        /* d: width of each tap, of f_ctx and of the draft state */
  int32_t n_heads;        /* H query heads */
  int32_t n_kv_heads;     /* KVH key/value heads; H % KVH == 0 */
  int32_t head_dim;       /* hd (multiple of 16; 64 or 128 on the bf16 path) */
  int32_t ffn_dim;        /* F: SwiGLU inner width */
  int32_t n_head_hidden;  /* hidden Linear+ReLU layers of MLP_len (1 .. OUTLETS_MAX_HEAD_HIDDEN) */
  int32_t head_hidden[OUTLETS_MAX_HEAD_HIDDEN];  /* their widths; the last Linear maps to 1 */
  float rope_theta;       /* RoPE base */
  float rms_eps;          /* RMSNorm epsilon */
  int32_t dtype;          /* outlets_dtype */
  int32_t max_tokens;     /* most packed rows in one prefill call */
  int32_t max_batch;      /* most sequences per prefill call / requests per step call */
  int32_t max_position;   /* positions 0 .. max_position-1 are supported (RoPE table) */
  int32_t device;         /* CUDA device ordinal */
  int32_t vocab;          /* V: rows of the draft LM head W_lm (Eq. 2), 8 .. 262144;
                             0 = no draft head (the *_dual calls and
                             outlets_draft_head then return OUTLETS_EUNSUPPORTED) */
  int32_t embed_vocab;    /* rows of the token-embedding table of the input-embedding
                             branch (EAGLE-3-style layer input, Sec. 5.4); 0 = no
                             branch.  With the branch every prediction needs token
                             ids (the *_ex calls). */
} outlets_config;

/* Host pointers to f32 weights, nn.Linear layout [out, in], row-major.
 * On the bf16 path every value is rounded to bf16 (nearest even) on upload.
 *   w_proj [d, 3d]           the FC of Eq. 1 (taps concatenated low, mid, high)
 *   w_q [H*hd, d], w_k [KVH*hd, d], w_v [KVH*hd, d], w_o [d, H*hd]
 *   g_in, g_post, g_final [d] RMSNorm gains (input, post-attention, final)
 *   w_gate [F, d], w_up [F, d], w_down [d, F]
 *   head_w[i] [w_{i+1}, w_i], head_b[i] [w_{i+1}] for i = 0 .. n_head_hidden,
 *   widths w_0 = d, w_1.. = head_hidden, last = 1.
 *   w_attn_gate [H*hd, d] or NULL: gated attention (Sec. 4.1 uses the cited
 *     Gated Attention for the draft layer).  When given, the attention output
 *     o [rows, H*hd] is multiplied elementwise by sigmoid(x_hat w_attn_gate^T)
 *     (x_hat: the RMS-normalized layer input that also feeds QKV) before W_o;
 *     NULL gives standard attention.
 *   w_lm [V, d]              the draft LM head of Eq. 2 (required when vocab > 0,
 *     ignored otherwise).
 *   w_embed [embed_vocab, d], g_emb [d]: the input-embedding branch (required
 *     when embed_vocab > 0).  The layer input is then
 *     Concat(RMSNorm(w_embed[token]; g_emb), RMSNorm(f_ctx; g_in)), width 2d:
 *     w_q, w_k, w_v (and w_attn_gate) are [out, 2d], their columns 0 .. d-1
 *     read the normalized embedding and d .. 2d-1 the normalized fused
 *     feature.  The residual stream stays f_ctx.
 * The library copies everything during outlets_create; the caller may free
 * its arrays afterwards. */
typedef struct outlets_weights {
  const float* w_proj;
  const float* w_q;
  const float* w_k;
  const float* w_v;
  const float* w_o;
  const float* g_in;
  const float* g_post;
  const float* g_final;
  const float* w_gate;
  const float* w_up;
  const float* w_down;
  const float* head_w[OUTLETS_MAX_HEAD_HIDDEN + 1];
  const float* head_b[OUTLETS_MAX_HEAD_HIDDEN + 1];
  const float* w_attn_gate;
  const float* w_lm;
  const float* w_embed;
  const float* g_emb;
} outlets_weights;

typedef struct outlets_ctx outlets_ctx;
typedef struct outlets_kv outlets_kv;

/* Validates cfg, uploads the weights (re-laid out for the kernels), builds the
 * RoPE table in fp64 on the host and allocates the workspace for max_tokens
 * rows.  Synchronous.  On failure *out is NULL and no memory is held. */
outlets_status outlets_create(const outlets_config* cfg, const outlets_weights* w, outlets_ctx** out);

/* Frees everything the context owns (after synchronizing its device). */
void outlets_destroy(outlets_ctx* ctx);

/* Details of the last failed call on ctx ("" if none); valid until the next call. */
const char* outlets_last_error(const outlets_ctx* ctx);

/* Number of bytes the context holds on the device (weights + workspace). */
size_t outlets_device_bytes(const outlets_ctx* ctx);

/* Draft KV cache: post-RoPE keys and values of every cached position, bf16 or
 * f32 like the context, in pages of 64 positions; pools [pages][KVH][64][hd].
 * Slots 0 .. max_slots-1 each hold one request; max_tokens_total bounds the
 * positions cached over all slots together.  Needed by the dynamic prediction
 * of Sec. 3.2. */
outlets_status outlets_kv_create(outlets_ctx* ctx, int32_t max_slots, int32_t max_tokens_total,
                                 outlets_kv** out);
void outlets_kv_destroy(outlets_kv* kv);
/* Empties one slot (host bookkeeping only; ordered after earlier calls). */
outlets_status outlets_kv_reset_slot(outlets_kv* kv, int32_t slot);
/* Cached positions of a slot, or -1 for an invalid slot. */
int32_t outlets_kv_slot_length(const outlets_kv* kv, int32_t slot);
/* Pages not held by any slot. */
int32_t outlets_kv_free_pages(const outlets_kv* kv);

#define OUTLETS_ALL_TOKENS 1u /* prefill flag: predict at every packed row, not only each sequence's last */
/* Prefill flag: run the whole draft layer on every packed row even when only
 * each sequence's last row is predicted.  Without it (bf16 contexts, T > 256)
 * only the keys and values are projected for every row.  These feed the last
 * rows' attention and the KV cache.  Queries, attention, O, the MLP, the
 * final norm and the head run on the B predicted rows only.  The outputs are
 * the same either way.  The flag keeps every row's q / attention / a / y for
 * outlets_get_intermediate. */
#define OUTLETS_KEEP_ROWS 2u

/* Static prediction over a packed varlen batch (Sec. 3.2, t = 0).
 *   taps[3]     device or host, [T, d] each (bf16 or f32 like the context),
 *               row-major, 16-byte aligned: hidden states of target layers
 *               2, floor(N/2), N-2 for every prompt token (Eq. 1).
 *   cu_seqlens  host int32 [B+1]: cu[0] = 0, strictly increasing, cu[B] = T.
 *   kv, slots   optional (both or neither): slots is host int32 [B], distinct;
 *               each slot is reset and then holds its sequence's post-RoPE
 *               keys/values, ready for outlets_predict_step.
 *   flags       0, or OUTLETS_ALL_TOKENS and / or OUTLETS_KEEP_ROWS.
 *   z_out, len_out  device or host f32 [B] (or [T] with OUTLETS_ALL_TOKENS):
 *               z_hat and max(0, expm1(z_hat)) = predicted remaining length.
 *               len_out may be NULL.
 * Errors: EINVAL (shapes, pointers, cu_seqlens), ECAPACITY (T > max_tokens,
 * B > max_batch, a position >= max_position, or too few free KV pages). */
outlets_status outlets_predict_prefill(outlets_ctx* ctx, const void* const taps[3], const int32_t* cu_seqlens,
                                       int32_t B, int32_t T, outlets_kv* kv, const int32_t* slots, uint32_t flags,
                                       float* z_out, float* len_out, void* stream);

/* Dynamic prediction for one new token per request (Sec. 3.2, t >= 1).
 *   taps[3]   device or host [B, d] each: the new token's tapped hidden states.
 *   slots     host int32 [B], distinct.  The new token takes position
 *             L = outlets_kv_slot_length(slot), attends to the slot's L cached
 *             positions and itself, and is appended (slot length L + 1).
 *   z_out, len_out  device or host f32 [B].
 * Errors: EINVAL, ECAPACITY (no free page / position >= max_position / B >
 * max_batch); on error no slot changes. */
outlets_status outlets_predict_step(outlets_ctx* ctx, const void* const taps[3], int32_t B, outlets_kv* kv,
                                    const int32_t* slots, float* z_out, float* len_out, void* stream);

/* ---- Dual head: the draft LM head (Sec. 4.2, Eq. 2).
 * P_draft(v) = softmax(W_lm h^draft)_v over the V vocabulary entries, for
 * every predicted row (the rows whose z_hat a prediction call returns).  The
 * library reports the k most probable tokens of each row, most probable first
 * (equal logits: smaller token id first), their log-probabilities
 * log P_draft(v) = l_v - logsumexp_v'(l_v'), l = W_lm h^draft, and optionally
 * the logsumexp and the logits themselves.  The [rows, V] logits are never
 * materialized unless `logits` is given: the tensor-core GEMM reduces each
 * tile of logits to its softmax statistics and best tokens on chip.
 * Arithmetic: bf16 operands (h^draft as the length head reads it, W_lm
 * rounded on upload), f32 accumulation and softmax statistics. */
#define OUTLETS_MAX_TOPK 8

typedef struct outlets_draft_out {
  int32_t k;              /* tokens per row, 1 .. OUTLETS_MAX_TOPK and <= vocab */
  int32_t* topk_ids;      /* device or host int32 [rows, k]: token ids */
  float* topk_logprob;    /* device or host f32 [rows, k]: their log P_draft */
  float* logsumexp;       /* device or host f32 [rows], or NULL */
  float* logits;          /* device or host f32 [rows, vocab] (W_lm h^draft), or NULL */
} outlets_draft_out;

/* outlets_predict_prefill plus the draft head on the same rows (one pass of
 * the backbone serves both heads).  draft must not be NULL.  Extra errors:
 * EUNSUPPORTED (vocab == 0), EINVAL (bad k or NULL topk pointers). */
outlets_status outlets_predict_prefill_dual(outlets_ctx* ctx, const void* const taps[3], const int32_t* cu_seqlens,
                                            int32_t B, int32_t T, outlets_kv* kv, const int32_t* slots,
                                            uint32_t flags, float* z_out, float* len_out,
                                            const outlets_draft_out* draft, void* stream);

/* outlets_predict_step plus the draft head on the same rows. */
outlets_status outlets_predict_step_dual(outlets_ctx* ctx, const void* const taps[3], int32_t B, outlets_kv* kv,
                                         const int32_t* slots, float* z_out, float* len_out,
                                         const outlets_draft_out* draft, void* stream);

/* ---- Input-embedding branch (contexts with embed_vocab > 0).
 * The same calls with one token id per row: tokens is device or host int32,
 * [T] for prefill (every packed prompt token) and [B] for a step (each
 * request's new token), ids in 0 .. embed_vocab-1 (host ids are checked on
 * the host, EINVAL; device ids a kernel refuses set the device error word,
 * OUTLETS_EDEVICE from outlets_check).  draft may be NULL (length head only)
 * or request the draft head as in the *_dual calls.  Contexts without the
 * branch take tokens == NULL; contexts with it reject the calls without
 * tokens (EINVAL). */
outlets_status outlets_predict_prefill_ex(outlets_ctx* ctx, const void* const taps[3], const int32_t* tokens,
                                          const int32_t* cu_seqlens, int32_t B, int32_t T, outlets_kv* kv,
                                          const int32_t* slots, uint32_t flags, float* z_out, float* len_out,
                                          const outlets_draft_out* draft, void* stream);

outlets_status outlets_predict_step_ex(outlets_ctx* ctx, const void* const taps[3], const int32_t* tokens, int32_t B,
                                       outlets_kv* kv, const int32_t* slots, float* z_out, float* len_out,
                                       const outlets_draft_out* draft, void* stream);

/* ---- Draft rollouts (EAGLE-3-style multi-token drafting).
 * One more draft position per request: the feature input is the draft
 * layer's own output state y (the residual stream before the final norm) of
 * the request's previous position, in place of Eq. 1's fused taps, so no
 * target hidden states are needed.  It must follow a step (tapped or draft)
 * of this context over the same slots in the same order (EINVAL otherwise);
 * each request's position is its slot length, which grows by one.  tokens:
 * device or host int32 [B], the drafted tokens (e.g. the previous call's
 * top-1 draft ids, left on the device), required iff the context has the
 * input-embedding branch.  draft: optional, as in the *_dual calls.
 * The outputs are the length prediction at the draft position. */
outlets_status outlets_predict_draft_step(outlets_ctx* ctx, const int32_t* tokens, int32_t B, outlets_kv* kv,
                                          const int32_t* slots, float* z_out, float* len_out,
                                          const outlets_draft_out* draft, void* stream);

/* Keeps the first `length` cached positions of a slot (0 <= length <= its
 * length), e.g. to drop draft positions the target rejected.  Host
 * bookkeeping only, ordered after earlier calls like outlets_kv_reset_slot. */
outlets_status outlets_kv_truncate(outlets_kv* kv, int32_t slot, int32_t length);

/* The draft head alone on caller-given states.
 *   h_draft  device [rows, d] (bf16 or f32 like the context), 16-byte aligned.
 *   draft    outputs as above, rows rows. */
outlets_status outlets_draft_head(outlets_ctx* ctx, const void* h_draft, int32_t rows, const outlets_draft_out* draft,
                                  void* stream);

/* Synchronizes the stream, then reports (and clears) the device error word. */
outlets_status outlets_check(outlets_ctx* ctx, void* stream);

/* Intermediates of the last prediction call, for parity testing.  Rows: every
 * row of the call.  After a prefill that predicts only the last rows without
 * OUTLETS_KEEP_ROWS, q, attention, a and y hold the B predicted rows instead.
 * They are in sequence order, and the info's rows says which. */
typedef enum outlets_tensor {
  OUTLETS_T_FCTX = 0,   /* f_ctx [rows, d] f32 (Eq. 1) */
  OUTLETS_T_XIN = 1,    /* input-normed x [rows, d] act */
  OUTLETS_T_Q = 2,      /* post-RoPE q [rows, H, hd] act */
  OUTLETS_T_ATTN = 3,   /* attention output [rows, H*hd] act */
  OUTLETS_T_A = 4,      /* after attention residual [rows, d] f32 */
  OUTLETS_T_Y = 5,      /* layer output [rows, d] f32 */
  OUTLETS_T_HDRAFT = 6  /* final-normed draft state h^draft [out_rows, d] act */
} outlets_tensor;

typedef struct outlets_tensor_info {
  int32_t dtype;  /* outlets_dtype of the stored values */
  int32_t rows;
  int32_t cols;
} outlets_tensor_info;

/* Describes intermediate `which` of the last call in *info and, if dst is not
 * NULL, copies it (rows * cols elements, row-major) to dst (device or host,
 * dst_bytes large enough) on the stream. */
outlets_status outlets_get_intermediate(outlets_ctx* ctx, int32_t which, void* dst, size_t dst_bytes,
                                        outlets_tensor_info* info, void* stream);

/* Per-stage device timing.  While enabled, every prediction call records a
 * CUDA event pair around each selected stage on the call's stream (a stage is
 * one kernel, or the two kernels of split-KV decode attention).  An event pair
 * serializes its stage with its neighbours (no launch overlap across it), so
 * time only the stages you need inside a measured region. */
typedef enum outlets_stage {
  OUTLETS_S_FC = 0,          /* Eq. 1 tap-fusion GEMM */
  OUTLETS_S_NORM_IN = 1,     /* input RMSNorm */
  OUTLETS_S_QKV = 2,         /* QKV projection GEMM */
  OUTLETS_S_ROPE = 3,        /* RoPE + q / K / V scatter (cache append) */
  OUTLETS_S_ATTN = 4,        /* varlen causal attention or decode attention */
  OUTLETS_S_O = 5,           /* O projection GEMM + residual */
  OUTLETS_S_NORM_POST = 6,   /* post-attention RMSNorm */
  OUTLETS_S_GATEUP = 7,      /* gate/up GEMM with SwiGLU */
  OUTLETS_S_DOWN = 8,        /* down projection GEMM + residual */
  OUTLETS_S_FINAL_NORM = 9,  /* final RMSNorm of the predicted rows (h^draft) */
  OUTLETS_S_HEAD = 10,       /* length head (Sec. 4.2): Linear+ReLU layers and output row */
  OUTLETS_S_DRAFT = 11,      /* draft LM head (Eq. 2): GEMM with on-chip softmax/top-k, merge */
  OUTLETS_N_STAGES = 12
} outlets_stage;

/* Times the stages whose bit (1 << outlets_stage) is set in stage_mask for
 * later calls (-1: all, 0: off); clears recorded times. */
outlets_status outlets_profile_enable(outlets_ctx* ctx, int32_t stage_mask);

/* Waits for the recorded events, then writes for each stage the summed
 * duration in milliseconds (ms[OUTLETS_N_STAGES]) and how many times it ran
 * (count[OUTLETS_N_STAGES], may be NULL), and clears the records. */
outlets_status outlets_profile_read(outlets_ctx* ctx, double* ms, int32_t* count);

/* Static name of a stage ("fc_gemm", ...), or "" for an invalid id. */
const char* outlets_stage_name(int32_t stage);

/* Failure-path self-test (the paper has no counterpart).  Enqueues one kernel
 * whose bounded wait on an mbarrier can never complete -- the wait every
 * prediction pipeline uses -- so it gives up after timeout_ns (1 us .. 1 s)
 * and raises the context's device error word, as a stalled pipeline would.
 * The next outlets_check then returns OUTLETS_ETIMEOUT (and clears the word);
 * the context stays usable.  Faults nothing, hangs nothing. */
outlets_status outlets_selftest_bounded_wait(outlets_ctx* ctx, uint64_t timeout_ns, void* stream);

/* Number of kernels this context has launched for prediction calls so far. */
uint64_t outlets_launch_count(const outlets_ctx* ctx);

/* Length head without device allocation.  The paper has no counterpart: this
 * exists for callers that cannot call cudaMalloc while they serve (a process
 * that gives all spare device memory to its KV-cache pool at start-up and
 * treats later allocations as failures, or a latency-critical caller that
 * cannot accept cudaMalloc's implicit device synchronization).
 *   h_draft  device [rows, d] (bf16 or f32 like the context), 16-byte aligned:
 *            final-normed draft states (OUTLETS_T_HDRAFT of a prediction call).
 *   z_out, len_out  device f32 [rows]: z_hat and max(0, expm1(z_hat));
 *            len_out may be NULL.
 * The same length head as the prediction calls, agreeing with their z_hat
 * within the bf16 / f32 tolerances (the prediction calls may split the first
 * layer's sum over K for small batches, so the rounding order can differ).
 * The hidden activations live in a 16 MiB array inside the library image
 * instead of allocated memory; the array is reserved on a device when
 * outlets_create makes a context there (it looks up the array's address) and
 * stays until the process exits.  rows x (widest hidden layer) x (2 if the
 * head has more than one hidden layer) must fit in 4 Mi floats, else
 * OUTLETS_ECAPACITY with a message in outlets_last_error.  All calls on a
 * device share the array: calls that overlap on the GPU race.  Allocates
 * nothing (no cudaMalloc, cudaFree or allocating library routine). */
outlets_status outlets_length_head_noalloc(outlets_ctx* ctx, const void* h_draft, int32_t rows, float* z_out,
                                           float* len_out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* OUTLETS_H_ */
