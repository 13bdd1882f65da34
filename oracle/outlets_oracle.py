"""CPU oracle for the OUTLETS length-prediction forward.  TEST INFRASTRUCTURE ONLY.

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module.  The library never calls it, and it
shares no code with the CUDA path (it does not import the package).

Everything is float64 numpy; a matrix product (``@``) is the only library
primitive used as a step.  The steps follow the paper in order:

  Eq. 1 (Sec. 4.1)      f_ctx = W_proj · Concat(h^(2), h^(N/2), h^(N-2))
  Sec. 4.1 "Draft Decoder Layer": one Transformer decoder layer with
                        self-attention and MLP blocks, read as a pre-norm
                        Llama layer: RMSNorm -> RoPE causal GQA attention ->
                        residual -> RMSNorm -> SwiGLU MLP -> residual
  Sec. 4.2 "Length Regression Head": final RMSNorm gives h^draft_t;
                        z_hat_t = MLP_len(h^draft_t), Linear/ReLU/.../Linear;
                        z = log(1 + length), so length_hat = exp(z_hat) - 1
  Sec. 3.2 static prediction: r_0 read once after prefill, from the prompt's
                        last position; dynamic prediction: r_t at each decode
                        step t >= 1, the new token attending to the cached
                        draft keys/values of all earlier positions.

Readings where the paper is silent (the same list is kept in the design notes):
  * attention is standard causal GQA softmax(q k^T / sqrt(hd)) v; q-head h
    uses kv-head floor(h * KVH / H);
  * gated attention (Sec. 4.1 instantiates the layer's attention with the
    cited Gated Attention, no formula given): read as that work's elementwise,
    head-specific sigmoid gate computed from the normalized layer input,
    o <- o * sigmoid(x_hat W_ag^T) with W_ag [H*hd, d], applied to the
    attention output before W_o.  Used when the weights carry "w_attn_gate";
    the default path has no gate;
  * RMSNorm y = x * g / sqrt(mean(x^2) + eps);
  * RoPE rotates pairs (i, i + hd/2) by angle pos * theta^(-2i/hd);
    positions restart at 0 for each packed sequence; a decode step's token
    has position = number of tokens already cached for its request;
  * Linear layers of the decoder have no bias; the length head has biases;
  * static pooling takes the last prompt position;
  * length_hat = max(0, expm1(z_hat)) (clamped because expm1 < 0 for z < 0);
  * input-embedding branch of the EAGLE-3-style backbone (an ablated
    component in Sec. 5.4, no formula given): the layer input is
    Concat(RMSNorm(E[token]; g_emb), RMSNorm(f_ctx; g_in)), width 2d, so the
    QKV projections (and the attention gate) take 2d inputs; the residual
    stream stays f_ctx.  Used when the weights carry "w_embed" and the call
    gives one token id per row;
  * draft rollouts (EAGLE-3-style multi-token drafting, Sec. 2): a draft
    position after the first takes the draft layer's output state y (the
    residual stream before the final norm) of the previous position as its
    feature input in place of the fused taps, with the drafted token's
    embedding; its K/V are cached like any position (and dropped again when
    the target rejects it);
  * dual head (Sec. 4.2, Eq. 2): the draft branch reads the same final-normed
    state h^draft as the length head; its output is the log of the softmax of
    W_lm h^draft over the vocabulary, reported as the k most probable tokens
    (ties: smaller token id first), their log-probabilities and the row's
    logsumexp.  Used when the weights carry "w_lm" and draft_k is given.

Parity pins: every function here is checked by ``tests/test_oracle_pins.py``
against closed forms, special cases, brute force on tiny inputs, invariants and
a library routine (torch CPU scaled_dot_product_attention).  No value the
paper prints pins the forward numerically (it prints no worked example).
"""
from __future__ import annotations

import numpy as np

F64 = np.float64


def _f64(a):
    return np.asarray(a, dtype=F64)


# ------------------------------------------------------------------ Eq. 1
def fuse_taps(taps, w_proj):
    """f_ctx = W_proj · Concat(taps) for each token row (Eq. 1, Sec. 4.1).

    taps: three [T, d] arrays (low, mid, high tapped layers, in that order).
    w_proj: [d, 3d], nn.Linear convention (output row, input column).
    """
    cat = np.concatenate([_f64(t) for t in taps], axis=1)
    return cat @ _f64(w_proj).T


# ------------------------------------------------------------------ RMSNorm
def rms_norm(x, g, eps):
    """x * g / sqrt(mean(x^2) + eps) over the last axis (pre-norm layer reading)."""
    x = _f64(x)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * _f64(g)


# ------------------------------------------------------------------ RoPE
def rope_inv_freq(head_dim, theta):
    """theta^(-2i/hd) for i in [0, hd/2)."""
    i = np.arange(head_dim // 2, dtype=F64)
    return np.power(F64(theta), -2.0 * i / head_dim)


def apply_rope(x, pos, theta):
    """Rotate pairs (i, i + hd/2) of x [T, n_heads, hd] by pos[t] * inv_freq[i]."""
    x = _f64(x)
    half = x.shape[-1] // 2
    ang = _f64(pos)[:, None] * rope_inv_freq(x.shape[-1], theta)[None, :]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def positions_from_cu(cu):
    """Per-token position inside its packed sequence (restarts at 0)."""
    cu = np.asarray(cu, dtype=np.int64)
    pos = np.empty(int(cu[-1]), dtype=np.int64)
    for b in range(len(cu) - 1):
        pos[cu[b]:cu[b + 1]] = np.arange(cu[b + 1] - cu[b])
    return pos


# ------------------------------------------------------------------ attention
def _softmax_rows(s):
    m = np.max(s, axis=-1, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=-1, keepdims=True)


def kv_head_of(h, n_heads, n_kv_heads):
    """GQA: contiguous groups of H/KVH query heads share one kv head."""
    return (h * n_kv_heads) // n_heads


def causal_gqa_attention(q, k, v, cu):
    """Per packed sequence: o = softmax(q k^T / sqrt(hd) + causal mask) v.

    q: [T, H, hd]; k, v: [T, KVH, hd]; cu: [B+1] sequence offsets.
    Key j is visible to query i iff both are in the same sequence and j <= i.
    """
    q, k, v = _f64(q), _f64(k), _f64(v)
    T, H, hd = q.shape
    KVH = k.shape[1]
    out = np.zeros((T, H, hd), dtype=F64)
    scale = 1.0 / np.sqrt(hd)
    for b in range(len(cu) - 1):
        s0, s1 = int(cu[b]), int(cu[b + 1])
        if s1 == s0:
            continue
        L = s1 - s0
        mask = np.tril(np.ones((L, L), dtype=bool))
        for h in range(H):
            g = kv_head_of(h, H, KVH)
            s = (q[s0:s1, h] @ k[s0:s1, g].T) * scale
            s = np.where(mask, s, -np.inf)
            out[s0:s1, h] = _softmax_rows(s) @ v[s0:s1, g]
    return out


def attend_single(q_row, k_all, v_all):
    """One query token [H, hd] against all its keys [L, KVH, hd] (no mask needed:
    every cached key precedes or is the query itself)."""
    q_row, k_all, v_all = _f64(q_row), _f64(k_all), _f64(v_all)
    H, hd = q_row.shape
    KVH = k_all.shape[1]
    out = np.zeros((H, hd), dtype=F64)
    for h in range(H):
        g = kv_head_of(h, H, KVH)
        s = (k_all[:, g] @ q_row[h]) / np.sqrt(hd)
        out[h] = _softmax_rows(s[None, :])[0] @ v_all[:, g]
    return out


# ------------------------------------------------------------------ input embeddings (Sec. 5.4)
def layer_input(w, f, tokens, eps):
    """Normalized input of the draft decoder layer.

    Without the input-embedding branch: RMSNorm(f_ctx; g_in).  With it
    (weights carry "w_embed" [V, d] and "g_emb" [d]): the token's embedding
    row, normalized on its own, followed by the normalized fused feature:
    Concat(RMSNorm(E[token]; g_emb), RMSNorm(f_ctx; g_in)), width 2d.
    """
    x = rms_norm(f, w["g_in"], eps)
    if w.get("w_embed") is None:
        return x
    e = _f64(np.asarray(w["w_embed"])[np.asarray(tokens, dtype=np.int64)])  # row lookup, then widen
    return np.concatenate([rms_norm(e, w["g_emb"], eps), x], axis=1)


# ------------------------------------------------------------------ gated attention (Sec. 4.1)
def sigmoid(x):
    x = _f64(x)
    return 1.0 / (1.0 + np.exp(-x))


def attention_gate(x, w_attn_gate):
    """Elementwise gate of gated attention: sigmoid(x_hat W_ag^T), [rows, H*hd]."""
    return sigmoid(_f64(x) @ _f64(w_attn_gate).T)


# ------------------------------------------------------------------ MLP
def silu(x):
    x = _f64(x)
    return x / (1.0 + np.exp(-x))


def swiglu_mlp(x, w_gate, w_up, w_down):
    """down( silu(x W_gate^T) * (x W_up^T) )."""
    x = _f64(x)
    return (silu(x @ _f64(w_gate).T) * (x @ _f64(w_up).T)) @ _f64(w_down).T


# ------------------------------------------------------------------ head (Sec. 4.2)
def length_head(h, head_ws, head_bs):
    """MLP_len: Linear -> ReLU -> ... -> Linear to one scalar per row (z_hat)."""
    x = _f64(h)
    n = len(head_ws)
    for i in range(n):
        x = x @ _f64(head_ws[i]).T + _f64(head_bs[i])
        if i < n - 1:
            x = np.maximum(x, 0.0)
    return x[:, 0]


def z_to_length(z):
    """Invert z = log(1 + length): length_hat = max(0, exp(z) - 1)."""
    return np.maximum(0.0, np.expm1(_f64(z)))


def head_weights(w):
    ws, bs, i = [], [], 0
    while f"head_w{i}" in w:
        ws.append(w[f"head_w{i}"])
        bs.append(w[f"head_b{i}"])
        i += 1
    return ws, bs


# ------------------------------------------------------------------ draft head (Sec. 4.2, Eq. 2)
def draft_logits(h, w_lm):
    """W_lm h^draft for every row: the vector Eq. 2 passes to the softmax.
    w_lm: [V, d] (one row per vocabulary entry)."""
    return _f64(h) @ _f64(w_lm).T


def log_softmax_rows(logits):
    """log of the softmax of Eq. 2 over the vocabulary axis, and the logsumexp.

    logsumexp = m + log(sum_v exp(l_v - m)) with m the row maximum (the shift
    keeps every exponent <= 0); log P(v) = l_v - logsumexp.
    """
    l = _f64(logits)
    m = np.max(l, axis=-1, keepdims=True)
    lse = m + np.log(np.sum(np.exp(l - m), axis=-1, keepdims=True))
    return l - lse, lse[..., 0]


def top_k_tokens(values, k):
    """Indices of the k largest entries of each row, largest first; equal
    values are ordered by smaller index (a total order, so the answer is unique)."""
    values = _f64(values)
    ids = np.arange(values.shape[-1])
    out = np.empty((values.shape[0], k), dtype=np.int64)
    for r in range(values.shape[0]):
        out[r] = np.lexsort((ids, -values[r]))[:k]
    return out


def draft_head(h, w_lm, k):
    """Draft branch of the dual head: P_draft = softmax(W_lm h^draft) (Eq. 2),
    reported as the top-k tokens with their log-probabilities."""
    logits = draft_logits(h, w_lm)
    logp, lse = log_softmax_rows(logits)
    ids = top_k_tokens(logits, k)
    return dict(logits=logits, logprob=logp, lse=lse, topk_ids=ids,
                topk_logprob=np.take_along_axis(logp, ids, axis=1))


# ------------------------------------------------------------------ forward
def predict_prefill(w, shape, taps, cu, all_tokens=False, draft_k=None, tokens=None):
    """Static prediction over a packed varlen batch (Sec. 3.2, Sec. 4).

    Returns a dict with the hidden states of every step (for parity tests),
    the post-RoPE keys/values of every token (the draft KV cache), z_hat and
    length_hat at each sequence's last token (or every token if all_tokens).
    With draft_k and weights carrying "w_lm", "draft" holds the draft head's
    output (draft_head) on the same rows.  tokens: [T] token ids, required
    with the input-embedding branch (layer_input).
    """
    H, KVH, hd = shape.n_heads, shape.n_kv_heads, shape.head_dim
    eps, theta = shape.rms_eps, shape.rope_theta
    cu = np.asarray(cu, dtype=np.int64)
    T = int(cu[-1])
    pos = positions_from_cu(cu)

    f = fuse_taps(taps, w["w_proj"])                         # Eq. 1
    x = layer_input(w, f, tokens, eps)
    q = (x @ _f64(w["w_q"]).T).reshape(T, H, hd)
    k = (x @ _f64(w["w_k"]).T).reshape(T, KVH, hd)
    v = (x @ _f64(w["w_v"]).T).reshape(T, KVH, hd)
    q = apply_rope(q, pos, theta)
    k = apply_rope(k, pos, theta)
    o = causal_gqa_attention(q, k, v, cu).reshape(T, H * hd)
    if w.get("w_attn_gate") is not None:
        o = o * attention_gate(x, w["w_attn_gate"])
    a = f + o @ _f64(w["w_o"]).T
    ah = rms_norm(a, w["g_post"], eps)
    y = a + swiglu_mlp(ah, w["w_gate"], w["w_up"], w["w_down"])
    rows = np.arange(T) if all_tokens else cu[1:] - 1
    hd_state = rms_norm(y[rows], w["g_final"], eps)          # h^draft
    ws, bs = head_weights(w)
    z = length_head(hd_state, ws, bs)
    out = dict(f=f, x=x, q=q, k=k, v=v, attn=o, a=a, y=y, rows=rows,
               h_draft=hd_state, z=z, length=z_to_length(z))
    if draft_k:
        out["draft"] = draft_head(hd_state, w["w_lm"], draft_k)
    return out


def caches_from_prefill(out, cu):
    """Split the prefill's post-RoPE K/V into one cache per sequence."""
    cu = np.asarray(cu, dtype=np.int64)
    return [(out["k"][cu[b]:cu[b + 1]].copy(), out["v"][cu[b]:cu[b + 1]].copy())
            for b in range(len(cu) - 1)]


def predict_step(w, shape, taps_rows, caches, draft_k=None, tokens=None, f_rows=None):
    """Dynamic prediction for one new token per request (Sec. 3.2, t >= 1).

    taps_rows: three [B, d] arrays; caches: list of B (k [L, KVH, hd],
    v [L, KVH, hd]) already-cached post-RoPE keys/values.  The new token sits
    at position L of its request.  Returns z_hat, length_hat, intermediates and
    the caches extended by the new token (and "draft" as in predict_prefill).
    tokens: [B] ids of the new tokens (input-embedding branch).
    f_rows: [B, d] feature input in place of Eq. 1's fused taps: a draft
    rollout step (EAGLE-3-style multi-token drafting) feeds the draft layer's
    own output state y of the request's previous position back in.
    """
    H, KVH, hd = shape.n_heads, shape.n_kv_heads, shape.head_dim
    eps, theta = shape.rms_eps, shape.rope_theta
    B = len(caches)
    pos = np.array([c[0].shape[0] for c in caches], dtype=np.int64)

    f = fuse_taps(taps_rows, w["w_proj"]) if f_rows is None else _f64(f_rows)
    x = layer_input(w, f, tokens, eps)
    q = apply_rope((x @ _f64(w["w_q"]).T).reshape(B, H, hd), pos, theta)
    k = apply_rope((x @ _f64(w["w_k"]).T).reshape(B, KVH, hd), pos, theta)
    v = (x @ _f64(w["w_v"]).T).reshape(B, KVH, hd)
    new_caches, o = [], np.zeros((B, H, hd), dtype=F64)
    for b in range(B):
        kc = np.concatenate([_f64(caches[b][0]), k[b:b + 1]], axis=0)
        vc = np.concatenate([_f64(caches[b][1]), v[b:b + 1]], axis=0)
        o[b] = attend_single(q[b], kc, vc)
        new_caches.append((kc, vc))
    o = o.reshape(B, H * hd)
    if w.get("w_attn_gate") is not None:
        o = o * attention_gate(x, w["w_attn_gate"])
    a = f + o @ _f64(w["w_o"]).T
    y = a + swiglu_mlp(rms_norm(a, w["g_post"], eps), w["w_gate"], w["w_up"], w["w_down"])
    hd_state = rms_norm(y, w["g_final"], eps)
    ws, bs = head_weights(w)
    z = length_head(hd_state, ws, bs)
    out = dict(f=f, x=x, q=q, k=k, v=v, attn=o, a=a, y=y, h_draft=hd_state,
               z=z, length=z_to_length(z), caches=new_caches)
    if draft_k:
        out["draft"] = draft_head(hd_state, w["w_lm"], draft_k)
    return out


def sample_prefill_rows(w, shape, taps, cu, seqs, draft_k=None, tokens=None):
    """Oracle for a subset of sequences of a large packed batch.

    Every sequence is independent (attention never crosses sequences), so the
    prediction for sequence b only needs its own rows.  Used to check sampled
    outputs of full-size runs.
    """
    cu = np.asarray(cu, dtype=np.int64)
    sub_taps = [np.concatenate([t[cu[b]:cu[b + 1]] for b in seqs]) for t in taps]
    sub_tok = None if tokens is None else np.concatenate([np.asarray(tokens)[cu[b]:cu[b + 1]] for b in seqs])
    sub_len = np.array([cu[b + 1] - cu[b] for b in seqs], dtype=np.int64)
    sub_cu = np.zeros(len(seqs) + 1, dtype=np.int64)
    np.cumsum(sub_len, out=sub_cu[1:])
    return predict_prefill(w, shape, sub_taps, sub_cu, draft_k=draft_k, tokens=sub_tok)
