"""Seeded synthetic inputs for the OUTLETS length-prediction forward.

This module only draws random numbers and packs them; it holds none of the
method's arithmetic.  Both the CUDA path and the CPU oracle are fed from here.

Shapes follow the draft backbones the method is evaluated with (Sec. 5.1,
"Models": Llama-3.1-8B and larger targets) and the tap definition of Eq. 1
(three hidden states of width d from layers {2, floor(N/2), N-2}).

Recipe (all draws from numpy PCG64 streams spawned from one SeedSequence):
  * stream 0 -> sequence / cache lengths;  stream 1 -> taps;  stream 2 -> weights;
    stream 3 -> draft LM head W_lm (Eq. 2) and stand-in draft states;
    stream 4 -> input-embedding branch (embedding table, its QKV columns, token ids);
    stream 5 -> serving workloads (arrivals, prompt and output lengths, prediction noise).
  * lengths: rint(lognormal(ln(median), sigma=1)) clipped to the stated range.
  * taps ~ N(0, 1); every Linear weight ~ N(0, 0.02); RMSNorm gains = 1;
    head hidden biases ~ N(0, 0.02); output bias = ln(1 + 256).
  * on the bf16 path every tap and weight is rounded to bf16 (round to nearest
    even) before either side sees it, so both compute on identical values.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

__all__ = [
    "ModelShape", "TINY", "LLAMA8B", "LLAMA70B", "SHAPES",
    "round_bf16", "bf16_bits", "tap_layer_indices",
    "lengths_tiny", "lengths_8b_prefill", "lengths_8b_step_cache",
    "lengths_70b_prefill", "lengths_sweep", "cu_seqlens",
    "make_weights", "make_taps", "weight_names",
    "LLAMA3_VOCAB", "make_lm_head", "make_draft_states", "make_tokens", "make_serving_requests",
]


@dataclasses.dataclass(frozen=True)
class ModelShape:
    """Draft-backbone shape (one decoder layer + length head)."""

    name: str
    d: int              # draft / target hidden width
    n_heads: int        # query heads H
    n_kv_heads: int     # key/value heads KVH (GQA)
    head_dim: int       # hd
    ffn: int            # SwiGLU inner width F
    head_widths: tuple  # hidden widths of the length MLP (output width 1 implied)
    rope_theta: float
    rms_eps: float
    dtype: str          # "f32" or "bf16"

    @property
    def qkv_out(self) -> int:
        return (self.n_heads + 2 * self.n_kv_heads) * self.head_dim


TINY = ModelShape("tiny-f32", 256, 4, 2, 64, 688, (128,), 10000.0, 1e-5, "f32")
LLAMA8B = ModelShape("llama3.1-8b-eagle3", 4096, 32, 8, 128, 14336, (1024,), 500000.0, 1e-5, "bf16")
LLAMA70B = ModelShape("llama3.3-70b-eagle3", 8192, 64, 8, 128, 28672, (1024,), 500000.0, 1e-5, "bf16")
SHAPES = {s.name: s for s in (TINY, LLAMA8B, LLAMA70B)}


def tap_layer_indices(n_layers: int) -> tuple:
    """Target layers whose hidden states are tapped: {2, floor(N/2), N-2} (Sec. 4.1)."""
    return (2, n_layers // 2, n_layers - 2)


# ----------------------------------------------------------------------------- bf16
def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even); returns float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) & np.uint32(0xFFFF0000)
    return r.view(np.float32)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of float32 values that are already bf16-representable."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    return (x.view(np.uint32) >> np.uint32(16)).astype(np.uint16)


def _streams(seed: int):
    return [np.random.Generator(np.random.PCG64(s)) for s in np.random.SeedSequence(seed).spawn(3)]


def _lognormal_lengths(rng, n, median, lo, hi):
    x = rng.lognormal(mean=math.log(median), sigma=1.0, size=n)
    return np.clip(np.rint(x), lo, hi).astype(np.int64)


# -------------------------------------------------------------------------- lengths
def lengths_tiny() -> np.ndarray:
    return np.array([16, 32, 48, 64], dtype=np.int64)


def lengths_8b_prefill(seed: int = 0, n: int = 64) -> np.ndarray:
    """64 ragged prompts, lognormal median 256, clipped to [16, 2048]."""
    return _lognormal_lengths(_streams(seed)[0], n, 256, 16, 2048)


def lengths_8b_step_cache(seed: int = 0, n: int = 256) -> np.ndarray:
    """Existing draft-cache lengths of 256 live requests: lognormal median 512, [1, 4096]."""
    return _lognormal_lengths(_streams(seed)[0], n, 512, 1, 4096)


def lengths_70b_prefill(seed: int = 0, n: int = 32) -> np.ndarray:
    """32 ragged prompts, lognormal median 1024, clipped to [64, 4096]."""
    return _lognormal_lengths(_streams(seed)[0], n, 1024, 64, 4096)


def lengths_sweep(seed: int = 0, n: int = 1024) -> np.ndarray:
    """Heavy-tailed mixture: 70% lognormal median 128, 30% median 2048, in [1, 8192]."""
    rng = _streams(seed)[0]
    pick_long = rng.random(n) < 0.3
    short = rng.lognormal(math.log(128), 1.0, n)
    long = rng.lognormal(math.log(2048), 1.0, n)
    x = np.where(pick_long, long, short)
    return np.clip(np.rint(x), 1, 8192).astype(np.int64)


def cu_seqlens(lengths) -> np.ndarray:
    """Packed-varlen offsets: cu[0] = 0, cu[b+1] = cu[b] + len[b] (int32)."""
    lengths = np.asarray(lengths, dtype=np.int64)
    cu = np.zeros(len(lengths) + 1, dtype=np.int64)
    np.cumsum(lengths, out=cu[1:])
    return cu.astype(np.int32)


# -------------------------------------------------------------------------- tensors
def weight_names(shape: ModelShape):
    n_head = len(shape.head_widths) + 1
    names = ["w_proj", "w_q", "w_k", "w_v", "w_o", "g_in", "g_post", "g_final",
             "w_gate", "w_up", "w_down"]
    for i in range(n_head):
        names += [f"head_w{i}", f"head_b{i}"]
    return names


def make_weights(shape: ModelShape, seed: int = 0, std: float = 0.02,
                 out_bias: float = math.log(257.0), gated: bool = False, embed_vocab: int = 0) -> dict:
    """All draft weights, nn.Linear [out, in] row-major, float32 arrays.

    On the bf16 path the matrices and head parameters are bf16-representable.
    gated=True adds the attention gate "w_attn_gate" [H*hd, d] (gated
    attention), drawn after every other weight so the rest are unchanged.
    embed_vocab > 0 adds the input-embedding branch: the embedding table
    "w_embed" [embed_vocab, d] ~ N(0, std), its RMSNorm gain "g_emb" = 1, and
    d input columns in front of w_q, w_k, w_v (and w_attn_gate) for the
    normalized embedding, all from stream 4, so the columns that read the
    fused feature are the weights drawn without the branch.
    """
    rng = _streams(seed)[2]
    d, H, KVH, hd, F = shape.d, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn
    rnd = round_bf16 if shape.dtype == "bf16" else (lambda a: np.ascontiguousarray(a, np.float32))

    def lin(o, i):
        return rnd(rng.standard_normal((o, i), dtype=np.float32) * np.float32(std))

    w = {}
    w["w_proj"] = lin(d, 3 * d)
    w["w_q"] = lin(H * hd, d)
    w["w_k"] = lin(KVH * hd, d)
    w["w_v"] = lin(KVH * hd, d)
    w["w_o"] = lin(d, H * hd)
    w["g_in"] = np.ones(d, np.float32)
    w["g_post"] = np.ones(d, np.float32)
    w["g_final"] = np.ones(d, np.float32)
    w["w_gate"] = lin(F, d)
    w["w_up"] = lin(F, d)
    w["w_down"] = lin(d, F)
    widths = (d,) + tuple(shape.head_widths) + (1,)
    for i in range(len(widths) - 1):
        w[f"head_w{i}"] = lin(widths[i + 1], widths[i])
        if i < len(widths) - 2:
            w[f"head_b{i}"] = rnd(rng.standard_normal(widths[i + 1], dtype=np.float32) * np.float32(std))
        else:
            w[f"head_b{i}"] = rnd(np.full(1, out_bias, np.float32))
    if gated:
        w["w_attn_gate"] = lin(H * hd, d)
    if embed_vocab:
        erng = np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed).spawn(5)[4]))

        def elin(o, i):
            return rnd(erng.standard_normal((o, i), dtype=np.float32) * np.float32(std))

        w["g_emb"] = np.ones(d, np.float32)
        for name in ("w_q", "w_k", "w_v") + (("w_attn_gate",) if gated else ()):
            w[name] = np.ascontiguousarray(np.concatenate([elin(w[name].shape[0], d), w[name]], axis=1))
        table = np.empty((embed_vocab, d), np.float32)
        step = max(1, (1 << 24) // d)
        for r0 in range(0, embed_vocab, step):
            r1 = min(embed_vocab, r0 + step)
            table[r0:r1] = elin(r1 - r0, d)
        w["w_embed"] = table
    return w


def make_tokens(n: int, vocab: int, seed: int = 0, stream_offset: int = 0) -> np.ndarray:
    """Token ids [n] uniform in [0, vocab) (int32), for the input-embedding branch."""
    ss = np.random.SeedSequence(seed).spawn(5)[4]
    ss = np.random.SeedSequence(entropy=ss.entropy, spawn_key=ss.spawn_key + (2000 + stream_offset,))
    return np.random.Generator(np.random.PCG64(ss)).integers(0, vocab, size=n, dtype=np.int64).astype(np.int32)


LLAMA3_VOCAB = 128256  # vocabulary of the Llama-3 targets (the draft head's output width)


def make_lm_head(shape: ModelShape, vocab: int, seed: int = 0, std: float = 0.02) -> np.ndarray:
    """Draft LM head W_lm [vocab, d] ~ N(0, std) (Eq. 2), from its own stream
    (stream 3), so drawing it leaves every other weight unchanged."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed).spawn(4)[3]))
    rnd = round_bf16 if shape.dtype == "bf16" else (lambda a: np.ascontiguousarray(a, np.float32))
    out = np.empty((vocab, shape.d), np.float32)
    step = max(1, (1 << 24) // shape.d)
    for r0 in range(0, vocab, step):  # bounded temporaries at vocab ~128k
        r1 = min(vocab, r0 + step)
        out[r0:r1] = rnd(rng.standard_normal((r1 - r0, shape.d), dtype=np.float32) * np.float32(std))
    return out


def make_draft_states(shape: ModelShape, rows: int, seed: int = 0, stream_offset: int = 0) -> np.ndarray:
    """Stand-in final-normed draft states h^draft [rows, d] for testing the
    draft head on its own: N(0, 1) entries (unit RMS, like an RMSNorm output
    with unit gains), bf16-rounded on the bf16 path."""
    ss = np.random.SeedSequence(seed).spawn(4)[3]
    ss = np.random.SeedSequence(entropy=ss.entropy, spawn_key=ss.spawn_key + (1000 + stream_offset,))
    rng = np.random.Generator(np.random.PCG64(ss))
    rnd = round_bf16 if shape.dtype == "bf16" else (lambda a: a)
    return rnd(rng.standard_normal((rows, shape.d), dtype=np.float32))


def make_taps(shape: ModelShape, n_tokens: int, seed: int = 0, stream_offset: int = 0):
    """Three tapped hidden states [T, d] ~ N(0, 1) (the h^(i) of Eq. 1)."""
    ss = np.random.SeedSequence(seed).spawn(3)[1]
    if stream_offset:
        ss = np.random.SeedSequence(entropy=ss.entropy, spawn_key=ss.spawn_key + (stream_offset,))
    rng = np.random.Generator(np.random.PCG64(ss))
    rnd = round_bf16 if shape.dtype == "bf16" else (lambda a: a)
    return [rnd(rng.standard_normal((n_tokens, shape.d), dtype=np.float32)) for _ in range(3)]


def make_serving_requests(n: int, qps: float, seed: int = 0, pred_sigma: float = 0.5,
                          prompt_median: float = 256, output_median: float = 700):
    """A serving trace for the scheduling model: Poisson arrivals at qps,
    prompt lengths lognormal (median prompt_median, sigma 1, clipped 16-4096),
    output lengths lognormal (median output_median, sigma 0.8, clipped 1-8192),
    and stand-in static predictions output * exp(pred_sigma * N(0, 1)) as f32
    (pred_sigma = 0: exact predictions).  Returns a dict of numpy arrays."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed).spawn(6)[5]))
    arrival = np.cumsum(rng.exponential(1.0 / qps, size=n))
    prompt = np.clip(np.rint(rng.lognormal(math.log(prompt_median), 1.0, n)), 16, 4096).astype(np.int32)
    output = np.clip(np.rint(rng.lognormal(math.log(output_median), 0.8, n)), 1, 8192).astype(np.int32)
    noise = np.exp(pred_sigma * rng.standard_normal(n))
    predicted = (output * noise).astype(np.float32)
    return {"arrival": arrival, "prompt": prompt, "output": output, "predicted": predicted}
