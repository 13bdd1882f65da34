"""Shared helpers of the GPU parity tests (inputs, tolerances, comparisons)."""
import numpy as np

from paper_2609_01068_gb300 import synth

# Tolerances: hidden states as max_i |g - r| / max_i |r| per tensor; z_hat absolute;
# length relative to max(length, 1).
HIDDEN_TOL = {"f32": 1e-4, "bf16": 2e-2}
Z_TOL = {"f32": 1e-4, "bf16": 1e-2}
LEN_TOL = 1e-2


def maxrel(g, r):
    g = np.asarray(g, dtype=np.float64)
    r = np.asarray(r, dtype=np.float64)
    return float(np.max(np.abs(g - r)) / max(float(np.max(np.abs(r))), 1e-30))


def to_device(arr, dtype):
    """float32 numpy -> CUDA tensor in the path's dtype (bit-exact for bf16-representable values)."""
    import torch
    if dtype == "bf16":
        bits = synth.bf16_bits(arr).view(np.int16)
        return torch.from_numpy(bits).view(torch.bfloat16).cuda()
    return torch.from_numpy(np.ascontiguousarray(arr, np.float32)).cuda()


def to_np(t):
    return t.float().cpu().numpy().astype(np.float64)


def check_z_len(z_gpu, len_gpu, z_ref, len_ref, dtype, what=""):
    z_gpu, len_gpu = to_np(z_gpu), to_np(len_gpu)
    dz = np.max(np.abs(z_gpu - z_ref))
    assert dz <= Z_TOL[dtype], f"{what} z_hat max abs error {dz}"
    dl = np.max(np.abs(len_gpu - len_ref) / np.maximum(len_ref, 1.0))
    assert dl <= LEN_TOL, f"{what} length max rel error {dl}"
    return dz, dl


def check_hidden(g, r, dtype, what):
    e = maxrel(to_np(g) if not isinstance(g, np.ndarray) else g, r)
    assert e <= HIDDEN_TOL[dtype], f"{what}: max relative error {e}"
    return e


def pruned(dtype, T, keep_rows=False, all_tokens=False):
    """Whether a static prediction runs past the K/V projection on the
    predicted rows only: bf16, more than 256 rows, last rows predicted, and
    keep_rows not asked for."""
    return dtype == "bf16" and T > 256 and not keep_rows and not all_tokens


def check_rows(g, r_all, cu, dtype, what, is_pruned):
    """A per-row intermediate against the oracle: every row, or each
    sequence's last row (in sequence order) after a pruned prediction."""
    r = np.asarray(r_all)[np.asarray(cu[1:]) - 1] if is_pruned else r_all
    g = to_np(g) if not isinstance(g, np.ndarray) else g
    assert g.shape[0] == r.shape[0], f"{what}: {g.shape[0]} rows, expected {r.shape[0]}"
    return check_hidden(g, r, dtype, what)
