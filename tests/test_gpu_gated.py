"""Gated attention (Sec. 4.1) on the GPU against the oracle.

With gate weights W_ag the QKV GEMM carries H*hd extra columns; RoPE/scatter
turns them into sigmoid(x_hat W_ag^T) and every attention kernel multiplies its
output by that gate.  Covered: the f32 CUDA-core path, the bf16 tensor-core
prefill path (large M), the small-M split-K path of dynamic prediction, and the
split-KV decode merge (long caches).
"""
import numpy as np
import pytest

from oracle import outlets_oracle as OR
from paper_2609_01068_gb300 import synth
from _util import check_hidden, check_rows, check_z_len, pruned, to_device

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

MID128 = synth.ModelShape("mid-bf16-hd128", 1024, 8, 2, 128, 2816, (256,), 500000.0, 1e-5, "bf16")
MID64 = synth.ModelShape("mid-bf16-hd64", 512, 8, 4, 64, 1000, (128, 64), 10000.0, 1e-5, "bf16")
SHAPES = {"tiny-f32": synth.TINY, "mid128": MID128, "mid64": MID64}
PREFILL_LENGTHS = {"tiny-f32": [16, 32, 48, 64], "mid128": [1, 5, 63, 64, 65, 130, 200, 333],
                   "mid64": [2, 64, 129, 71, 1]}
STEP_PREFIX = {"tiny-f32": [1, 15, 63, 64, 65], "mid128": [1, 63, 64, 65, 511, 512, 513, 2700],
               "mid64": [3, 64, 600, 1100]}

_cache = {}


def gated_predictor(name, max_tokens=4096, max_batch=64):
    from paper_2609_01068_gb300 import outlets
    key = (name, max_tokens, max_batch)
    if key not in _cache:
        shape = SHAPES[name]
        w = synth.make_weights(shape, 0, gated=True)
        _cache[key] = (outlets.Predictor(shape, w, max_tokens=max_tokens, max_batch=max_batch, max_position=8192), w)
    return _cache[key]


@pytest.mark.parametrize("name", list(SHAPES))
def test_gated_prefill_matches_oracle_every_intermediate(name):
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    pred, w = gated_predictor(name)
    cu = synth.cu_seqlens(PREFILL_LENGTHS[name])
    taps = synth.make_taps(shape, int(cu[-1]), 0, 31)
    ref = OR.predict_prefill(w, shape, taps, cu)
    z, ln = pred.prefill([to_device(t, shape.dtype) for t in taps], cu)
    torch.cuda.synchronize()
    pred.check()
    T = int(cu[-1])
    pr = pruned(shape.dtype, T)
    for which, r, what in [(OT.T_Q, ref["q"].reshape(T, -1), "q"), (OT.T_ATTN, ref["attn"], "gated attn"),
                           (OT.T_A, ref["a"], "a")]:
        check_rows(pred.intermediate(which), r, cu, shape.dtype, f"gated {name} {what}", pr)
    check_hidden(pred.intermediate(OT.T_HDRAFT), ref["h_draft"], shape.dtype, f"gated {name} h_draft")
    check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"gated {name}")


@pytest.mark.parametrize("name", list(SHAPES))
def test_gated_steps_match_oracle(name):
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    pred, w = gated_predictor(name, max_tokens=8192)
    pref = STEP_PREFIX[name]
    B, n_steps = len(pref), 2
    kv = OT.KVCache(pred, max_slots=B, max_tokens_total=sum(pref) + B * (n_steps + 64))
    slots = np.arange(B, dtype=np.int32)
    cu = synth.cu_seqlens(pref)
    taps = synth.make_taps(shape, int(cu[-1]), 0, 32)
    pred.prefill([to_device(t, shape.dtype) for t in taps], cu, kv=kv, slots=slots)
    caches = OR.caches_from_prefill(OR.predict_prefill(w, shape, taps, cu), cu)
    for step in range(n_steps):
        st = synth.make_taps(shape, B, 0, 40 + step)
        z, ln = pred.step([to_device(t, shape.dtype) for t in st], kv, slots)
        torch.cuda.synchronize()
        pred.check()
        ref = OR.predict_step(w, shape, st, caches)
        caches = ref["caches"]
        check_hidden(pred.intermediate(OT.T_ATTN), ref["attn"], shape.dtype, f"gated {name} step {step} attn")
        check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"gated {name} step {step}")
    kv.close()


def test_gate_changes_the_prediction():
    """The gate is really applied: the same inputs without gate weights give a
    different attention output (and the ungated library matches the ungated
    oracle, so the difference is the gate)."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred_g, w = gated_predictor("mid128")
    w0 = {k: v for k, v in w.items() if k != "w_attn_gate"}
    pred_0 = OT.Predictor(shape, w0, max_tokens=1024, max_batch=8, max_position=2048)
    cu = synth.cu_seqlens([70, 33])
    taps = synth.make_taps(shape, int(cu[-1]), 0, 33)
    dev = [to_device(t, "bf16") for t in taps]
    pred_g.prefill(dev, cu)
    a_g = pred_g.intermediate(OT.T_ATTN).float().cpu().numpy()
    pred_0.prefill(dev, cu)
    a_0 = pred_0.intermediate(OT.T_ATTN).float().cpu().numpy()
    ref0 = OR.predict_prefill(w0, shape, taps, cu)
    check_hidden(pred_0.intermediate(OT.T_ATTN), ref0["attn"], "bf16", "ungated attn")
    assert np.max(np.abs(a_g - a_0)) > 0.1 * np.max(np.abs(a_0))
    pred_0.close()
