"""outlets_length_head_noalloc: the length head for callers that cannot allocate.

The entry point serves callers that cannot call cudaMalloc while they serve
(all spare device memory handed to a KV-cache pool at start-up, or no
tolerance for cudaMalloc's implicit device synchronization).  Given the draft
states of a prefill call it must return the oracle's z_hat and lengths for
those states, and the same values as the prediction call's own head, on every
call (its scratch array keeps the previous call's contents), without taking
any device memory.
"""
import numpy as np
import pytest

from oracle import outlets_oracle as OR
from paper_2609_01068_gb300 import synth
from _util import LEN_TOL, Z_TOL, to_device, to_np

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

SHAPES = {
    "bf16-head-1-hidden": synth.ModelShape("na-a", 1024, 8, 2, 128, 2816, (256,), 500000.0, 1e-5, "bf16"),
    "bf16-head-2-hidden": synth.ModelShape("na-b", 512, 8, 4, 64, 1000, (128, 64), 10000.0, 1e-5, "bf16"),
    "f32-head-1-hidden": synth.TINY,
    "f32-head-2-hidden": synth.ModelShape("na-c", 256, 4, 2, 64, 688, (128, 64), 10000.0, 1e-5, "f32"),
}


@pytest.mark.parametrize("name", list(SHAPES))
def test_noalloc_head_matches_oracle_and_prefill_head(name):
    from paper_2609_01068_gb300 import outlets as OT
    lib = OT.load()
    shape = SHAPES[name]
    w = synth.make_weights(shape, 0)
    pred = OT.Predictor(shape, w, max_tokens=1024, max_batch=16, max_position=2048)
    lengths = [5, 64, 130, 1, 77]
    cu = synth.cu_seqlens(lengths)
    taps = synth.make_taps(shape, int(cu[-1]), 0, 21)
    z_pred, l_pred = pred.prefill([to_device(t, shape.dtype) for t in taps], cu)
    h = pred.intermediate(OT.T_HDRAFT)
    torch.cuda.synchronize()
    z_pred, l_pred = to_np(z_pred), to_np(l_pred)
    # the oracle's head (fp64) on the very states the entry point is given
    ws, bs = OR.head_weights(w)
    z_ref = OR.length_head(to_np(h), ws, bs)
    l_ref = OR.z_to_length(z_ref)
    B = len(lengths)
    stream = torch.cuda.current_stream().cuda_stream
    outs = [(torch.full((B,), float("nan"), dtype=torch.float32, device="cuda"),
             torch.full((B,), float("nan"), dtype=torch.float32, device="cuda")) for _ in range(2)]
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for z, ln in outs:  # two calls in a row
        st = lib.outlets_length_head_noalloc(pred.h, h.data_ptr(), B, z.data_ptr(), ln.data_ptr(), stream)
        assert st == OT.OK, lib.outlets_last_error(pred.h)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, f"free device memory changed by {free0 - free1} bytes across the calls"
    for call, (z, ln) in enumerate(outs):
        z, ln = to_np(z), to_np(ln)
        for what, zr, lr in (("oracle", z_ref, l_ref), ("prediction call", z_pred, l_pred)):
            dz = np.max(np.abs(z - zr))
            dl = np.max(np.abs(ln - lr) / np.maximum(lr, 1.0))
            assert dz <= Z_TOL[shape.dtype], f"call {call}: z_hat differs from the {what} by {dz}"
            assert dl <= LEN_TOL, f"call {call}: length differs from the {what} by {dl}"
    pred.check()
    pred.close()


def test_noalloc_head_rejects_rows_beyond_its_scratch():
    from paper_2609_01068_gb300 import outlets as OT
    lib = OT.load()
    shape = SHAPES["bf16-head-1-hidden"]
    pred = OT.Predictor(shape, synth.make_weights(shape, 0), max_tokens=256, max_batch=16, max_position=512)
    rows = (4 << 20) // shape.head_widths[0] + 1
    h = torch.zeros((rows, shape.d), dtype=torch.bfloat16, device="cuda")
    z = torch.empty(rows, dtype=torch.float32, device="cuda")
    st = lib.outlets_length_head_noalloc(pred.h, h.data_ptr(), rows, z.data_ptr(), None,
                                         torch.cuda.current_stream().cuda_stream)
    assert st == OT.ECAPACITY
    assert b"scratch" in lib.outlets_last_error(pred.h)
    pred.close()


def test_noalloc_head_at_its_row_limit():
    """The largest batch the scratch admits (a multi-wave head GEMM) still
    matches the oracle."""
    from paper_2609_01068_gb300 import outlets as OT
    lib = OT.load()
    shape = SHAPES["bf16-head-1-hidden"]
    w = synth.make_weights(shape, 0)
    pred = OT.Predictor(shape, w, max_tokens=256, max_batch=16, max_position=512)
    rows = (4 << 20) // shape.head_widths[0]
    hs = synth.make_draft_states(shape, rows, 0, 33)
    h = to_device(hs, "bf16")
    z = torch.empty(rows, dtype=torch.float32, device="cuda")
    st = lib.outlets_length_head_noalloc(pred.h, h.data_ptr(), rows, z.data_ptr(), None,
                                         torch.cuda.current_stream().cuda_stream)
    assert st == OT.OK, lib.outlets_last_error(pred.h)
    torch.cuda.synchronize()
    ws, bs = OR.head_weights(w)
    sample = np.arange(0, rows, 997)
    z_ref = OR.length_head(hs[sample].astype(np.float64), ws, bs)
    dz = np.max(np.abs(to_np(z)[sample] - z_ref))
    assert dz <= Z_TOL["bf16"], f"z_hat differs from the oracle by {dz}"
    pred.check()
    pred.close()
