"""outlets_length_head_noalloc against the prediction call's own length head.

The entry point serves callers that cannot call cudaMalloc while they serve
(all spare device memory handed to a KV-cache pool, or no tolerance for
cudaMalloc's implicit device synchronization).  Given the draft states of a
prefill call it must return the same z_hat and lengths as that call, on every
call (its scratch array keeps the previous call's contents).
"""
import numpy as np
import pytest

from paper_2609_01068_gb300 import synth
from _util import LEN_TOL, Z_TOL, to_device, to_np

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

SHAPES = {
    "bf16-head-1-hidden": synth.ModelShape("na-a", 1024, 8, 2, 128, 2816, (256,), 500000.0, 1e-5, "bf16"),
    "bf16-head-2-hidden": synth.ModelShape("na-b", 512, 8, 4, 64, 1000, (128, 64), 10000.0, 1e-5, "bf16"),
    "f32-head-1-hidden": synth.TINY,
}


@pytest.mark.parametrize("name", list(SHAPES))
def test_noalloc_head_matches_prefill_head(name):
    from paper_2609_01068_gb300 import outlets as OT
    lib = OT.load()
    shape = SHAPES[name]
    w = synth.make_weights(shape, 0)
    pred = OT.Predictor(shape, w, max_tokens=1024, max_batch=16, max_position=2048)
    lengths = [5, 64, 130, 1, 77]
    cu = synth.cu_seqlens(lengths)
    taps = synth.make_taps(shape, int(cu[-1]), 0, 21)
    z_ref, l_ref = pred.prefill([to_device(t, shape.dtype) for t in taps], cu)
    h = pred.intermediate(OT.T_HDRAFT)
    torch.cuda.synchronize()
    z_ref, l_ref = to_np(z_ref), to_np(l_ref)
    B = len(lengths)
    stream = torch.cuda.current_stream().cuda_stream
    for call in range(2):
        z = torch.full((B,), float("nan"), dtype=torch.float32, device="cuda")
        ln = torch.full((B,), float("nan"), dtype=torch.float32, device="cuda")
        st = lib.outlets_length_head_noalloc(pred.h, h.data_ptr(), B, z.data_ptr(), ln.data_ptr(), stream)
        assert st == OT.OK, lib.outlets_last_error(pred.h)
        torch.cuda.synchronize()
        dz = np.max(np.abs(to_np(z) - z_ref))
        dl = np.max(np.abs(to_np(ln) - l_ref) / np.maximum(l_ref, 1.0))
        assert dz <= Z_TOL[shape.dtype], f"call {call}: z_hat differs by {dz}"
        assert dl <= LEN_TOL, f"call {call}: length differs by {dl}"
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
