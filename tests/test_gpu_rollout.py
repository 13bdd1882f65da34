"""Draft rollouts (EAGLE-3-style multi-token drafting) on the GPU.

After a tapped step, outlets_predict_draft_step feeds each request's own
output state y back as the feature input for one more draft position (with
the drafted token's embedding when the context has the input-embedding
branch); outlets_kv_truncate drops draft positions the target rejected.
Compared with the oracle chain (predict_step with f_rows = previous y), and
rollback is checked bit-exactly against a run that never drafted.
"""
import numpy as np
import pytest

from oracle import outlets_oracle as OR
from paper_2609_01068_gb300 import synth
from _util import check_hidden, check_z_len, to_device, to_np

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

MID128 = synth.ModelShape("mid-bf16-hd128", 1024, 8, 2, 128, 2816, (256,), 500000.0, 1e-5, "bf16")
EV = 3001


def _setup(shape, embed, dual, pref, seed_off):
    from paper_2609_01068_gb300 import outlets as OT
    w = synth.make_weights(shape, 0, embed_vocab=EV if embed else 0)
    if dual:
        w["w_lm"] = synth.make_lm_head(shape, 2000, 0)
    pred = OT.Predictor(shape, w, max_tokens=4096, max_batch=16, max_position=4096)
    B = len(pref)
    kv = OT.KVCache(pred, max_slots=B, max_tokens_total=sum(pref) + 64 * B * 2)
    cu = synth.cu_seqlens(pref)
    taps = synth.make_taps(shape, int(cu[-1]), 0, seed_off)
    tok = synth.make_tokens(int(cu[-1]), EV, 0, seed_off) if embed else None
    slots = np.arange(B, dtype=np.int32)
    pred.prefill([to_device(t, shape.dtype) for t in taps], cu, kv=kv, slots=slots, tokens=tok)
    caches = OR.caches_from_prefill(OR.predict_prefill(w, shape, taps, cu, tokens=tok), cu)
    return pred, kv, w, slots, caches


@pytest.mark.parametrize("name,embed,dual", [("tiny-f32", False, False), ("mid128", True, True), ("mid128", False, False)])
def test_rollout_matches_oracle_chain(name, embed, dual):
    from paper_2609_01068_gb300 import outlets as OT
    shape = synth.TINY if name == "tiny-f32" else MID128
    pref = [1, 63, 64, 65, 300]
    pred, kv, w, slots, caches = _setup(shape, embed, dual, pref, 80)
    B = len(pref)
    st = synth.make_taps(shape, B, 0, 81)
    stok = synth.make_tokens(B, EV, 0, 81) if embed else None
    pred.step([to_device(t, shape.dtype) for t in st], kv, slots, tokens=stok)
    ref = OR.predict_step(w, shape, st, caches, tokens=stok)
    for k in range(3):  # three draft positions
        dtok = synth.make_tokens(B, EV, 0, 90 + k) if embed else None
        if dual:
            z, ln, out = pred.draft_step(kv, slots, tokens=dtok, k=4)
        else:
            z, ln = pred.draft_step(kv, slots, tokens=dtok)
        torch.cuda.synchronize()
        pred.check()
        ref = OR.predict_step(w, shape, None, ref["caches"], tokens=dtok, f_rows=ref["y"],
                              draft_k=4 if dual else None)
        check_hidden(pred.intermediate(OT.T_ATTN), ref["attn"], shape.dtype, f"{name} draft {k} attn")
        check_hidden(pred.intermediate(OT.T_Y), ref["y"], shape.dtype, f"{name} draft {k} y")
        check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"{name} draft {k}")
        if dual:
            np.testing.assert_allclose(to_np(out["lse"]), ref["draft"]["lse"], rtol=0, atol=3e-2)
        assert [kv.slot_length(int(s)) for s in slots] == [p + 2 + k for p in pref]
    kv.close()
    pred.close()


def test_rollback_is_bit_exact_with_never_drafting():
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pref = [7, 130, 64]
    B = len(pref)
    st1 = [to_device(t, "bf16") for t in synth.make_taps(shape, B, 0, 82)]
    st2 = [to_device(t, "bf16") for t in synth.make_taps(shape, B, 0, 83)]
    t1, t2 = synth.make_tokens(B, EV, 0, 82), synth.make_tokens(B, EV, 0, 83)
    # with two rejected draft positions
    pred, kv, w, slots, _ = _setup(shape, True, False, pref, 84)
    pred.step(st1, kv, slots, tokens=t1)
    pred.draft_step(kv, slots, tokens=synth.make_tokens(B, EV, 0, 85))
    pred.draft_step(kv, slots, tokens=synth.make_tokens(B, EV, 0, 86))
    for s, p in zip(slots, pref):
        kv.truncate(int(s), p + 1)
    za, la = pred.step(st2, kv, slots, tokens=t2)
    za, la = to_np(za), to_np(la)
    kv.close()
    pred.close()
    # never drafting
    pred, kv, w, slots, caches = _setup(shape, True, False, pref, 84)
    pred.step(st1, kv, slots, tokens=t1)
    zb, lb = pred.step(st2, kv, slots, tokens=t2)
    torch.cuda.synchronize()
    pred.check()
    np.testing.assert_array_equal(za, to_np(zb))
    np.testing.assert_array_equal(la, to_np(lb))
    r1 = OR.predict_step(w, shape, synth.make_taps(shape, B, 0, 82), caches, tokens=t1)
    r2 = OR.predict_step(w, shape, synth.make_taps(shape, B, 0, 83), r1["caches"], tokens=t2)
    check_z_len(zb, lb, r2["z"], r2["length"], "bf16", "after rollback")
    kv.close()
    pred.close()


def test_device_draft_ids_feed_the_next_draft_step():
    """The serving loop: the top-1 draft ids stay on the device and are the next
    draft step's tokens; the same ids passed from the host give the same result."""
    shape = MID128
    pref = [33, 200]
    B = len(pref)
    res = []
    for host in (False, True):
        pred, kv, w, slots, _ = _setup(shape, True, True, pref, 87)
        _, _, out = pred.step_dual([to_device(t, "bf16") for t in synth.make_taps(shape, B, 0, 88)], kv, slots, 1,
                                   tokens=synth.make_tokens(B, EV, 0, 88))
        ids = out["ids"][:, 0].contiguous() % EV  # draft vocabulary 2000 < EV
        z, ln, out2 = pred.draft_step(kv, slots, tokens=ids.cpu().numpy() if host else ids, k=1)
        torch.cuda.synchronize()
        pred.check()
        res.append((to_np(z), to_np(out2["lse"]), to_np(out2["ids"])))
        kv.close()
        pred.close()
    for a, b in zip(*res):
        np.testing.assert_array_equal(a, b)


def test_draft_step_misuse_is_rejected():
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pref = [5, 9]
    pred, kv, w, slots, _ = _setup(shape, True, False, pref, 89)
    tok = synth.make_tokens(2, EV, 0, 89)
    with pytest.raises(OT.OutletsError) as e:  # follows a prefill, not a step
        pred.draft_step(kv, slots, tokens=tok)
    assert e.value.status == OT.EINVAL
    pred.step([to_device(t, "bf16") for t in synth.make_taps(shape, 2, 0, 90)], kv, slots, tokens=tok)
    with pytest.raises(OT.OutletsError) as e:  # other slot order
        pred.draft_step(kv, slots[::-1].copy(), tokens=tok)
    assert e.value.status == OT.EINVAL
    with pytest.raises(OT.OutletsError) as e:  # the branch needs ids
        pred.draft_step(kv, slots)
    assert e.value.status == OT.EINVAL
    pred.draft_step(kv, slots, tokens=tok)  # still allowed after the rejected calls
    with pytest.raises(OT.OutletsError):
        kv.truncate(0, pref[0] + 3)  # longer than the slot
    kv.truncate(0, 0)
    assert kv.slot_length(0) == 0
    kv.close()
    pred.close()
