"""Input-embedding branch of the EAGLE-3-style draft layer (Sec. 5.4) on the GPU.

The layer input is Concat(RMSNorm(E[token]; g_emb), RMSNorm(f_ctx; g_in)):
the embedding kernel writes the normalized embedding rows and the QKV GEMM
reads them as the first d of its 2d input columns.  Compared with the oracle
on every intermediate (small shapes), through steps (host and device token
ids, with gated attention and the draft head), with chunked host taps, on
the error paths, and sampled at the 8B shape with the Llama-3 vocabulary.
"""
import numpy as np
import pytest

from oracle import outlets_oracle as OR
from paper_2609_01068_gb300 import synth
from _util import check_hidden, check_rows, check_z_len, pruned, to_device, to_np

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

MID128 = synth.ModelShape("mid-bf16-hd128", 1024, 8, 2, 128, 2816, (256,), 500000.0, 1e-5, "bf16")
MID64 = synth.ModelShape("mid-bf16-hd64", 512, 8, 4, 64, 1000, (128, 64), 10000.0, 1e-5, "bf16")
SHAPES = {"tiny-f32": synth.TINY, "mid128": MID128, "mid64": MID64}
EV = 3001
PREFILL_LENGTHS = {"tiny-f32": [16, 32, 48, 64], "mid128": [1, 5, 63, 64, 65, 130, 200, 333],
                   "mid64": [2, 64, 129, 71, 1]}

_cache = {}


def embed_predictor(name, gated=False, dual=False, max_tokens=8192, max_batch=64):
    from paper_2609_01068_gb300 import outlets
    key = (name, gated, dual, max_tokens, max_batch)
    if key not in _cache:
        shape = SHAPES[name]
        w = synth.make_weights(shape, 0, gated=gated, embed_vocab=EV)
        if dual:
            w["w_lm"] = synth.make_lm_head(shape, 2000, 0)
        _cache[key] = (outlets.Predictor(shape, w, max_tokens=max_tokens, max_batch=max_batch, max_position=8192), w)
    return _cache[key]


@pytest.mark.parametrize("name", list(SHAPES))
def test_embed_prefill_matches_oracle_every_intermediate(name):
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    pred, w = embed_predictor(name)
    cu = synth.cu_seqlens(PREFILL_LENGTHS[name])
    T = int(cu[-1])
    taps = synth.make_taps(shape, T, 0, 70)
    tok = synth.make_tokens(T, EV, 0, 1)
    ref = OR.predict_prefill(w, shape, taps, cu, tokens=tok)
    z, ln = pred.prefill([to_device(t, shape.dtype) for t in taps], cu, tokens=tok)
    torch.cuda.synchronize()
    pred.check()
    d = shape.d
    pr = pruned(shape.dtype, T)
    for which, r, what in [(OT.T_XIN, ref["x"][:, d:], "x_in (fused-feature half)"),
                           (OT.T_HDRAFT, ref["h_draft"], "h_draft")]:
        check_hidden(pred.intermediate(which), r, shape.dtype, f"embed {name} {what}")
    for which, r, what in [(OT.T_Q, ref["q"].reshape(T, -1), "q"), (OT.T_ATTN, ref["attn"], "attn"),
                           (OT.T_A, ref["a"], "a")]:
        check_rows(pred.intermediate(which), r, cu, shape.dtype, f"embed {name} {what}", pr)
    check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"embed {name}")


@pytest.mark.parametrize("name,gated", [("tiny-f32", False), ("mid128", True), ("mid64", False)])
def test_embed_steps_match_oracle(name, gated):
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    pred, w = embed_predictor(name, gated=gated)
    pref = [1, 63, 64, 65, 511, 1100] if shape.dtype == "bf16" else [1, 15, 63, 64, 65]
    B = len(pref)
    kv = OT.KVCache(pred, max_slots=B, max_tokens_total=sum(pref) + 64 * B)
    slots = np.arange(B, dtype=np.int32)
    cu = synth.cu_seqlens(pref)
    taps = synth.make_taps(shape, int(cu[-1]), 0, 71)
    tok = synth.make_tokens(int(cu[-1]), EV, 0, 2)
    pred.prefill([to_device(t, shape.dtype) for t in taps], cu, kv=kv, slots=slots, tokens=tok)
    caches = OR.caches_from_prefill(OR.predict_prefill(w, shape, taps, cu, tokens=tok), cu)
    for step in range(2):
        st = synth.make_taps(shape, B, 0, 72 + step)
        stok = synth.make_tokens(B, EV, 0, 10 + step)
        dev_tok = torch.from_numpy(stok).cuda() if step == 1 else stok  # device ids on the second step
        z, ln = pred.step([to_device(t, shape.dtype) for t in st], kv, slots, tokens=dev_tok)
        torch.cuda.synchronize()
        pred.check()
        ref = OR.predict_step(w, shape, st, caches, tokens=stok)
        caches = ref["caches"]
        check_hidden(pred.intermediate(OT.T_ATTN), ref["attn"], shape.dtype, f"embed {name} step {step} attn")
        check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"embed {name} step {step}")
    kv.close()


def test_embed_with_draft_head_step():
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred, w = embed_predictor("mid128", dual=True)
    pref = [7, 300, 64]
    B = len(pref)
    kv = OT.KVCache(pred, max_slots=B, max_tokens_total=sum(pref) + 64 * B)
    slots = np.arange(B, dtype=np.int32)
    cu = synth.cu_seqlens(pref)
    taps = synth.make_taps(shape, int(cu[-1]), 0, 73)
    tok = synth.make_tokens(int(cu[-1]), EV, 0, 3)
    z0, l0, d0 = pred.prefill_dual([to_device(t, "bf16") for t in taps], cu, 4, kv=kv, slots=slots, tokens=tok)
    ref0 = OR.predict_prefill(w, shape, taps, cu, tokens=tok, draft_k=4)
    check_z_len(z0, l0, ref0["z"], ref0["length"], "bf16", "embed dual prefill")
    np.testing.assert_allclose(to_np(d0["lse"]), ref0["draft"]["lse"], rtol=0, atol=3e-2)
    caches = OR.caches_from_prefill(OR.predict_prefill(w, shape, taps, cu, tokens=tok), cu)
    st = synth.make_taps(shape, B, 0, 74)
    stok = synth.make_tokens(B, EV, 0, 20)
    z, ln, d = pred.step_dual([to_device(t, "bf16") for t in st], kv, slots, 4, tokens=stok)
    torch.cuda.synchronize()
    pred.check()
    ref = OR.predict_step(w, shape, st, caches, tokens=stok, draft_k=4)
    check_z_len(z, ln, ref["z"], ref["length"], "bf16", "embed dual step")
    np.testing.assert_allclose(to_np(d["lse"]), ref["draft"]["lse"], rtol=0, atol=3e-2)
    np.testing.assert_allclose(to_np(d["logprob"]), ref["draft"]["topk_logprob"], rtol=0, atol=3e-2)
    kv.close()


def test_embed_chunked_host_taps_match_device_taps():
    """Host taps of a large call are copied in row chunks; every chunk's
    embedding rows must line up with its own rows."""
    shape = MID128
    pred, w = embed_predictor("mid128")
    cu = synth.cu_seqlens([1500, 2100, 1400, 37])
    T = int(cu[-1])
    taps = synth.make_taps(shape, T, 0, 75)
    tok = synth.make_tokens(T, EV, 0, 4)
    dev = [to_device(t, "bf16") for t in taps]
    zd, _ = pred.prefill(dev, cu, tokens=tok)
    zd = to_np(zd)
    host = [t.cpu().pin_memory() for t in dev]
    zh, _ = pred.prefill(host, cu, tokens=torch.from_numpy(tok).cuda())
    torch.cuda.synchronize()
    pred.check()
    np.testing.assert_array_equal(to_np(zh), zd)
    ref = OR.sample_prefill_rows(w, shape, taps, cu, [1, 3], tokens=tok)
    np.testing.assert_allclose(zd[[1, 3]], ref["z"], rtol=0, atol=1e-2)


def test_embed_token_errors():
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred, w = embed_predictor("mid128")
    cu = synth.cu_seqlens([5, 9])
    taps = [to_device(t, "bf16") for t in synth.make_taps(shape, 14, 0, 76)]
    tok = synth.make_tokens(14, EV, 0, 5)
    with pytest.raises(OT.OutletsError) as e:  # the branch needs ids
        pred.prefill(taps, cu)
    assert e.value.status == OT.EINVAL
    bad = tok.copy()
    bad[3] = EV
    with pytest.raises(OT.OutletsError) as e:  # host ids are checked on the host
        pred.prefill(taps, cu, tokens=bad)
    assert e.value.status == OT.EINVAL
    z_ok, _ = pred.prefill(taps, cu, tokens=tok)
    z_ok = to_np(z_ok)
    dbad = torch.from_numpy(bad).cuda()
    pred.prefill(taps, cu, tokens=dbad)  # device ids: the kernel refuses id EV and reports it
    with pytest.raises(OT.OutletsError) as e:
        pred.check()
    assert e.value.status == OT.EDEVICE
    z2, _ = pred.prefill(taps, cu, tokens=tok)  # the context still works
    pred.check()
    np.testing.assert_array_equal(to_np(z2), z_ok)
    plain = OT.Predictor(shape, synth.make_weights(shape, 0), max_tokens=256, max_batch=8, max_position=1024)
    with pytest.raises(OT.OutletsError) as e:  # ids without the branch
        plain.prefill(taps, cu, tokens=tok)
    assert e.value.status == OT.EINVAL
    plain.close()


def test_llama8b_embed_prefill_full_size_sampled():
    """8B shape, Llama-3 vocabulary embedding table (128 256 x 4096), the 64
    static-prediction prompts; the oracle computes sampled prompts."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = synth.LLAMA8B
    w = synth.make_weights(shape, 0, embed_vocab=synth.LLAMA3_VOCAB)
    lengths = synth.lengths_8b_prefill(0)
    cu = synth.cu_seqlens(lengths)
    T = int(cu[-1])
    pred = OT.Predictor(shape, w, max_tokens=32768, max_batch=len(lengths), max_position=8192)
    taps = synth.make_taps(shape, T, 0, 0)
    tok = synth.make_tokens(T, synth.LLAMA3_VOCAB, 0, 0)
    z, ln = pred.prefill([to_device(t, "bf16") for t in taps], cu, tokens=tok)
    torch.cuda.synchronize()
    pred.check()
    order = np.argsort(lengths)
    sample = [int(order[0]), int(order[len(order) // 2])]
    ref = OR.sample_prefill_rows(w, shape, taps, cu, sample, tokens=tok)
    check_z_len(z[sample], ln[sample], ref["z"], ref["length"], "bf16", "8b embed")
    check_hidden(to_np(pred.intermediate(OT.T_HDRAFT))[sample], ref["h_draft"], "bf16", "8b embed h_draft")
    pred.close()
