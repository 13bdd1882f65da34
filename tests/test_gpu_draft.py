"""Dual head, draft branch (Sec. 4.2, Eq. 2) on the GPU against the oracle.

P_draft = softmax(W_lm h^draft): the library returns each row's k most
probable tokens, their log-probabilities and the logsumexp (and, on request,
the logits).  The tensor-core path never writes the logits: its GEMM epilogue
reduces every tile to softmax statistics and a local top-k, and a merge
kernel combines the tiles.

Token ids are an integer decided by floating point: where the oracle's
neighbouring logits are further apart than the comparison tolerance the id
must match exactly; inside a near-tie any of the tied tokens is accepted
(its oracle logit must be within tolerance of the oracle's value at that
rank).  Tolerances: given states (identical bf16 inputs on both sides, f32
accumulation) 1e-3 absolute on logits and log-probabilities; through the
bf16 backbone (the state itself carries bf16 rounding) 3e-2.
"""
import numpy as np
import pytest

from oracle import outlets_oracle as OR
from paper_2609_01068_gb300 import synth
from _util import check_z_len, to_device, to_np

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

MID128 = synth.ModelShape("mid-bf16-hd128", 1024, 8, 2, 128, 2816, (256,), 500000.0, 1e-5, "bf16")
SHAPES = {"tiny-f32": synth.TINY, "mid128": MID128}
VOCAB = {"tiny-f32": 1000, "mid128": 5003}  # not a multiple of any tile width: ragged last tile
TOL_GIVEN = {"f32": 1e-4, "bf16": 1e-3}
TOL_BACKBONE = {"f32": 1e-4, "bf16": 3e-2}

_cache = {}


def dual_predictor(name, vocab=None, max_tokens=4096, max_batch=300):
    from paper_2609_01068_gb300 import outlets
    shape = SHAPES[name] if isinstance(name, str) else name
    vocab = vocab or VOCAB[shape.name if shape.name in VOCAB else name]
    key = (shape.name, vocab, max_tokens, max_batch)
    if key not in _cache:
        w = synth.make_weights(shape, 0)
        w["w_lm"] = synth.make_lm_head(shape, vocab, 0)
        _cache[key] = (outlets.Predictor(shape, w, max_tokens=max_tokens, max_batch=max_batch, max_position=8192), w)
    return _cache[key]


def check_draft(got, ref_logits, k, tol, what):
    """got: {"ids", "logprob", "lse"[, "logits"]} (torch or numpy); ref_logits: oracle logits [rows, V]."""
    ids = to_np(torch.as_tensor(got["ids"])).astype(np.int64)
    lp = to_np(torch.as_tensor(got["logprob"]))
    lse = to_np(torch.as_tensor(got["lse"]))
    ref_lp, ref_lse = OR.log_softmax_rows(ref_logits)
    rows, V = ref_logits.shape
    assert ids.shape == (rows, k) and lp.shape == (rows, k)
    err = np.max(np.abs(lse - ref_lse))
    assert err <= tol, f"{what}: logsumexp error {err}"
    ref_ids = OR.top_k_tokens(ref_logits, min(k + 1, V))
    for r in range(rows):
        assert len(set(ids[r].tolist())) == k and ids[r].min() >= 0 and ids[r].max() < V, f"{what}: row {r} ids {ids[r]}"
        assert np.all(np.diff(lp[r]) <= 1e-6), f"{what}: row {r} not sorted"
        vals = ref_logits[r, ref_ids[r]]
        for i in range(k):
            g = ids[r, i]
            # the reported log-probability is that of the reported token
            assert abs(lp[r, i] - ref_lp[r, g]) <= tol, f"{what}: row {r} rank {i} logprob {lp[r, i]} vs {ref_lp[r, g]}"
            # the token holds rank i up to the tolerance
            assert abs(ref_logits[r, g] - vals[i]) <= 2 * tol, f"{what}: row {r} rank {i} token {g} not a valid choice"
            gap = min(vals[i - 1] - vals[i] if i > 0 else np.inf, vals[i] - vals[i + 1] if i + 1 < len(vals) else np.inf)
            if gap > 2 * tol:
                assert g == ref_ids[r, i], f"{what}: row {r} rank {i}: {g} != {ref_ids[r, i]} (gap {gap})"
    if "logits" in got:
        e = np.max(np.abs(to_np(torch.as_tensor(got["logits"])) - ref_logits))
        assert e <= tol, f"{what}: logits error {e}"


@pytest.mark.parametrize("name", list(SHAPES))
@pytest.mark.parametrize("rows", [1, 100, 129, 256, 300])
@pytest.mark.parametrize("k", [1, 5, 8])
def test_draft_head_on_given_states_matches_oracle(name, rows, k):
    shape = SHAPES[name]
    pred, w = dual_predictor(name)
    h = synth.make_draft_states(shape, rows, 0, rows * 10 + k)
    out = pred.draft_head(to_device(h, shape.dtype), k, logits=(k == 5))
    torch.cuda.synchronize()
    pred.check()
    check_draft(out, OR.draft_logits(h, w["w_lm"]), k, TOL_GIVEN[shape.dtype], f"{name} rows={rows} k={k}")


def test_draft_head_smallest_vocab_is_a_full_sort():
    shape = MID128
    pred, w = dual_predictor(shape, vocab=8, max_batch=64)
    h = synth.make_draft_states(shape, 37, 0, 7)
    out = pred.draft_head(to_device(h, "bf16"), 8)
    torch.cuda.synchronize()
    check_draft(out, OR.draft_logits(h, w["w_lm"]), 8, TOL_GIVEN["bf16"], "V=8")


@pytest.mark.parametrize("name", list(SHAPES))
def test_dual_prefill_matches_oracle(name):
    shape = SHAPES[name]
    pred, w = dual_predictor(name)
    cu = synth.cu_seqlens([1, 5, 63, 64, 65, 130, 200, 333] if shape.dtype == "bf16" else [16, 32, 48, 64])
    taps = synth.make_taps(shape, int(cu[-1]), 0, 50)
    ref = OR.predict_prefill(w, shape, taps, cu, draft_k=8)
    z, ln, out = pred.prefill_dual([to_device(t, shape.dtype) for t in taps], cu, 8, logits=True)
    torch.cuda.synchronize()
    pred.check()
    check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"dual {name}")
    check_draft(out, ref["draft"]["logits"], 8, TOL_BACKBONE[shape.dtype], f"dual prefill {name}")


@pytest.mark.parametrize("name", list(SHAPES))
def test_dual_steps_match_oracle(name):
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    pred, w = dual_predictor(name)
    pref = [1, 63, 64, 65, 511, 700] if shape.dtype == "bf16" else [1, 15, 63, 64, 65]
    B = len(pref)
    kv = OT.KVCache(pred, max_slots=B, max_tokens_total=sum(pref) + 64 * B)
    slots = np.arange(B, dtype=np.int32)
    cu = synth.cu_seqlens(pref)
    taps = synth.make_taps(shape, int(cu[-1]), 0, 51)
    pred.prefill([to_device(t, shape.dtype) for t in taps], cu, kv=kv, slots=slots)
    caches = OR.caches_from_prefill(OR.predict_prefill(w, shape, taps, cu), cu)
    for step in range(2):
        st = synth.make_taps(shape, B, 0, 60 + step)
        z, ln, out = pred.step_dual([to_device(t, shape.dtype) for t in st], kv, slots, 4)
        torch.cuda.synchronize()
        pred.check()
        ref = OR.predict_step(w, shape, st, caches, draft_k=4)
        caches = ref["caches"]
        check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"dual {name} step {step}")
        check_draft(out, ref["draft"]["logits"], 4, TOL_BACKBONE[shape.dtype], f"dual step {name} {step}")
    kv.close()


def test_dual_all_tokens_spans_several_passes():
    """600 predicted rows: three 256-row passes of the draft head."""
    shape = MID128
    pred, w = dual_predictor("mid128")
    cu = synth.cu_seqlens([300, 1, 299])
    taps = synth.make_taps(shape, int(cu[-1]), 0, 52)
    ref = OR.predict_prefill(w, shape, taps, cu, all_tokens=True, draft_k=2)
    z, ln, out = pred.prefill_dual([to_device(t, "bf16") for t in taps], cu, 2, all_tokens=True)
    torch.cuda.synchronize()
    pred.check()
    check_z_len(z, ln, ref["z"], ref["length"], "bf16", "dual all tokens")
    check_draft(out, ref["draft"]["logits"], 2, TOL_BACKBONE["bf16"], "dual all tokens")


def test_host_outputs_equal_device_outputs():
    shape = MID128
    pred, w = dual_predictor("mid128")
    h = to_device(synth.make_draft_states(shape, 260, 0, 3), "bf16")
    dev = pred.draft_head(h, 8, logits=True)
    host = {"ids": np.zeros((260, 8), np.int32), "logprob": np.zeros((260, 8), np.float32),
            "lse": np.zeros(260, np.float32), "logits": np.zeros((260, pred.vocab), np.float32)}
    pred.draft_head(h, 8, out=host)
    torch.cuda.synchronize()
    for key in host:
        np.testing.assert_array_equal(host[key], torch.as_tensor(dev[key]).cpu().numpy(), err_msg=key)


def test_draft_argument_errors():
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred, _ = dual_predictor("mid128")
    h = to_device(synth.make_draft_states(shape, 4, 0, 4), "bf16")
    for k in (0, 9):
        with pytest.raises(OT.OutletsError) as e:
            pred.draft_head(h, k)
        assert e.value.status == OT.EINVAL
    plain = OT.Predictor(shape, synth.make_weights(shape, 0), max_tokens=256, max_batch=8, max_position=1024)
    with pytest.raises(OT.OutletsError) as e:
        plain.draft_head(h, 1)
    assert e.value.status == OT.EUNSUPPORTED
    plain.close()


@pytest.mark.parametrize("rows", [64, 256])
def test_llama3_vocab_full_size_sampled(rows):
    """The draft head at the Llama-3 vocabulary (V = 128256, d = 4096) in the
    launch shapes of static (64 rows) and dynamic (256 rows) prediction; the
    oracle computes sampled rows."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = synth.LLAMA8B
    w = synth.make_weights(shape, 0)
    w["w_lm"] = synth.make_lm_head(shape, synth.LLAMA3_VOCAB, 0)
    pred = OT.Predictor(shape, w, max_tokens=512, max_batch=256, max_position=1024)
    h = synth.make_draft_states(shape, rows, 0, 11)
    out = pred.draft_head(to_device(h, "bf16"), 8)
    torch.cuda.synchronize()
    pred.check()
    sample = [0, rows // 2 + 1, rows - 1]
    got = {key: torch.as_tensor(out[key])[sample] for key in ("ids", "logprob", "lse")}
    check_draft(got, OR.draft_logits(h[sample], w["w_lm"]), 8, TOL_GIVEN["bf16"], f"llama3 vocab rows={rows}")
    pred.close()


def test_uniform_distribution_ties_go_to_smallest_ids():
    """W_lm = 0: every logit ties at 0 (the uniform case of Eq. 2).  With
    V = 40000 every partial tile keeps 8 tied entries, more than the merge
    gathers in shared memory, so this also covers its fallback path."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    w = synth.make_weights(shape, 0)
    V = 40000
    w["w_lm"] = np.zeros((V, shape.d), np.float32)
    pred = OT.Predictor(shape, w, max_tokens=256, max_batch=64, max_position=1024)
    h = synth.make_draft_states(shape, 37, 0, 5)
    for k in (1, 8):
        out = pred.draft_head(to_device(h, "bf16"), k)
        torch.cuda.synchronize()
        pred.check()
        assert torch.as_tensor(out["ids"]).cpu().numpy().tolist() == [list(range(k))] * 37
        np.testing.assert_allclose(to_np(torch.as_tensor(out["logprob"])), -np.log(V), rtol=0, atol=1e-4)
        ref = OR.draft_head(h, w["w_lm"], k)
        np.testing.assert_array_equal(ref["topk_ids"], np.tile(np.arange(k), (37, 1)))
    pred.close()
