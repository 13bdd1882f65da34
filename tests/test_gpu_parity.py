"""CUDA path vs the CPU oracle, element by element, through the C ABI.

Small cases span several tiles and ragged tails (every intermediate checked);
the full-size configurations check sampled outputs the oracle computes one
sequence / request at a time (sequences never interact, Sec. 3.2).
"""
import numpy as np
import pytest

from oracle import outlets_oracle as OR
from paper_2609_01068_gb300 import synth
from _util import pruned, check_rows, HIDDEN_TOL, check_hidden, check_z_len, maxrel, to_device, to_np

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

MID128 = synth.ModelShape("mid-bf16-hd128", 1024, 8, 2, 128, 2816, (256,), 500000.0, 1e-5, "bf16")
MID64 = synth.ModelShape("mid-bf16-hd64", 512, 8, 4, 64, 1000, (128, 64), 10000.0, 1e-5, "bf16")
SHAPES = {"tiny-f32": synth.TINY, "mid128": MID128, "mid64": MID64}
PREFILL_LENGTHS = {
    "tiny-f32": [16, 32, 48, 64],
    "mid128": [1, 5, 63, 64, 65, 130, 200, 333],
    "mid64": [2, 64, 129, 71, 1],
}
STEP_PREFIX = {
    "tiny-f32": [1, 15, 63, 64, 65],
    "mid128": [1, 63, 64, 65, 511, 512, 513, 700],
    "mid64": [3, 64, 600, 1100],
}

_cache = {}


def predictor(name, max_tokens=4096, max_batch=64):
    from paper_2609_01068_gb300 import outlets
    key = (name, max_tokens, max_batch)
    if key not in _cache:
        shape = SHAPES[name]
        w = synth.make_weights(shape, 0)
        _cache[key] = (outlets.Predictor(shape, w, max_tokens=max_tokens, max_batch=max_batch, max_position=8192), w)
    return _cache[key]


def _taps(shape, T, off=0):
    return synth.make_taps(shape, T, 0, off)


@pytest.mark.parametrize("keep_rows", [True, False])
@pytest.mark.parametrize("name", list(SHAPES))
def test_prefill_matches_oracle_every_intermediate(name, keep_rows):
    """keep_rows: the whole layer on every row; otherwise (bf16, T > 256) q,
    attention, a and y exist for each sequence's last row only."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    pred, w = predictor(name)
    cu = synth.cu_seqlens(PREFILL_LENGTHS[name])
    taps = _taps(shape, int(cu[-1]))
    ref = OR.predict_prefill(w, shape, taps, cu)
    z, ln = pred.prefill([to_device(t, shape.dtype) for t in taps], cu, keep_rows=keep_rows)
    torch.cuda.synchronize()
    pred.check()
    T = int(cu[-1])
    pr = pruned(shape.dtype, T, keep_rows)
    for which, r, what in [(OT.T_FCTX, ref["f"], "f_ctx"), (OT.T_XIN, ref["x"], "x_in"),
                           (OT.T_HDRAFT, ref["h_draft"], "h_draft")]:
        check_hidden(pred.intermediate(which), r, shape.dtype, f"{name} {what}")
    for which, r, what in [(OT.T_Q, ref["q"].reshape(T, -1), "q"), (OT.T_ATTN, ref["attn"], "attn"),
                           (OT.T_A, ref["a"], "a"), (OT.T_Y, ref["y"], "y")]:
        check_rows(pred.intermediate(which), r, cu, shape.dtype, f"{name} {what}", pr)
    check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, name)


@pytest.mark.parametrize("name", ["mid128", "mid64"])
def test_pruned_prefill_writes_the_same_cache_as_the_whole_layer(name):
    """The static prediction of the last rows only projects keys and values
    for every row with the same GEMM tiles as the whole layer: the KV caches
    agree bit for bit (the steps after them do), and both predictions match
    the oracle."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    pred, w = predictor(name)
    lengths = PREFILL_LENGTHS[name]
    B = len(lengths)
    cu = synth.cu_seqlens(lengths)
    T = int(cu[-1])
    assert pruned(shape.dtype, T)
    taps_np = _taps(shape, T, off=81)
    taps = [to_device(t, shape.dtype) for t in taps_np]
    st = [to_device(t, shape.dtype) for t in synth.make_taps(shape, B, 0, 82)]
    slots = np.arange(B, dtype=np.int32)
    out = {}
    for keep in (True, False):
        kv = OT.KVCache(pred, max_slots=B, max_tokens_total=T + 64 * B)
        z, ln = pred.prefill(taps, cu, kv=kv, slots=slots, keep_rows=keep)
        z2, _ = pred.step(st, kv, slots)
        torch.cuda.synchronize()
        pred.check()
        out[keep] = (z.clone(), ln.clone(), to_np(z2))
        kv.close()
    np.testing.assert_array_equal(out[False][2], out[True][2])
    ref = OR.predict_prefill(w, shape, taps_np, cu)
    for keep in (True, False):
        check_z_len(out[keep][0], out[keep][1], ref["z"], ref["length"], shape.dtype, f"{name} keep_rows={keep}")


def test_pruned_prefill_more_than_256_prompts():
    """300 short prompts: the predicted rows take the large-M path (q / k / v
    of the last rows by the tcgen05 GEMM, O / MLP / head on 300 rows)."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID64
    pred, w = predictor("mid64", max_tokens=2048, max_batch=320)
    rng = np.random.default_rng(7)
    lengths = rng.integers(1, 7, size=300)
    B = len(lengths)
    cu = synth.cu_seqlens(lengths)
    T = int(cu[-1])
    assert pruned(shape.dtype, T) and B > 256
    taps_np = _taps(shape, T, off=91)
    taps = [to_device(t, shape.dtype) for t in taps_np]
    st = [to_device(t, shape.dtype) for t in synth.make_taps(shape, B, 0, 92)]
    slots = np.arange(B, dtype=np.int32)
    out = {}
    for keep in (True, False):
        kv = OT.KVCache(pred, max_slots=B, max_tokens_total=T + 64 * B)
        z, ln = pred.prefill(taps, cu, kv=kv, slots=slots, keep_rows=keep)
        torch.cuda.synchronize()
        pred.check()
        h = to_np(pred.intermediate(OT.T_HDRAFT))
        z2, ln2 = pred.step(st, kv, slots)
        torch.cuda.synchronize()
        pred.check()
        out[keep] = (z.clone(), ln.clone(), h, z2.clone(), ln2.clone())
        kv.close()
    np.testing.assert_array_equal(to_np(out[False][3]), to_np(out[True][3]))
    ref = OR.predict_prefill(w, shape, taps_np, cu)
    for keep in (True, False):
        check_z_len(out[keep][0], out[keep][1], ref["z"], ref["length"], shape.dtype, f"300 prompts keep_rows={keep}")
        check_hidden(out[keep][2], ref["h_draft"], shape.dtype, f"300 prompts h_draft keep_rows={keep}")
    ref2 = OR.predict_step(w, shape, synth.make_taps(shape, B, 0, 92), OR.caches_from_prefill(ref, cu))
    check_z_len(out[False][3], out[False][4], ref2["z"], ref2["length"], shape.dtype, "300 prompts step")


@pytest.mark.parametrize("name", ["tiny-f32", "mid128"])
def test_all_tokens_mode_and_causal_prefix(name):
    shape = SHAPES[name]
    pred, w = predictor(name)
    cu = synth.cu_seqlens(PREFILL_LENGTHS[name][-3:])
    taps = _taps(shape, int(cu[-1]), off=1)
    ref = OR.predict_prefill(w, shape, taps, cu, all_tokens=True)
    z, ln = pred.prefill([to_device(t, shape.dtype) for t in taps], cu, all_tokens=True)
    check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, name)
    # the per-token prediction at row k equals the prediction of the prompt cut after k
    zall = to_np(z)
    for b in range(len(cu) - 1):
        k = int(cu[b]) + (int(cu[b + 1]) - int(cu[b])) // 2
        sub = [t[int(cu[b]):k + 1] for t in taps]
        zk, _ = pred.prefill([to_device(t, shape.dtype) for t in sub], np.array([0, len(sub[0])], np.int32))
        assert abs(to_np(zk)[0] - zall[k]) <= (1e-5 if shape.dtype == "f32" else 2e-3)


@pytest.mark.parametrize("name", list(SHAPES))
def test_steps_match_oracle(name):
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    pred, w = predictor(name)
    pref = STEP_PREFIX[name]
    n_steps = 3
    B = len(pref)
    kv = OT.KVCache(pred, max_slots=B + 3, max_tokens_total=sum(pref) + B * (n_steps + 64))
    slots = np.arange(3, 3 + B, dtype=np.int32)[::-1].copy()
    cu = synth.cu_seqlens(pref)
    taps = _taps(shape, int(cu[-1]), off=2)
    free0 = kv.free_pages
    pred.prefill([to_device(t, shape.dtype) for t in taps], cu, kv=kv, slots=slots)
    assert [kv.slot_length(int(s)) for s in slots] == pref
    assert kv.free_pages == free0 - sum((L + 63) // 64 for L in pref)
    ref_pre = OR.predict_prefill(w, shape, taps, cu)
    caches = OR.caches_from_prefill(ref_pre, cu)
    for step in range(n_steps):
        st_taps = _taps(shape, B, off=10 + step)
        z, ln = pred.step([to_device(t, shape.dtype) for t in st_taps], kv, slots)
        torch.cuda.synchronize()
        pred.check()
        ref = OR.predict_step(w, shape, st_taps, caches)
        caches = ref["caches"]
        check_hidden(pred.intermediate(OT.T_ATTN), ref["attn"], shape.dtype, f"{name} step {step} attn")
        check_hidden(pred.intermediate(OT.T_HDRAFT), ref["h_draft"], shape.dtype, f"{name} step {step} h_draft")
        check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"{name} step {step}")
    assert [kv.slot_length(int(s)) for s in slots] == [L + n_steps for L in pref]
    kv.close()


@pytest.mark.parametrize("name", ["tiny-f32", "mid128"])
def test_prefill_then_steps_equals_all_tokens_on_gpu(name):
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    pred, w = predictor(name)
    lengths = [70, 9, 130]
    cu = synth.cu_seqlens(lengths)
    taps = _taps(shape, int(cu[-1]), off=3)
    z_all, _ = pred.prefill([to_device(t, shape.dtype) for t in taps], cu, all_tokens=True)
    z_all = to_np(z_all)
    kpre = [64, 1, 126]
    kv = OT.KVCache(pred, max_slots=3, max_tokens_total=1024)
    pre = [np.concatenate([t[cu[b]:cu[b] + kpre[b]] for b in range(3)]) for t in taps]
    pred.prefill([to_device(t, shape.dtype) for t in pre], synth.cu_seqlens(kpre), kv=kv, slots=[0, 1, 2])
    tol = 1e-5 if shape.dtype == "f32" else 5e-3
    for s in range(4):
        rows = [int(cu[b]) + kpre[b] + s for b in range(3)]
        z, _ = pred.step([to_device(t[rows], shape.dtype) for t in taps], kv, [0, 1, 2])
        assert np.max(np.abs(to_np(z) - z_all[rows])) <= tol
    kv.close()


def test_batch_permutation_invariance_gpu():
    shape = MID128
    pred, w = predictor("mid128")
    lengths = [40, 200, 3, 129]
    cu = synth.cu_seqlens(lengths)
    taps = _taps(shape, int(cu[-1]), off=4)
    z, _ = pred.prefill([to_device(t, "bf16") for t in taps], cu)
    z = to_np(z)
    perm = [3, 1, 0, 2]
    ptaps = [np.concatenate([t[cu[b]:cu[b + 1]] for b in perm]) for t in taps]
    zp, _ = pred.prefill([to_device(t, "bf16") for t in ptaps], synth.cu_seqlens([lengths[b] for b in perm]))
    np.testing.assert_allclose(to_np(zp), z[perm], rtol=0, atol=1e-5)


def test_host_buffers_match_device_buffers():
    shape = MID128
    pred, w = predictor("mid128")
    cu = synth.cu_seqlens([17, 90])
    taps = _taps(shape, int(cu[-1]), off=5)
    dev = [to_device(t, "bf16") for t in taps]
    z_d, l_d = pred.prefill(dev, cu)
    host = [t.cpu() for t in dev]
    z_h = torch.empty(2, dtype=torch.float32)
    l_h = torch.empty(2, dtype=torch.float32)
    pred.prefill(host, cu, z_out=z_h, len_out=l_h)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(z_h.numpy(), z_d.cpu().numpy())
    np.testing.assert_array_equal(l_h.numpy(), l_d.cpu().numpy())


def test_chunked_host_taps_match_device_taps():
    """Host taps of a large call are copied in row chunks that the front of the
    pipeline consumes as they land (a chunk boundary falls inside a sequence):
    the predictions, every cached key and the draft states must be identical to
    the same call on device taps."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred, w = predictor("mid128", max_tokens=8192)
    lengths = [1500, 2100, 1400, 37]
    cu = synth.cu_seqlens(lengths)
    T = int(cu[-1])
    taps = _taps(shape, T, off=13)
    dev = [to_device(t, "bf16") for t in taps]
    z_d, l_d = pred.prefill(dev, cu, all_tokens=True)
    h_d = to_np(pred.intermediate(OT.T_HDRAFT)).copy()
    host = [t.cpu().pin_memory() for t in dev]
    z_h = torch.empty(T, dtype=torch.float32).pin_memory()
    l_h = torch.empty(T, dtype=torch.float32).pin_memory()
    pred.prefill(host, cu, all_tokens=True, z_out=z_h, len_out=l_h)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(z_h.numpy(), z_d.cpu().numpy())
    np.testing.assert_array_equal(l_h.numpy(), l_d.cpu().numpy())
    np.testing.assert_array_equal(to_np(pred.intermediate(OT.T_HDRAFT)), h_d)
    ref = OR.predict_prefill(w, shape, taps, cu)
    last = torch.as_tensor(np.asarray(cu[1:]) - 1, dtype=torch.long)
    check_z_len(z_h[last], l_h[last], ref["z"], ref["length"], "bf16", "chunked host taps")


def test_wave_aligned_tap_chunks_match_device_taps():
    """A large call's host taps in chunks of whole FC waves (9 728 rows at
    d = 1024, 256 x 256 tiles over 152 SMs): T = 21 957 gives chunks starting
    at 0, 9 728 and 19 456, the last one partial and boundaries inside
    sequences. Every prediction and draft state must be identical to the same
    call on device taps."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred, w = predictor("mid128", max_tokens=24576)
    lengths = [8000, 7000, 6000, 957]
    cu = synth.cu_seqlens(lengths)
    T = int(cu[-1])
    taps = _taps(shape, T, off=17)
    dev = [to_device(t, "bf16") for t in taps]
    z_d, l_d = pred.prefill(dev, cu, all_tokens=True)
    h_d = to_np(pred.intermediate(OT.T_HDRAFT)).copy()
    host = [t.cpu().pin_memory() for t in dev]
    z_h = torch.empty(T, dtype=torch.float32).pin_memory()
    l_h = torch.empty(T, dtype=torch.float32).pin_memory()
    pred.prefill(host, cu, all_tokens=True, z_out=z_h, len_out=l_h)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(z_h.numpy(), z_d.cpu().numpy())
    np.testing.assert_array_equal(l_h.numpy(), l_d.cpu().numpy())
    np.testing.assert_array_equal(to_np(pred.intermediate(OT.T_HDRAFT)), h_d)


def test_argument_errors_change_nothing():
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred, w = predictor("mid128")
    kv = OT.KVCache(pred, max_slots=4, max_tokens_total=128)
    taps = [to_device(t, "bf16") for t in _taps(shape, 40, off=6)]
    with pytest.raises(OT.OutletsError) as e:
        pred.prefill(taps, np.array([0, 30, 20, 40], np.int32))       # not increasing
    assert e.value.status == OT.EINVAL
    with pytest.raises(OT.OutletsError) as e:
        pred.prefill(taps, np.array([0, 40], np.int32), kv=kv, slots=[7])  # slot out of range
    assert e.value.status == OT.EINVAL
    with pytest.raises(OT.OutletsError) as e:
        pred.prefill(taps, np.array([0, 20, 40], np.int32), kv=kv, slots=[1, 1])  # duplicate slots
    assert e.value.status == OT.EINVAL
    pred.prefill(taps, np.array([0, 40], np.int32), kv=kv, slots=[0])
    free = kv.free_pages
    # the pool holds ceil(128 / 64) + 4 = 6 pages; one is taken, 400 rows need 7
    assert free == 5
    big = [to_device(t, "bf16") for t in _taps(shape, 400, off=7)]
    with pytest.raises(OT.OutletsError) as e:
        pred.prefill(big, np.array([0, 400], np.int32), kv=kv, slots=[1])
    assert e.value.status == OT.ECAPACITY
    assert kv.free_pages == free and kv.slot_length(1) == 0 and kv.slot_length(0) == 40
    with pytest.raises(OT.OutletsError) as e:
        pred.step([t[:2] for t in taps], kv, [0, 0])
    assert e.value.status == OT.EINVAL
    assert kv.slot_length(0) == 40
    import ctypes
    z = torch.empty(1, dtype=torch.float32, device="cuda")
    tp = (ctypes.c_void_p * 3)(*[t.data_ptr() for t in taps])
    cu = np.array([0, 40], np.int32)
    for flags in (4, OT.ALL_TOKENS | OT.KEEP_ROWS | 8):  # unknown flag bits
        st = pred.lib.outlets_predict_prefill(pred.h, tp, cu.ctypes.data, 1, 40, None, None, flags, z.data_ptr(),
                                              None, None)
        assert st == OT.EINVAL
    pred.check()
    kv.close()


# ---------------------------------------------------------------- full-size configurations
def _sampled_prefill(shape, lengths, max_tokens, sample, seed_off, rows_too=False):
    """Full-size static prediction, sampled prompts against the oracle; with
    rows_too also the last rows of q, attention, a and y (the pruned order
    keeps them for each prompt's last row, in prompt order)."""
    from paper_2609_01068_gb300 import outlets as OT
    w = synth.make_weights(shape, 0)
    pred = OT.Predictor(shape, w, max_tokens=max_tokens, max_batch=len(lengths), max_position=8192)
    cu = synth.cu_seqlens(lengths)
    T = int(cu[-1])
    taps = synth.make_taps(shape, T, 0, seed_off)
    z, ln = pred.prefill([to_device(t, "bf16") for t in taps], cu)
    torch.cuda.synchronize()
    pred.check()
    hd = to_np(pred.intermediate(OT.T_HDRAFT))
    ref = OR.sample_prefill_rows(w, shape, taps, cu, sample)
    errs = {"z": check_z_len(z[sample], ln[sample], ref["z"], ref["length"], "bf16", shape.name)[0],
            "h_draft": check_hidden(hd[sample], ref["h_draft"], "bf16", f"{shape.name} h_draft")}
    if rows_too:
        assert pruned("bf16", T)
        sub_last = np.cumsum([lengths[b] for b in sample]) - 1
        for which, key in ((OT.T_Q, "q"), (OT.T_ATTN, "attn"), (OT.T_A, "a"), (OT.T_Y, "y")):
            g = to_np(pred.intermediate(which))[sample]
            r = np.asarray(ref[key]).reshape(len(ref[key]), -1)[sub_last]
            errs[key] = check_hidden(g, r, "bf16", f"{shape.name} {key}")
    pred.close()
    return errs


def test_llama8b_prefill_full_size_sampled():
    lengths = synth.lengths_8b_prefill(0)
    order = np.argsort(lengths)
    sample = [int(order[0]), int(order[1]), int(order[len(order) // 2]), int(order[-1])]
    _sampled_prefill(synth.LLAMA8B, lengths, 32768, sample, 0)


def test_llama70b_prefill_sampled():
    """The shortest, the median and the longest (4096-token) prompt of the
    70B-shaped workload: z, h_draft and the last rows of q, attention, a, y."""
    lengths = synth.lengths_70b_prefill(0)
    order = np.argsort(lengths, kind="stable")
    sample = [int(order[0]), int(order[len(order) // 2]), int(order[-1])]
    assert lengths[sample[-1]] == 4096
    errs = _sampled_prefill(synth.LLAMA70B, lengths, 65536, sample, 0, rows_too=True)
    print("70B sampled errors:", errs)


def test_long_prompt_positions_to_8191_match_oracle():
    """A prompt of 8192 tokens (the largest position the sweep reaches) with
    short ones: RoPE and attention at positions up to 8191, in both orders of
    the static prediction (whole layer on every row, last rows only)."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred, w = predictor("mid128", max_tokens=9216)
    lengths = [3, 8192, 700, 64]
    cu = synth.cu_seqlens(lengths)
    T = int(cu[-1])
    taps = _taps(shape, T, off=71)
    ref = OR.predict_prefill(w, shape, taps, cu)
    taps_d = [to_device(t, shape.dtype) for t in taps]
    for keep in (True, False):
        z, ln = pred.prefill(taps_d, cu, keep_rows=keep)
        torch.cuda.synchronize()
        pred.check()
        pr = pruned(shape.dtype, T, keep)
        for which, r, what in [(OT.T_Q, ref["q"].reshape(T, -1), "q"), (OT.T_ATTN, ref["attn"], "attn"),
                               (OT.T_A, ref["a"], "a"), (OT.T_Y, ref["y"], "y")]:
            check_rows(pred.intermediate(which), r, cu, shape.dtype, f"8192-token prompt keep_rows={keep} {what}",
                       pr)
        check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"8192-token prompt keep_rows={keep}")


def test_steps_at_long_cache_lengths():
    """Steps whose cache lengths cross a 64-position page boundary far out
    (4095 -> 4096 -> 4097) and reach the last position (8190 -> 8191)."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred, w = predictor("mid128", max_tokens=16896)
    pref = [8190, 4095, 4096, 5]
    B = len(pref)
    kv = OT.KVCache(pred, max_slots=B, max_tokens_total=sum(pref) + 64 * B)
    slots = np.arange(B, dtype=np.int32)
    cu = synth.cu_seqlens(pref)
    taps = _taps(shape, int(cu[-1]), off=72)
    pred.prefill([to_device(t, shape.dtype) for t in taps], cu, kv=kv, slots=slots)
    caches = OR.caches_from_prefill(OR.predict_prefill(w, shape, taps, cu), cu)
    for step in range(2):
        st_taps = _taps(shape, B, off=73 + step)
        z, ln = pred.step([to_device(t, shape.dtype) for t in st_taps], kv, slots)
        torch.cuda.synchronize()
        pred.check()
        ref = OR.predict_step(w, shape, st_taps, caches)
        caches = ref["caches"]
        check_hidden(pred.intermediate(OT.T_Q), ref["q"].reshape(B, -1), shape.dtype, f"long step {step} q")
        check_hidden(pred.intermediate(OT.T_ATTN), ref["attn"], shape.dtype, f"long step {step} attn")
        check_hidden(pred.intermediate(OT.T_Y), ref["y"], shape.dtype, f"long step {step} y")
        check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"long step {step}")
    assert [kv.slot_length(int(s)) for s in slots] == [L + 2 for L in pref]
    kv.close()


def test_llama8b_step_full_size_sampled():
    from paper_2609_01068_gb300 import outlets as OT
    shape = synth.LLAMA8B
    w = synth.make_weights(shape, 0)
    lens = synth.lengths_8b_step_cache(0)
    B = len(lens)
    pred = OT.Predictor(shape, w, max_tokens=32768, max_batch=B, max_position=8192)
    kv = OT.KVCache(pred, max_slots=B, max_tokens_total=int(lens.sum()) + 64 * B)
    order = np.argsort(lens)
    sample = [int(order[0]), int(order[1]), int(np.argmin(np.abs(lens - 700))), int(np.argmin(np.abs(lens - 1500)))]
    gen = torch.Generator(device="cuda").manual_seed(0)
    sample_taps = {b: synth.make_taps(shape, int(lens[b]), 0, 100 + b) for b in sample}
    # fill the cache: prompts packed into prefill calls of <= 32768 rows
    b = 0
    while b < B:
        e, tot = b, 0
        while e < B and tot + lens[e] <= 32768:
            tot += int(lens[e])
            e += 1
        parts = [[], [], []]
        for r in range(b, e):
            for i in range(3):
                if r in sample_taps:
                    parts[i].append(to_device(sample_taps[r][i], "bf16"))
                else:
                    parts[i].append(torch.randn(int(lens[r]), shape.d, device="cuda", generator=gen).to(torch.bfloat16))
        taps = [torch.cat(p).contiguous() for p in parts]
        pred.prefill(taps, synth.cu_seqlens(lens[b:e]), kv=kv, slots=np.arange(b, e, dtype=np.int32))
        b = e
    step_taps = synth.make_taps(shape, B, 0, 99)
    z, ln = pred.step([to_device(t, "bf16") for t in step_taps], kv, np.arange(B, dtype=np.int32))
    torch.cuda.synchronize()
    pred.check()
    attn = to_np(pred.intermediate(OT.T_ATTN))
    for r in sample:
        pre = OR.predict_prefill(w, shape, sample_taps[r], np.array([0, lens[r]]))
        ref = OR.predict_step(w, shape, [t[r:r + 1] for t in step_taps], OR.caches_from_prefill(pre, [0, lens[r]]))
        check_z_len(z[r:r + 1], ln[r:r + 1], ref["z"], ref["length"], "bf16", f"step request {r} (Lc={lens[r]})")
        check_hidden(attn[r:r + 1], ref["attn"], "bf16", f"step attn request {r}")
    kv.close()
    pred.close()


def test_sweep_batch_full_size_sampled():
    """The serving sweep's largest prefill batch (<= 131072 tokens of the heavy-tailed
    mixture, arrival order) and one step over its requests, sampled against the oracle."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = synth.LLAMA8B
    w = synth.make_weights(shape, 0)
    lengths = synth.lengths_sweep(0)
    batch, tot = [], 0
    for i, L in enumerate(lengths):
        if tot + L > 131072:
            break
        batch.append(i)
        tot += int(L)
    lens = lengths[batch]
    B = len(batch)
    pred = OT.Predictor(shape, w, max_tokens=131072, max_batch=512, max_position=16384)
    kv = OT.KVCache(pred, max_slots=B, max_tokens_total=tot + 128 * B)
    order = np.argsort(lens)
    sample = [int(order[0]), int(order[1]), int(np.argmin(np.abs(lens - 600)))]
    sample_taps = {b: synth.make_taps(shape, int(lens[b]), 0, 500 + b) for b in sample}
    gen = torch.Generator(device="cuda").manual_seed(3)
    parts = [[], [], []]
    for r in range(B):
        for i in range(3):
            if r in sample_taps:
                parts[i].append(to_device(sample_taps[r][i], "bf16"))
            else:
                parts[i].append(torch.randn(int(lens[r]), shape.d, device="cuda", generator=gen).to(torch.bfloat16))
    taps = [torch.cat(p).contiguous() for p in parts]
    z, ln = pred.prefill(taps, synth.cu_seqlens(lens), kv=kv, slots=np.arange(B, dtype=np.int32))
    torch.cuda.synchronize()
    pred.check()
    step_taps = synth.make_taps(shape, B, 0, 501)
    zs, ls = pred.step([to_device(t, "bf16") for t in step_taps], kv, np.arange(B, dtype=np.int32))
    torch.cuda.synchronize()
    pred.check()
    for r in sample:
        pre = OR.predict_prefill(w, shape, sample_taps[r], np.array([0, lens[r]]))
        check_z_len(z[r:r + 1], ln[r:r + 1], pre["z"], pre["length"], "bf16", f"sweep prefill request {r}")
        st = OR.predict_step(w, shape, [t[r:r + 1] for t in step_taps], OR.caches_from_prefill(pre, [0, lens[r]]))
        check_z_len(zs[r:r + 1], ls[r:r + 1], st["z"], st["length"], "bf16", f"sweep step request {r}")
    kv.close()
    pred.close()


def test_bounded_wait_timeout_is_reported_and_context_survives():
    """A kernel whose wait never completes gives up after its limit, the host
    reads OUTLETS_ETIMEOUT, and the next prediction is still correct."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = MID128
    pred, w = predictor("mid128")
    pred.check()
    pred.selftest_bounded_wait(timeout_ns=2_000_000)
    with pytest.raises(OT.OutletsError) as e:
        pred.check()
    assert e.value.status == OT.ETIMEOUT
    pred.check()  # the error word was cleared
    cu = synth.cu_seqlens([9, 70])
    taps = _taps(shape, int(cu[-1]), off=8)
    z, ln = pred.prefill([to_device(t, "bf16") for t in taps], cu)
    ref = OR.predict_prefill(w, shape, taps, cu)
    check_z_len(z, ln, ref["z"], ref["length"], "bf16", "after timeout")
    pred.check()


@pytest.mark.parametrize("name,gated,embed", [("tiny-f32", False, False), ("mid128", False, False),
                                              ("mid128", True, True), ("mid64", False, False)])
def test_nonunit_norm_gains(name, gated, embed):
    """RMSNorm gains other than 1.  On the bf16 path g_in and g_post are folded
    into the QKV and gate/up weights at upload and the large-M path folds the
    norms into its GEMMs (bf16 copies, sums of squares, row scales), so unit
    gains would not test any of it.  Prefill (large M) and steps (small M)."""
    from paper_2609_01068_gb300 import outlets as OT
    shape = SHAPES[name]
    ev = 500 if embed else 0
    w = synth.make_weights(shape, 0, gated=gated, embed_vocab=ev)
    rng = np.random.default_rng(17)
    for g in ("g_in", "g_post", "g_final") + (("g_emb",) if embed else ()):
        w[g] = (1.0 + 0.2 * rng.standard_normal(shape.d)).astype(np.float32)
    pred = OT.Predictor(shape, w, max_tokens=4096, max_batch=16, max_position=8192)
    lengths = PREFILL_LENGTHS[name]
    B = len(lengths)
    cu = synth.cu_seqlens(lengths)
    T = int(cu[-1])
    taps = synth.make_taps(shape, T, 0, 61)
    tok = synth.make_tokens(T, ev, 0, 61) if embed else None
    kv = OT.KVCache(pred, max_slots=B, max_tokens_total=T + 64 * B)
    slots = np.arange(B, dtype=np.int32)
    z, ln = pred.prefill([to_device(t, shape.dtype) for t in taps], cu, kv=kv, slots=slots, tokens=tok)
    torch.cuda.synchronize()
    pred.check()
    ref = OR.predict_prefill(w, shape, taps, cu, tokens=tok)
    d = shape.d
    pr = pruned(shape.dtype, T)
    for which, r, what in [(OT.T_XIN, ref["x"][:, -d:], "x_in"), (OT.T_HDRAFT, ref["h_draft"], "h_draft")]:
        check_hidden(pred.intermediate(which), r, shape.dtype, f"gains {name} {what}")
    for which, r, what in [(OT.T_Q, ref["q"].reshape(T, -1), "q"), (OT.T_A, ref["a"], "a"), (OT.T_Y, ref["y"], "y")]:
        check_rows(pred.intermediate(which), r, cu, shape.dtype, f"gains {name} {what}", pr)
    check_z_len(z, ln, ref["z"], ref["length"], shape.dtype, f"gains {name} prefill")
    caches = OR.caches_from_prefill(ref, cu)
    st = synth.make_taps(shape, B, 0, 62)
    stok = synth.make_tokens(B, ev, 0, 62) if embed else None
    z2, ln2 = pred.step([to_device(t, shape.dtype) for t in st], kv, slots, tokens=stok)
    torch.cuda.synchronize()
    pred.check()
    ref2 = OR.predict_step(w, shape, st, caches, tokens=stok)
    check_hidden(pred.intermediate(OT.T_XIN), ref2["x"][:, -d:], shape.dtype, f"gains {name} step x_in")
    check_hidden(pred.intermediate(OT.T_Y), ref2["y"], shape.dtype, f"gains {name} step y")
    check_z_len(z2, ln2, ref2["z"], ref2["length"], shape.dtype, f"gains {name} step")
    kv.close()
    pred.close()


_L2_KEEP_SCRIPT = r"""
import sys, numpy as np, torch
sys.path.insert(0, sys.argv[1]); sys.path.insert(0, sys.argv[1] + "/tests")
from paper_2609_01068_gb300 import outlets, synth
from _util import to_device
shape = synth.ModelShape("mid-bf16-hd128", 1024, 8, 2, 128, 2816, (256,), 500000.0, 1e-5, "bf16")
w = synth.make_weights(shape, 0)
pred = outlets.Predictor(shape, w, max_tokens=2048, max_batch=8, max_position=4096)
lengths = [70, 300, 5, 129]
cu = synth.cu_seqlens(lengths)
kv = outlets.KVCache(pred, max_slots=4, max_tokens_total=1024)
taps = [to_device(t, "bf16") for t in synth.make_taps(shape, int(cu[-1]), 0, 95)]
z0, _ = pred.prefill(taps, cu, kv=kv, slots=[0, 1, 2, 3])
st = [to_device(t, "bf16") for t in synth.make_taps(shape, 4, 0, 96)]
z1, _ = pred.step(st, kv, [0, 1, 2, 3])
torch.cuda.synchronize()
pred.check()
np.save(sys.argv[2], np.concatenate([z0.cpu().numpy(), z1.cpu().numpy()]))
"""


def test_slice_discard_changes_no_value(tmp_path):
    """Dropping the split-K slices from L2 after their last read
    (OUTLETS_L2_DISCARD, default on) changes no output bit: the same static
    prediction and step in two processes, with the discards and without."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    script = tmp_path / "run.py"
    script.write_text(_L2_KEEP_SCRIPT)
    out = {}
    for v in ("1", "0"):
        env = dict(os.environ, OUTLETS_L2_DISCARD=v)
        f = tmp_path / f"z{v}.npy"
        r = subprocess.run([sys.executable, str(script), root, str(f)], env=env, capture_output=True, text=True,
                           timeout=600)
        assert r.returncode == 0, r.stderr[-2000:]
        out[v] = np.load(f)
    np.testing.assert_array_equal(out["1"], out["0"])
