"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks one oracle function against something other than itself:
a closed form, a special case, brute force on a tiny input, an invariant, a
library routine, or a fact the paper states (tests/golden/paper_facts.json).
"""
import json
import math
import os

import numpy as np
import pytest

from oracle import outlets_oracle as O
from paper_2609_01068_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_facts.json")


def _facts():
    with open(GOLDEN) as fh:
        return json.load(fh)


SMALL = synth.ModelShape("pin-small", 32, 4, 2, 8, 48, (16,), 10000.0, 1e-5, "f32")


def _weights(shape=SMALL, seed=0):
    return synth.make_weights(shape, seed)


def _taps(shape, T, seed=0, off=0):
    return synth.make_taps(shape, T, seed, off)


# ---------------------------------------------------------------- golden facts
def test_tap_layer_indices_match_paper():
    """Pins the input generator's tap selection (which target layers feed Eq. 1), not the oracle."""
    for c in _facts()["tap_layers"]["cases"]:
        assert list(synth.tap_layer_indices(c["n_layers"])) == c["layers"]


def test_log_space_target_round_trip():
    # z = log(1 + length) (Sec. 4.2) and the oracle's inverse
    for c in _facts()["log_space_target"]["cases"]:
        assert math.isclose(math.log1p(c["length"]), c["z"], rel_tol=0, abs_tol=1e-15)
        assert O.z_to_length(np.array([c["z"]]))[0] == pytest.approx(c["length"], rel=1e-12, abs=1e-12)
    assert O.z_to_length(np.array([-3.0]))[0] == 0.0


def test_head_parameter_count_consistent_with_paper():
    fact = _facts()["head_params_d2048"]

    def count(widths):
        shape = synth.ModelShape("p", widths[0], 1, 1, 2, 2, tuple(widths[1:-1]), 1e4, 1e-5, "f32")
        n = 0
        w = {}
        for i in range(len(widths) - 1):
            w[f"head_w{i}"] = np.zeros((widths[i + 1], widths[i]))
            w[f"head_b{i}"] = np.zeros(widths[i + 1])
        ws, bs = O.head_weights(w)
        for a, b in zip(ws, bs):
            n += a.size + b.size
        return n, shape

    n_ok, _ = count(fact["widths_consistent"])
    n_bad, _ = count(fact["widths_inconsistent"])
    assert abs(n_ok - fact["approx_params"]) / fact["approx_params"] < fact["rel_tol"]
    assert abs(n_bad - fact["approx_params"]) / fact["approx_params"] > fact["rel_tol"]


# ---------------------------------------------------------------- head
def test_zero_weight_head_returns_output_bias():
    w = _weights()
    h = np.random.default_rng(1).standard_normal((5, SMALL.d))
    ws, bs = O.head_weights(w)
    zero_ws = [np.zeros_like(a) for a in ws]
    z = O.length_head(h, zero_ws, bs)
    assert np.all(z == np.float64(bs[-1][0]))


def test_head_relu_all_active_is_affine():
    rng = np.random.default_rng(2)
    W1 = rng.standard_normal((6, 4))
    W2 = rng.standard_normal((1, 6))
    b1 = np.full(6, 1e3)     # every pre-activation positive: ReLU is the identity
    b2 = np.array([0.25])
    h = rng.standard_normal((7, 4))
    z = O.length_head(h, [W1, W2], [b1, b2])
    np.testing.assert_allclose(z, h @ (W2 @ W1).T[:, 0] + (W2 @ b1)[0] + b2[0], rtol=1e-12)


def test_head_relu_all_dead_gives_bias():
    rng = np.random.default_rng(3)
    W1 = rng.standard_normal((6, 4))
    W2 = rng.standard_normal((1, 6))
    z = O.length_head(rng.standard_normal((7, 4)), [W1, W2], [np.full(6, -1e3), np.array([1.5])])
    assert np.all(z == 1.5)


def test_head_relu_brute_force():
    rng = np.random.default_rng(4)
    W1, b1 = rng.standard_normal((5, 3)), rng.standard_normal(5)
    W2, b2 = rng.standard_normal((1, 5)), rng.standard_normal(1)
    h = rng.standard_normal((4, 3))
    z = O.length_head(h, [W1, W2], [b1, b2])
    for r in range(4):
        acc = b2[0]
        for j in range(5):
            pre = b1[j]
            for i in range(3):
                pre += W1[j, i] * h[r, i]
            if pre > 0:
                acc += W2[0, j] * pre
        assert z[r] == pytest.approx(acc, rel=1e-12, abs=1e-12)


# ---------------------------------------------------------------- Eq. 1
def test_fc_identity_blocks_select_each_tap():
    d = 8
    taps = [np.random.default_rng(i).standard_normal((5, d)) for i in range(3)]
    for j in range(3):
        w = np.zeros((d, 3 * d))
        w[:, j * d:(j + 1) * d] = np.eye(d)
        np.testing.assert_array_equal(O.fuse_taps(taps, w), taps[j])


def test_fc_is_linear_in_each_tap():
    rng = np.random.default_rng(5)
    d = 6
    w = rng.standard_normal((d, 3 * d))
    t = [rng.standard_normal((3, d)) for _ in range(3)]
    t2 = [rng.standard_normal((3, d)) for _ in range(3)]
    lhs = O.fuse_taps([a + 2 * b for a, b in zip(t, t2)], w)
    np.testing.assert_allclose(lhs, O.fuse_taps(t, w) + 2 * O.fuse_taps(t2, w), rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------- RMSNorm
def test_rmsnorm_hand_example():
    # [3, 4]: mean square 12.5
    y = O.rms_norm(np.array([[3.0, 4.0]]), np.ones(2), 0.0)
    np.testing.assert_allclose(y, [[3 / math.sqrt(12.5), 4 / math.sqrt(12.5)]], rtol=1e-15)


def test_rmsnorm_unit_rms_and_scale_invariance():
    x = np.random.default_rng(6).standard_normal((9, 64))
    y = O.rms_norm(x, np.ones(64), 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y * y, axis=1)), 1.0, rtol=1e-12)
    np.testing.assert_allclose(O.rms_norm(7.5 * x, np.ones(64), 0.0), y, rtol=1e-12)
    g = np.random.default_rng(7).standard_normal(64)
    np.testing.assert_allclose(O.rms_norm(x, g, 0.0), y * g, rtol=1e-12)


# ---------------------------------------------------------------- RoPE
def test_rope_position_zero_is_identity_and_isometry():
    x = np.random.default_rng(8).standard_normal((5, 3, 16))
    np.testing.assert_array_equal(O.apply_rope(x, np.zeros(5, int), 1e4), x)
    y = O.apply_rope(x, np.arange(5) * 97, 5e5)
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-12)


def test_rope_frequency_schedule_closed_form():
    # Rotate unit vectors e_i at position 1 and read back each pair's angle.
    hd, theta = 16, 1e4
    half = hd // 2
    x = np.zeros((1, half, hd))
    for i in range(half):
        x[0, i, i] = 1.0
    y = O.apply_rope(x, np.array([1]), theta)[0]
    ang = np.array([math.atan2(y[i, i + half], y[i, i]) for i in range(half)])
    assert ang[0] == pytest.approx(1.0, abs=1e-15)             # theta^0 = 1 rad per position
    np.testing.assert_allclose(ang[1:] / ang[:-1], theta ** (-2.0 / hd), rtol=1e-12)
    # the rest of each rotated vector is zero: the pair is (i, i + hd/2)
    for i in range(half):
        rest = np.delete(y[i], [i, i + half])
        assert np.all(rest == 0)


def test_rope_composes_and_is_relative():
    rng = np.random.default_rng(9)
    q = rng.standard_normal((1, 1, 32))
    k = rng.standard_normal((1, 1, 32))
    theta = 5e5
    a = O.apply_rope(O.apply_rope(q, np.array([11]), theta), np.array([30]), theta)
    np.testing.assert_allclose(a, O.apply_rope(q, np.array([41]), theta), rtol=1e-10, atol=1e-12)
    s1 = np.sum(O.apply_rope(q, np.array([5]), theta) * O.apply_rope(k, np.array([2]), theta))
    s2 = np.sum(O.apply_rope(q, np.array([1005]), theta) * O.apply_rope(k, np.array([1002]), theta))
    assert s1 == pytest.approx(s2, rel=1e-9)


# ---------------------------------------------------------------- attention
def _rand_qkv(T, H, KVH, hd, seed):
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((T, H, hd)), rng.standard_normal((T, KVH, hd)),
            rng.standard_normal((T, KVH, hd)))


def test_attention_brute_force_loops():
    H, KVH, hd = 4, 2, 8
    cu = np.array([0, 3, 8, 9])
    q, k, v = _rand_qkv(9, H, KVH, hd, 10)
    out = O.causal_gqa_attention(q, k, v, cu)
    for b in range(3):
        for i in range(cu[b], cu[b + 1]):
            for h in range(H):
                g = h // (H // KVH)
                scores = []
                for j in range(cu[b], i + 1):
                    scores.append(sum(q[i, h, c] * k[j, g, c] for c in range(hd)) / math.sqrt(hd))
                mx = max(scores)
                ex = [math.exp(s - mx) for s in scores]
                tot = sum(ex)
                for c in range(hd):
                    ref = sum(ex[n] / tot * v[cu[b] + n, g, c] for n in range(len(ex)))
                    assert out[i, h, c] == pytest.approx(ref, rel=1e-10, abs=1e-12)


def test_attention_matches_torch_sdpa():
    torch = pytest.importorskip("torch")
    H, KVH, hd = 8, 2, 16
    cu = np.array([0, 5, 6, 30])
    q, k, v = _rand_qkv(30, H, KVH, hd, 11)
    out = O.causal_gqa_attention(q, k, v, cu)
    for b in range(3):
        s0, s1 = cu[b], cu[b + 1]
        tq = torch.from_numpy(q[s0:s1]).permute(1, 0, 2)[None]
        tk = torch.from_numpy(k[s0:s1]).permute(1, 0, 2).repeat_interleave(H // KVH, dim=0)[None]
        tv = torch.from_numpy(v[s0:s1]).permute(1, 0, 2).repeat_interleave(H // KVH, dim=0)[None]
        ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=True)
        np.testing.assert_allclose(out[s0:s1], ref[0].permute(1, 0, 2).numpy(), rtol=1e-10, atol=1e-12)


def test_gqa_with_replicated_kv_equals_mha():
    H, KVH, hd = 4, 2, 8
    cu = np.array([0, 7, 12])
    q, k, v = _rand_qkv(12, H, KVH, hd, 12)
    gqa = O.causal_gqa_attention(q, k, v, cu)
    mha = O.causal_gqa_attention(q, np.repeat(k, H // KVH, axis=1), np.repeat(v, H // KVH, axis=1), cu)
    np.testing.assert_allclose(gqa, mha, rtol=1e-13, atol=1e-14)


def test_attend_single_is_last_row_of_causal():
    H, KVH, hd = 4, 2, 8
    q, k, v = _rand_qkv(6, H, KVH, hd, 13)
    full = O.causal_gqa_attention(q, k, v, np.array([0, 6]))
    np.testing.assert_allclose(O.attend_single(q[5], k, v), full[5], rtol=1e-13, atol=1e-14)


# ---------------------------------------------------------------- SwiGLU
def test_silu_against_library_sigmoid():
    scipy_special = pytest.importorskip("scipy.special")
    x = np.linspace(-30, 30, 121)
    np.testing.assert_allclose(O.silu(x), x * scipy_special.expit(x), rtol=1e-13, atol=1e-300)
    assert O.silu(np.array([0.0]))[0] == 0.0


def test_swiglu_mlp_brute_force():
    """down(silu(x W_gate^T) * (x W_up^T)) (Sec. 4.1, the layer's MLP block read
    as SwiGLU) in scalar loops; distinct gate and up weights, so a swap fails."""
    rng = np.random.default_rng(31)
    d, F = 5, 4
    x = rng.standard_normal((3, d))
    wg, wu, wd = rng.standard_normal((F, d)), rng.standard_normal((F, d)), rng.standard_normal((d, F))
    got = O.swiglu_mlp(x, wg, wu, wd)
    for r in range(3):
        hid = []
        for n in range(F):
            g = sum(x[r, c] * wg[n, c] for c in range(d))
            u = sum(x[r, c] * wu[n, c] for c in range(d))
            hid.append(g / (1.0 + math.exp(-g)) * u)
        for i in range(d):
            assert got[r, i] == pytest.approx(sum(hid[n] * wd[i, n] for n in range(F)), rel=1e-12, abs=1e-12)
    # the two inner projections are not interchangeable
    assert np.max(np.abs(O.swiglu_mlp(x, wu, wg, wd) - got)) > 1e-3


def _scalar_layer(w, shape, taps, lengths):
    """One whole draft decoder layer and the length head in scalar Python loops,
    written from the definitions (Eq. 1; Sec. 4.1 pre-norm layer: RMSNorm,
    RoPE causal GQA attention, residual, RMSNorm, SwiGLU MLP, residual; final
    RMSNorm and MLP_len of Sec. 4.2 at each sequence's last row)."""
    d, H, KVH, hd, F = shape.d, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn
    eps, theta = shape.rms_eps, shape.rope_theta
    T = sum(lengths)

    def rms(vec, gain):
        ms = sum(v * v for v in vec) / len(vec)
        return [v / math.sqrt(ms + eps) * gn for v, gn in zip(vec, gain)]

    def matvec(W, vec):
        return [sum(W[o][c] * vec[c] for c in range(len(vec))) for o in range(len(W))]

    start, pos = [], []
    for b, L in enumerate(lengths):
        for p in range(L):
            start.append(sum(lengths[:b]))
            pos.append(p)
    f = []
    for t in range(T):
        f.append([sum(w["w_proj"][i][j * d + c] * taps[j][t][c] for j in range(3) for c in range(d))
                  for i in range(d)])
    x = [rms(f[t], w["g_in"]) for t in range(T)]

    def rope(vec, p):
        out = list(vec)
        half = hd // 2
        for i in range(half):
            ang = p * theta ** (-2.0 * i / hd)
            out[i] = vec[i] * math.cos(ang) - vec[i + half] * math.sin(ang)
            out[i + half] = vec[i + half] * math.cos(ang) + vec[i] * math.sin(ang)
        return out

    q = [[rope(matvec(w["w_q"], x[t])[h * hd:(h + 1) * hd], pos[t]) for h in range(H)] for t in range(T)]
    k = [[rope(matvec(w["w_k"], x[t])[g * hd:(g + 1) * hd], pos[t]) for g in range(KVH)] for t in range(T)]
    v = [[matvec(w["w_v"], x[t])[g * hd:(g + 1) * hd] for g in range(KVH)] for t in range(T)]
    a, y = [], []
    for t in range(T):
        o = []
        for h in range(H):
            g = h * KVH // H
            keys = range(start[t], t + 1)
            s = [sum(q[t][h][e] * k[j][g][e] for e in range(hd)) / math.sqrt(hd) for j in keys]
            m = max(s)
            p = [math.exp(si - m) for si in s]
            z = sum(p)
            o += [sum(p[n] * v[j][g][e] for n, j in enumerate(keys)) / z for e in range(hd)]
        at = [f[t][i] + sum(w["w_o"][i][c] * o[c] for c in range(H * hd)) for i in range(d)]
        ah = rms(at, w["g_post"])
        gate, up = matvec(w["w_gate"], ah), matvec(w["w_up"], ah)
        hid = [gate[n] / (1.0 + math.exp(-gate[n])) * up[n] for n in range(F)]
        a.append(at)
        y.append([at[i] + sum(w["w_down"][i][n] * hid[n] for n in range(F)) for i in range(d)])
    last = [sum(lengths[:b + 1]) - 1 for b in range(len(lengths))]
    hdraft = [rms(y[t], w["g_final"]) for t in last]
    zs = []
    for hrow in hdraft:
        cur = hrow
        n = len(shape.head_widths) + 1
        for i in range(n):
            nxt = [sum(w[f"head_w{i}"][o][c] * cur[c] for c in range(len(cur))) + w[f"head_b{i}"][o]
                   for o in range(len(w[f"head_w{i}"]))]
            cur = [max(0.0, u) for u in nxt] if i < n - 1 else nxt
        zs.append(cur[0])
    return dict(a=np.array(a), y=np.array(y), h_draft=np.array(hdraft), z=np.array(zs))


def test_whole_layer_scalar_brute_force():
    """The oracle's prefill against the scalar layer above on a tiny shape, with
    distinct random gate and up weights and distinct non-unit gains g_in,
    g_post and g_final, so a swapped projection, a norm of the wrong tensor or
    a gain used in the wrong place changes a, y, h_draft or z."""
    shape = synth.ModelShape("pin-layer", 8, 2, 1, 4, 6, (5,), 10000.0, 1e-5, "f32")
    rng = np.random.default_rng(41)
    w = {k: v.astype(np.float64) for k, v in synth.make_weights(shape, 3, std=0.4).items()}
    w["w_up"] = rng.standard_normal(w["w_up"].shape) * 0.5
    w["g_in"] = 1.0 + 0.5 * rng.standard_normal(shape.d)
    w["g_post"] = 1.0 + 0.5 * rng.standard_normal(shape.d)
    w["g_final"] = 1.0 + 0.5 * rng.standard_normal(shape.d)
    w["head_b1"] = np.array([0.3])
    lengths = [3, 2]
    taps = [rng.standard_normal((sum(lengths), shape.d)) for _ in range(3)]
    ref = _scalar_layer({k: np.asarray(v).tolist() for k, v in w.items()}, shape,
                        [t.tolist() for t in taps], lengths)
    out = O.predict_prefill(w, shape, taps, synth.cu_seqlens(lengths))
    for key in ("a", "y"):
        np.testing.assert_allclose(out[key], ref[key], rtol=1e-12, atol=1e-12, err_msg=key)
    np.testing.assert_allclose(out["h_draft"], ref["h_draft"], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(out["z"], ref["z"], rtol=1e-12, atol=1e-12)
    # the test is sensitive: the MLP and the attention both move y at this scale
    assert np.max(np.abs(ref["y"] - ref["a"])) > 1e-2
    assert np.max(np.abs(ref["a"] - out["f"])) > 1e-2


# ---------------------------------------------------------------- whole forward
def _prefill(w, shape, lengths, seed=0, off=0, **kw):
    cu = synth.cu_seqlens(lengths)
    taps = _taps(shape, int(cu[-1]), seed, off)
    return O.predict_prefill(w, shape, taps, cu, **kw), taps, cu


def test_zero_out_projections_make_layer_identity():
    w = dict(_weights())
    w["w_o"] = np.zeros_like(w["w_o"])
    w["w_down"] = np.zeros_like(w["w_down"])
    out, _, _ = _prefill(w, SMALL, [3, 5])
    np.testing.assert_array_equal(out["y"], out["f"])


def test_causal_prefix_invariance():
    w = _weights()
    out, taps, cu = _prefill(w, SMALL, [9], all_tokens=True)
    for kpos in (0, 3, 8):
        trunc = O.predict_prefill(w, SMALL, [t[:kpos + 1] for t in taps], np.array([0, kpos + 1]))
        assert trunc["z"][0] == pytest.approx(out["z"][kpos], rel=1e-12, abs=1e-12)


def test_batch_permutation_and_padding_invariance():
    w = _weights()
    lengths = [4, 7, 2]
    out, taps, cu = _prefill(w, SMALL, lengths)
    perm = [2, 0, 1]
    ptaps = [np.concatenate([t[cu[b]:cu[b + 1]] for b in perm]) for t in taps]
    pout = O.predict_prefill(w, SMALL, ptaps, synth.cu_seqlens([lengths[b] for b in perm]))
    np.testing.assert_allclose(pout["z"], out["z"][perm], rtol=1e-12, atol=1e-12)
    # an extra sequence in the pack changes nothing for the others
    extra = _taps(SMALL, 5, seed=3)
    xtaps = [np.concatenate([t, e]) for t, e in zip(taps, extra)]
    xout = O.predict_prefill(w, SMALL, xtaps, synth.cu_seqlens(lengths + [5]))
    np.testing.assert_allclose(xout["z"][:3], out["z"], rtol=1e-12, atol=1e-12)


def test_prefill_equals_prefix_then_steps():
    w = _weights()
    lengths = [6, 4]
    full, taps, cu = _prefill(w, SMALL, lengths, all_tokens=True)
    kpre = [2, 1]
    pre_taps = [np.concatenate([t[cu[b]:cu[b] + kpre[b]] for b in range(2)]) for t in taps]
    pre_cu = synth.cu_seqlens(kpre)
    pre = O.predict_prefill(w, SMALL, pre_taps, pre_cu)
    caches = O.caches_from_prefill(pre, pre_cu)
    for step in range(3):
        rows = [cu[b] + kpre[b] + step for b in range(2)]
        st = O.predict_step(w, SMALL, [t[rows] for t in taps], caches)
        np.testing.assert_allclose(st["z"], full["z"][rows], rtol=1e-11, atol=1e-11)
        caches = st["caches"]


def test_static_prediction_reads_only_the_last_rows_past_the_keys_and_values():
    """The evaluation order of the library's static prediction: keys and
    values of every prompt row, then queries, attention, O, the MLP, the final
    norm and the head for each prompt's last row only.  In the oracle that is
    a step of the last row over the K/V cache of the rows before it; it gives
    the whole-layer prediction (the prompt of length 1 has an empty cache)."""
    w = _weights()
    lengths = [6, 4, 1, 9]
    full, taps, cu = _prefill(w, SMALL, lengths)
    kpre = [L - 1 for L in lengths]
    caches = []
    for b, L in enumerate(lengths):
        if L > 1:
            sub = [t[cu[b]:cu[b] + L - 1] for t in taps]
            caches += O.caches_from_prefill(O.predict_prefill(w, SMALL, sub, np.array([0, L - 1])), [0, L - 1])
        else:
            kh = np.zeros((0, SMALL.n_kv_heads, SMALL.head_dim))
            caches.append((kh, kh.copy()))
    last = [cu[b] + kpre[b] for b in range(len(lengths))]
    st = O.predict_step(w, SMALL, [t[last] for t in taps], caches)
    np.testing.assert_allclose(st["z"], full["z"], rtol=1e-11, atol=1e-11)
    np.testing.assert_allclose(st["h_draft"], full["h_draft"], rtol=1e-11, atol=1e-11)


def test_sampled_rows_equal_full_batch():
    w = _weights()
    lengths = [5, 2, 7, 1]
    out, taps, cu = _prefill(w, SMALL, lengths)
    sub = O.sample_prefill_rows(w, SMALL, taps, cu, [3, 1])
    np.testing.assert_allclose(sub["z"], out["z"][[3, 1]], rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------- generator
def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    x = np.random.default_rng(14).standard_normal(10000).astype(np.float32) * 3
    ours = synth.round_bf16(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(ours, ref)
    bits = synth.bf16_bits(ours)
    back = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(back, ours)


def test_generator_is_seeded_and_shaped():
    a = synth.lengths_8b_prefill(0)
    assert len(a) == 64 and a.min() >= 16 and a.max() <= 2048
    np.testing.assert_array_equal(a, synth.lengths_8b_prefill(0))
    c = synth.lengths_8b_step_cache(0)
    assert len(c) == 256 and c.min() >= 1 and c.max() <= 4096
    s = synth.lengths_sweep(0)
    assert len(s) == 1024 and s.max() <= 8192
    cu = synth.cu_seqlens([3, 4])
    assert cu.tolist() == [0, 3, 7] and cu.dtype == np.int32


# ---------------------------------------------------------------- gated attention (Sec. 4.1)
def _gated_weights(shape=SMALL, seed=0):
    return synth.make_weights(shape, seed, gated=True)


def test_sigmoid_against_library_expit():
    scipy_special = pytest.importorskip("scipy.special")
    x = np.linspace(-40, 40, 161)
    np.testing.assert_allclose(O.sigmoid(x), scipy_special.expit(x), rtol=1e-13, atol=1e-300)


def test_zero_gate_weights_halve_the_attention_output():
    """W_ag = 0 gives sigmoid(0) = 1/2 on every element: the gated layer equals
    the ungated layer with W_o scaled by 1/2 (linearity of the output projection)."""
    w = dict(_gated_weights())
    w["w_attn_gate"] = np.zeros_like(w["w_attn_gate"])
    gated, _, _ = _prefill(w, SMALL, [5, 3])
    w2 = {k: v for k, v in w.items() if k != "w_attn_gate"}
    w2["w_o"] = w["w_o"] * 0.5
    plain, _, _ = _prefill(w2, SMALL, [5, 3])
    np.testing.assert_allclose(gated["y"], plain["y"], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(gated["z"], plain["z"], rtol=1e-12, atol=1e-12)


def test_gate_brute_force_elementwise():
    """attn[r, c] = o[r, c] / (1 + exp(-sum_j x_hat[r, j] W_ag[c, j])), element by element."""
    w = _gated_weights()
    w2 = {k: v for k, v in w.items() if k != "w_attn_gate"}
    gated, _, _ = _prefill(w, SMALL, [4, 3])
    plain, _, _ = _prefill(w2, SMALL, [4, 3])
    x, o, W = gated["x"], plain["attn"], w["w_attn_gate"].astype(np.float64)
    ref = np.empty_like(o)
    for r in range(o.shape[0]):
        for c in range(o.shape[1]):
            acc = 0.0
            for j in range(x.shape[1]):
                acc += float(x[r, j]) * float(W[c, j])
            ref[r, c] = o[r, c] / (1.0 + math.exp(-acc))
    np.testing.assert_allclose(gated["attn"], ref, rtol=1e-12, atol=1e-14)


def test_gate_is_elementwise_per_output_column():
    """Changing one row of W_ag changes only that column of the gated output."""
    w = dict(_gated_weights())
    base, _, _ = _prefill(w, SMALL, [6])
    col = 5
    w["w_attn_gate"] = w["w_attn_gate"].copy()
    w["w_attn_gate"][col] += 0.5
    moved, _, _ = _prefill(w, SMALL, [6])
    diff = np.abs(moved["attn"] - base["attn"]).max(axis=0)
    assert diff[col] > 0
    assert np.all(np.delete(diff, col) == 0)


def test_gated_prefill_equals_prefix_then_steps():
    w = _gated_weights()
    lengths = [5, 3]
    full, taps, cu = _prefill(w, SMALL, lengths, all_tokens=True)
    kpre = [2, 1]
    pre_taps = [np.concatenate([t[cu[b]:cu[b] + kpre[b]] for b in range(2)]) for t in taps]
    pre_cu = synth.cu_seqlens(kpre)
    caches = O.caches_from_prefill(O.predict_prefill(w, SMALL, pre_taps, pre_cu), pre_cu)
    for step in range(2):
        rows = [cu[b] + kpre[b] + step for b in range(2)]
        st = O.predict_step(w, SMALL, [t[rows] for t in taps], caches)
        np.testing.assert_allclose(st["z"], full["z"][rows], rtol=1e-11, atol=1e-11)
        caches = st["caches"]


def test_default_weights_have_no_gate():
    w = synth.make_weights(SMALL, 0)
    wg = synth.make_weights(SMALL, 0, gated=True)
    assert "w_attn_gate" not in w
    for k in w:
        np.testing.assert_array_equal(w[k], wg[k])


# ---------------------------------------------------------------- dual head, draft branch (Eq. 2)
def _draft_case(V=37, rows=5, seed=3):
    rng = np.random.default_rng(seed)
    h = rng.standard_normal((rows, SMALL.d))
    w_lm = rng.standard_normal((V, SMALL.d)) * 0.2
    return h, w_lm


def test_draft_softmax_is_a_distribution():
    h, w_lm = _draft_case()
    out = O.draft_head(h, w_lm, 4)
    np.testing.assert_allclose(np.exp(out["logprob"]).sum(axis=1), 1.0, rtol=0, atol=1e-12)
    assert np.all(out["logprob"] <= 0.0)


def test_draft_logsumexp_and_log_softmax_match_library():
    special = pytest.importorskip("scipy.special")
    rng = np.random.default_rng(4)
    logits = rng.standard_normal((6, 1000)) * 30.0  # large spread: the max shift matters
    logp, lse = O.log_softmax_rows(logits)
    np.testing.assert_allclose(lse, special.logsumexp(logits, axis=1), rtol=1e-13)
    np.testing.assert_allclose(logp, special.log_softmax(logits, axis=1), rtol=1e-12, atol=1e-12)


def test_draft_permutation_head_closed_form():
    """W_lm = a permutation matrix (V = d): logit v = h[perm[v]] exactly; a
    transposed operand would give h[perm^-1[v]] instead."""
    rng = np.random.default_rng(5)
    d = SMALL.d
    perm = rng.permutation(d)
    assert np.any(perm[perm] != np.arange(d))  # not an involution, so P != P^T
    w_lm = np.zeros((d, d))
    w_lm[np.arange(d), perm] = 1.0
    h = rng.standard_normal((3, d))
    out = O.draft_head(h, w_lm, 5)
    np.testing.assert_array_equal(out["logits"], h[:, perm])
    for r in range(3):
        vals = list(h[r, perm])
        expect = []
        for _ in range(5):  # brute force: repeatedly take the largest remaining
            best = max(range(d), key=lambda v: (vals[v], -v) if v not in expect else (-np.inf, 0))
            expect.append(best)
        assert list(out["topk_ids"][r]) == expect


def test_draft_zero_head_is_uniform_and_ties_go_to_smaller_ids():
    V = 50
    out = O.draft_head(np.ones((2, SMALL.d)), np.zeros((V, SMALL.d)), 6)
    np.testing.assert_allclose(out["logprob"], -math.log(V), rtol=0, atol=1e-14)
    np.testing.assert_allclose(out["lse"], math.log(V), rtol=1e-15)
    assert out["topk_ids"].tolist() == [list(range(6))] * 2


def test_draft_topk_brute_force_with_planted_ties():
    logits = np.array([[0.5, 2.0, -1.0, 2.0, 0.5, 3.0, 2.0, -4.0, 0.5, 3.0, 1.0]])
    ids = O.top_k_tokens(logits, 7)
    rows = sorted(range(logits.shape[1]), key=lambda v: (-logits[0, v], v))
    assert ids[0].tolist() == rows[:7] == [5, 9, 1, 3, 6, 10, 0]


def test_draft_row_shift_invariance():
    """Adding the same vector u to every row of W_lm adds h.u to every logit of
    the row: log-probabilities and top-k are unchanged, logsumexp moves by h.u."""
    h, w_lm = _draft_case()
    u = np.random.default_rng(6).standard_normal(SMALL.d)
    a = O.draft_head(h, w_lm, 5)
    b = O.draft_head(h, w_lm + u[None, :], 5)
    np.testing.assert_allclose(b["logprob"], a["logprob"], rtol=0, atol=1e-10)
    np.testing.assert_allclose(b["lse"], a["lse"] + h @ u, rtol=0, atol=1e-10)
    np.testing.assert_array_equal(b["topk_ids"], a["topk_ids"])


def test_dual_head_reads_the_length_heads_state():
    """Both branches of the dual head read the same h^draft (Sec. 4.2): the
    draft output of a prediction is the draft head of its h_draft, and asking
    for it changes nothing else."""
    w = _weights()
    w["w_lm"] = synth.make_lm_head(SMALL, 29, 0)
    cu = synth.cu_seqlens([4, 7])
    taps = _taps(SMALL, 11)
    plain = O.predict_prefill(w, SMALL, taps, cu)
    dual = O.predict_prefill(w, SMALL, taps, cu, draft_k=3)
    np.testing.assert_array_equal(dual["z"], plain["z"])
    ref = O.draft_head(plain["h_draft"], w["w_lm"], 3)
    np.testing.assert_array_equal(dual["draft"]["topk_ids"], ref["topk_ids"])
    np.testing.assert_array_equal(dual["draft"]["lse"], ref["lse"])


def test_lm_head_draw_leaves_other_weights_unchanged():
    a = synth.make_weights(SMALL, 0)
    w1 = synth.make_lm_head(SMALL, 40, 0)
    b = synth.make_weights(SMALL, 0)
    for k in a:
        np.testing.assert_array_equal(a[k], b[k])
    np.testing.assert_array_equal(w1, synth.make_lm_head(SMALL, 40, 0))
    assert w1.shape == (40, SMALL.d) and abs(float(w1.std()) - 0.02) < 0.004


# ---------------------------------------------------------------- input-embedding branch (Sec. 5.4)
EV = 40  # embedding rows of the pin cases


def _embed_case(lengths=(5, 3), gated=False, seed=0, off=0):
    w = synth.make_weights(SMALL, seed, gated=gated, embed_vocab=EV)
    cu = synth.cu_seqlens(list(lengths))
    T = int(cu[-1])
    return w, cu, _taps(SMALL, T, seed, off), synth.make_tokens(T, EV, seed, off)


def test_embedding_columns_zero_reduce_to_the_plain_layer():
    """With the embedding columns of W_q, W_k, W_v (and W_ag) set to zero the
    branch contributes nothing: every output equals the layer without it."""
    for gated in (False, True):
        w, cu, taps, tok = _embed_case(gated=gated)
        d = SMALL.d
        for name in ("w_q", "w_k", "w_v") + (("w_attn_gate",) if gated else ()):
            w[name] = w[name].copy()
            w[name][:, :d] = 0.0
        plain = synth.make_weights(SMALL, 0, gated=gated)
        a = O.predict_prefill(w, SMALL, taps, cu, tokens=tok)
        b = O.predict_prefill(plain, SMALL, taps, cu)
        np.testing.assert_allclose(a["y"], b["y"], rtol=0, atol=1e-13)
        np.testing.assert_allclose(a["z"], b["z"], rtol=0, atol=1e-13)


def test_embedding_is_a_row_lookup():
    """Permuting the table rows and relabelling the tokens the same way changes nothing."""
    w, cu, taps, tok = _embed_case()
    perm = np.random.default_rng(8).permutation(EV)
    w2 = dict(w)
    w2["w_embed"] = w["w_embed"][perm]          # new row r holds old row perm[r]
    inv = np.argsort(perm)                       # old token t sits at new row inv[t]
    a = O.predict_prefill(w, SMALL, taps, cu, tokens=tok)
    b = O.predict_prefill(w2, SMALL, taps, cu, tokens=inv[tok])
    np.testing.assert_array_equal(a["z"], b["z"])
    np.testing.assert_array_equal(a["x"], b["x"])


def test_embedding_layer_input_brute_force():
    """q of one row by explicit loops: the normalized embedding fills input
    columns 0..d-1, the normalized fused feature columns d..2d-1."""
    w, cu, taps, tok = _embed_case(lengths=(4,))
    out = O.predict_prefill(w, SMALL, taps, cu, tokens=tok)
    d, r, eps = SMALL.d, 2, SMALL.rms_eps
    e = [float(v) for v in w["w_embed"][tok[r]]]
    f = [sum(float(taps[j][r, i]) * float(w["w_proj"][c, j * d + i]) for j in range(3) for i in range(d))
         for c in range(d)]
    re = math.sqrt(sum(v * v for v in e) / d + eps)
    rf = math.sqrt(sum(v * v for v in f) / d + eps)
    x = [e[i] / re * float(w["g_emb"][i]) for i in range(d)] + [f[i] / rf * float(w["g_in"][i]) for i in range(d)]
    q = [sum(float(w["w_q"][j, i]) * x[i] for i in range(2 * d)) for j in range(SMALL.n_heads * SMALL.head_dim)]
    # the oracle's layer input (the rotation comes after the projection, so compare before it)
    np.testing.assert_allclose(out["x"][r], x, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(out["x"][r] @ w["w_q"].astype(np.float64).T, q, rtol=1e-11, atol=1e-12)


def test_embedding_token_change_is_causal():
    """Changing the token at position p of a sequence changes that sequence's
    outputs at positions >= p only, and no other sequence."""
    w, cu, taps, tok = _embed_case(lengths=(6, 4))
    a = O.predict_prefill(w, SMALL, taps, cu, all_tokens=True, tokens=tok)
    tok2 = tok.copy()
    tok2[3] = (tok2[3] + 1) % EV
    b = O.predict_prefill(w, SMALL, taps, cu, all_tokens=True, tokens=tok2)
    diff = np.abs(a["y"] - b["y"]).max(axis=1)
    assert np.all(diff[:3] == 0) and np.all(diff[3:6] > 0) and np.all(diff[6:] == 0)


def test_embedding_prefill_equals_prefix_then_steps():
    w, cu, taps, tok = _embed_case(lengths=(5, 3), gated=True)
    full = O.predict_prefill(w, SMALL, taps, cu, all_tokens=True, tokens=tok)
    kpre = [2, 1]
    pre_rows = np.concatenate([np.arange(cu[b], cu[b] + kpre[b]) for b in range(2)])
    pre_cu = synth.cu_seqlens(kpre)
    caches = O.caches_from_prefill(
        O.predict_prefill(w, SMALL, [t[pre_rows] for t in taps], pre_cu, tokens=tok[pre_rows]), pre_cu)
    for step in range(2):
        rows = [cu[b] + kpre[b] + step for b in range(2)]
        st = O.predict_step(w, SMALL, [t[rows] for t in taps], caches, tokens=tok[rows])
        np.testing.assert_allclose(st["z"], full["z"][rows], rtol=1e-11, atol=1e-11)
        caches = st["caches"]


def test_embedding_draw_keeps_the_fused_feature_columns():
    w = synth.make_weights(SMALL, 0, gated=True, embed_vocab=EV)
    p = synth.make_weights(SMALL, 0, gated=True)
    d = SMALL.d
    for name in ("w_q", "w_k", "w_v", "w_attn_gate"):
        assert w[name].shape == (p[name].shape[0], 2 * d)
        np.testing.assert_array_equal(w[name][:, d:], p[name])
    for name in p:
        if name not in ("w_q", "w_k", "w_v", "w_attn_gate"):
            np.testing.assert_array_equal(w[name], p[name])


# ---------------------------------------------------------------- draft rollouts
def test_draft_step_with_the_fused_feature_is_a_normal_step():
    """Feeding f_ctx itself as the feature input reproduces the tapped step."""
    w, cu, taps, tok = _embed_case(lengths=(4, 6))
    caches = O.caches_from_prefill(O.predict_prefill(w, SMALL, taps, cu, tokens=tok), cu)
    st = _taps(SMALL, 2, 0, 9)
    stok = synth.make_tokens(2, EV, 0, 9)
    a = O.predict_step(w, SMALL, st, caches, tokens=stok)
    b = O.predict_step(w, SMALL, None, caches, tokens=stok, f_rows=O.fuse_taps(st, w["w_proj"]))
    np.testing.assert_array_equal(a["z"], b["z"])
    np.testing.assert_array_equal(a["caches"][1][0], b["caches"][1][0])


def test_rollout_then_rollback_equals_never_drafting():
    """Two draft positions appended and dropped again (the target rejected
    them): the next tapped step sees exactly the cache it would have seen."""
    w, cu, taps, tok = _embed_case(lengths=(5, 3))
    caches = O.caches_from_prefill(O.predict_prefill(w, SMALL, taps, cu, tokens=tok), cu)
    st = _taps(SMALL, 2, 0, 11)
    s1 = O.predict_step(w, SMALL, st, caches, tokens=synth.make_tokens(2, EV, 0, 11))
    d1 = O.predict_step(w, SMALL, None, s1["caches"], tokens=synth.make_tokens(2, EV, 0, 12), f_rows=s1["y"])
    d2 = O.predict_step(w, SMALL, None, d1["caches"], tokens=synth.make_tokens(2, EV, 0, 13), f_rows=d1["y"])
    assert d2["caches"][0][0].shape[0] == s1["caches"][0][0].shape[0] + 2
    rolled = [(k[:-2], v[:-2]) for k, v in d2["caches"]]
    for (ka, va), (kb, vb) in zip(rolled, s1["caches"]):
        np.testing.assert_array_equal(ka, kb)
        np.testing.assert_array_equal(va, vb)
    nxt = _taps(SMALL, 2, 0, 14)
    t2 = synth.make_tokens(2, EV, 0, 14)
    np.testing.assert_array_equal(O.predict_step(w, SMALL, nxt, rolled, tokens=t2)["z"],
                                  O.predict_step(w, SMALL, nxt, s1["caches"], tokens=t2)["z"])
