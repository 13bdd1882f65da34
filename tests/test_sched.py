"""Length-aware serving model (Sec. 5.3): oracle pins and the C++ model
(include/outlets_sched.h) against the oracle.  Host code only: these run on
the CPU.  The decisions (instance per request) and the event times are
compared exactly: both sides take the same IEEE double operations in the same
order and the LB loads are integers."""
import math
import os
import shutil

import numpy as np
import pytest

from oracle import sched_oracle as S
from paper_2609_01068_gb300 import synth

BASE = dict(n_decode=3, max_running=8, route=S.LB, order=S.SJF, pf_base=0.01, pf_per_token=2e-5,
            step_base=0.02, step_per_seq=2e-4, step_per_kv=1e-7)


def _lists(w):
    return ([float(x) for x in w["arrival"]], [int(x) for x in w["prompt"]], [int(x) for x in w["output"]],
            [float(x) for x in w["predicted"]])


# ---------------------------------------------------------------- oracle pins
def test_prefill_is_a_single_fcfs_server():
    arrival = [0.0, 0.0, 0.5, 10.0]
    prompt = [100, 50, 10, 0]
    fin, order = S.prefill_finish_times(arrival, prompt, 0.1, 0.01)
    # 0 then 1 back to back from t=0; 2 arrives while busy; 3 finds the server idle
    assert order == [0, 1, 2, 3]
    assert fin[0] == pytest.approx(1.1) and fin[1] == pytest.approx(1.7)
    assert fin[2] == pytest.approx(1.9) and fin[3] == pytest.approx(10.1)


def test_uncontended_request_closed_form():
    """One request alone: prefill, then output_len steps of one sequence whose
    context grows by one token per step (an arithmetic series)."""
    cfg = dict(BASE, n_decode=1)
    p, o = 300, 57
    fin, inst = S.simulate(cfg, [2.0], [p], [o], [40.0])
    pre = cfg["pf_base"] + cfg["pf_per_token"] * p
    dec = o * (cfg["step_base"] + cfg["step_per_seq"]) + cfg["step_per_kv"] * (o * p + o * (o - 1) / 2)
    assert fin[0] == pytest.approx(2.0 + pre + dec, rel=1e-12) and inst == [0]


def test_single_serial_server_closed_form():
    """max_running = 1, FCFS, no KV term, free prefill: requests are served
    back to back in arrival order, each for output_len steps."""
    cfg = dict(BASE, n_decode=1, max_running=1, order=S.FCFS, pf_base=0.0, pf_per_token=0.0, step_per_kv=0.0)
    arrival = [0.0, 0.1, 0.2, 5.0]
    output = [10, 3, 7, 2]
    fin, _ = S.simulate(cfg, arrival, [5] * 4, output, [1.0] * 4)
    step = cfg["step_base"] + cfg["step_per_seq"]
    t, expect = 0.0, []
    for a, o in zip(arrival, output):
        t = max(t, a) + o * step
        expect.append(t)
    np.testing.assert_allclose(fin, expect, rtol=1e-12)


def test_sjf_with_equal_predictions_is_fcfs():
    w = _lists(synth.make_serving_requests(120, 30.0, 1))
    flat = w[:3] + ([500.0] * 120,)
    a = S.simulate(dict(BASE, order=S.SJF), *flat)
    b = S.simulate(dict(BASE, order=S.FCFS), *flat)
    assert a == b


def test_sjf_serves_the_shortest_prediction_first():
    """One instance with one slot, everything arriving at t = 0: request 0
    finds the instance idle and starts at once (no preemption); the others
    wait and are served by ascending predicted cost ceil(r_hat), ties by lower
    index."""
    cfg = dict(BASE, n_decode=1, max_running=1, pf_base=0.0, pf_per_token=0.0)
    pred = [50.0, 3.0, 20.0, 3.0, 7.5]
    fin, _ = S.simulate(cfg, [0.0] * 5, [1] * 5, [4] * 5, pred)
    assert list(np.argsort(fin, kind="stable")) == [0, 1, 3, 4, 2]
    fin, _ = S.simulate(dict(cfg, order=S.FCFS), [0.0] * 5, [1] * 5, [4] * 5, pred)
    assert list(np.argsort(fin, kind="stable")) == [0, 1, 2, 3, 4]


def test_rr_routes_cyclically():
    w = _lists(synth.make_serving_requests(40, 10.0, 2))
    _, inst = S.simulate(dict(BASE, route=S.RR), *w)
    ready, _ = S.prefill_finish_times(w[0], w[1], BASE["pf_base"], BASE["pf_per_token"])
    order = sorted(range(40), key=lambda i: (ready[i], i))
    assert [inst[i] for i in order] == [k % 3 for k in range(40)]


def test_lb_hand_example():
    """All requests reach the decode tier at t = 0 (free prefill), before any
    step ends: LB sees only the queued predictions.  Loads after each request:
    [100,0,0] -> [100,10,0] -> [100,10,10] -> [100,20,10] -> [100,20,20]."""
    cfg = dict(BASE, pf_base=0.0, pf_per_token=0.0)
    _, inst = S.simulate(cfg, [0.0] * 5, [1] * 5, [5] * 5, [100.0, 10.0, 9.2, 10.0, 10.0])
    assert inst == [0, 1, 2, 1, 2]


def test_every_request_finishes_after_its_own_work():
    w = _lists(synth.make_serving_requests(200, 50.0, 3))
    for route in (S.RR, S.LB):
        for order in (S.FCFS, S.SJF):
            cfg = dict(BASE, route=route, order=order)
            fin, inst = S.simulate(cfg, *w)
            ready, _ = S.prefill_finish_times(w[0], w[1], cfg["pf_base"], cfg["pf_per_token"])
            for i in range(200):
                assert 0 <= inst[i] < 3
                assert fin[i] >= ready[i] + w[2][i] * (cfg["step_base"] + cfg["step_per_seq"]) - 1e-9


def test_p99_is_the_nearest_rank_percentile():
    rng = np.random.default_rng(5)
    lat = list(rng.exponential(3.0, 257))
    out = [100] * 257  # all short
    m = S.summarize([0.0] * 257, out, lat)
    assert m["p99_short_s"] == float(np.percentile(lat, 99, method="inverted_cdf"))


def test_sjf_with_exact_predictions_cuts_the_short_tail_under_load():
    """The effect Sec. 5.3 reports, in the model: at saturation, SJF with
    exact predictions lowers the P99 latency of short requests vs FCFS."""
    w = _lists(synth.make_serving_requests(600, 40.0, 4, pred_sigma=0.0))
    base = S.summarize(w[0], w[2], S.simulate(dict(BASE, route=S.RR, order=S.FCFS), *w)[0])
    sjf = S.summarize(w[0], w[2], S.simulate(dict(BASE, route=S.RR, order=S.SJF), *w)[0])
    assert sjf["p99_short_s"] < 0.8 * base["p99_short_s"]


# ---------------------------------------------------------------- C++ model vs oracle
@pytest.fixture(scope="module")
def lib():
    from paper_2609_01068_gb300 import build as B, outlets as O
    if not os.path.exists(B.LIB_PATH) and not shutil.which("nvcc") and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc unavailable and library not built")
    B.build()
    return O


CASES = [
    ("saturated", dict(), 400, 40.0, 0.5),
    ("light load", dict(), 150, 2.0, 0.5),
    ("exact predictions", dict(), 300, 40.0, 0.0),
    ("one slot", dict(max_running=1), 80, 5.0, 0.8),
    ("one instance", dict(n_decode=1), 150, 20.0, 0.5),
    ("no kv term", dict(step_per_kv=0.0), 200, 30.0, 0.5),
    ("large batch", dict(max_running=256, n_decode=4), 500, 80.0, 0.3),
]


@pytest.mark.parametrize("name,over,n,qps,sigma", CASES)
@pytest.mark.parametrize("route", [S.RR, S.LB])
@pytest.mark.parametrize("order", [S.FCFS, S.SJF])
def test_cpp_model_equals_oracle(lib, name, over, n, qps, sigma, route, order):
    w = synth.make_serving_requests(n, qps, 7, pred_sigma=sigma)
    cfg = dict(BASE, **over, route=route, order=order)
    fin, inst = lib.simulate_serving(cfg, w["arrival"], w["prompt"], w["output"], w["predicted"])
    rf, ri = S.simulate(cfg, *_lists(w))
    np.testing.assert_array_equal(inst, ri)
    np.testing.assert_array_equal(fin, rf)


def test_cpp_model_ties_and_simultaneous_events(lib):
    """Simultaneous arrivals, equal predictions, equal lengths: every tie rule is exercised."""
    n = 60
    arrival = np.repeat(np.arange(6, dtype=np.float64) * 0.05, 10)
    prompt = np.full(n, 64, np.int32)
    output = np.tile(np.array([1, 2, 3, 40, 40], np.int32), 12)
    pred = np.tile(np.array([2.0, 2.0, 0.5, 40.0, 39.2], np.float32), 12)
    for route in (S.RR, S.LB):
        for order in (S.FCFS, S.SJF):
            cfg = dict(BASE, route=route, order=order, pf_base=0.0, pf_per_token=0.0)
            fin, inst = lib.simulate_serving(cfg, arrival, prompt, output, pred)
            rf, ri = S.simulate(cfg, list(arrival), list(map(int, prompt)), list(map(int, output)),
                                [float(x) for x in pred])
            np.testing.assert_array_equal(inst, ri)
            np.testing.assert_array_equal(fin, rf)


def test_cpp_model_rejects_bad_arguments(lib):
    w = synth.make_serving_requests(5, 1.0, 0)
    bad = [dict(BASE, n_decode=0), dict(BASE, max_running=0), dict(BASE, route=2), dict(BASE, order=5),
           dict(BASE, step_base=-1.0), dict(BASE, pf_per_token=math.nan)]
    for cfg in bad:
        with pytest.raises(lib.OutletsError):
            lib.simulate_serving(cfg, w["arrival"], w["prompt"], w["output"], w["predicted"])
    out = w["output"].copy()
    out[2] = 0
    with pytest.raises(lib.OutletsError):
        lib.simulate_serving(BASE, w["arrival"], w["prompt"], out, w["predicted"])
    pred = w["predicted"].copy()
    pred[1] = -1.0
    with pytest.raises(lib.OutletsError):
        lib.simulate_serving(BASE, w["arrival"], w["prompt"], w["output"], pred)
    f, i = lib.simulate_serving(BASE, [], [], [], [])
    assert len(f) == 0 and len(i) == 0
