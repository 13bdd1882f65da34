"""CPU oracle for the serving-side use of the static prediction.  TEST INFRASTRUCTURE ONLY.

Only the tests and bench.py's reference leg may import this module; the
library never calls it and shares no code with it.

Sec. 5.3 (and the appendix "System-Level Evaluation Details") compares, on a
disaggregated deployment with one prefill and three decode instances, two
decisions taken with the static prediction r_hat_0 as a proxy for decode cost:

  instance routing   RR: decode instances in a fixed cyclic order;
                     LB: the decode instance with the lowest estimated
                         remaining workload, summed over the predicted
                         remaining lengths of its queued and running requests;
  queue order        FCFS: arrival order;
                     SJF: shorter predicted generation first.

The paper runs these inside vLLM and prints no simulator.  This module is a
plain discrete-event model of that setting, written from the description; its
readings (kept in the design notes) are:

  * prefill: one instance, requests served one at a time in arrival order
    (ties: smaller id), service time pf_base + pf_per_token * prompt_len;
  * decode: continuous batching; an instance runs steps that give every
    running request one token; a step with running set R lasts
    step_base + step_per_seq * |R| + step_per_kv * sum_{r in R} (prompt_r + generated_r);
    at a step boundary finished requests leave (finish time = boundary),
    then waiting requests are admitted (FCFS or SJF key) while fewer than
    max_running run, then the next step starts; an idle instance starts at
    once when a request arrives; no preemption;
  * a request needs output_len decode tokens (>= 1);
  * LB cost of a request: ceil(r_hat) tokens, remaining = max(ceil(r_hat) -
    generated, 0) for running ones (as of the instance's last step
    boundary); ties go to the lower instance index; RR counts requests in
    order of reaching the decode tier;
  * SJF key (ceil(r_hat), decode arrival time, id); FCFS key (decode arrival
    time, id);
  * simultaneous events: step ends before arrivals, lower instance first.

Everything is plain Python floats (IEEE double) and ints.
"""
from __future__ import annotations

import math

RR, LB = 0, 1
FCFS, SJF = 0, 1


def prefill_finish_times(arrival, prompt, pf_base, pf_per_token):
    """One prefill instance, FCFS: finish_i = max(arrival_i, previous finish) + service_i."""
    order = sorted(range(len(arrival)), key=lambda i: (arrival[i], i))
    fin = [0.0] * len(arrival)
    t = -math.inf
    for i in order:
        start = arrival[i] if arrival[i] > t else t
        t = start + (pf_base + pf_per_token * prompt[i])
        fin[i] = t
    return fin, order


def simulate(cfg, arrival, prompt, output, predicted):
    """Returns (finish time, decode instance) of every request.

    cfg: dict with n_decode, max_running, pf_base, pf_per_token, step_base,
    step_per_seq, step_per_kv, route (RR / LB), order (FCFS / SJF).
    """
    n = len(arrival)
    cost = [int(math.ceil(p)) for p in predicted]
    ready, order = prefill_finish_times(arrival, prompt, cfg["pf_base"], cfg["pf_per_token"])
    arrivals = sorted(range(n), key=lambda i: (ready[i], i))  # reaching the decode tier
    nd = cfg["n_decode"]
    running = [[] for _ in range(nd)]   # request ids, in admission order
    waiting = [[] for _ in range(nd)]
    gen = [0] * n
    step_end = [None] * nd              # None: idle
    finish = [0.0] * n
    inst = [-1] * n
    rr = 0

    def key(i):
        return (cost[i], ready[i], i) if cfg["order"] == SJF else (ready[i], i)

    def start_step(j, t):
        # admit, then start a step if anything runs
        while waiting[j] and len(running[j]) < cfg["max_running"]:
            best = min(waiting[j], key=key)
            waiting[j].remove(best)
            running[j].append(best)
        if running[j]:
            kv = 0
            for r in running[j]:
                kv += prompt[r] + gen[r]
            dt = cfg["step_base"] + cfg["step_per_seq"] * len(running[j]) + cfg["step_per_kv"] * kv
            step_end[j] = t + dt
        else:
            step_end[j] = None

    a = 0
    while True:
        # next event: the earliest step end (lower instance on ties), else the next arrival
        j_next, t_next = -1, math.inf
        for j in range(nd):
            if step_end[j] is not None and step_end[j] < t_next:
                j_next, t_next = j, step_end[j]
        if a < n and ready[arrivals[a]] < t_next:
            i = arrivals[a]
            a += 1
            t = ready[i]
            if cfg["route"] == RR:
                j = rr % nd
                rr += 1
            else:
                loads = []
                for j2 in range(nd):
                    w = 0
                    for r in running[j2]:
                        w += max(cost[r] - gen[r], 0)
                    for q in waiting[j2]:
                        w += cost[q]
                    loads.append(w)
                j = min(range(nd), key=lambda j2: (loads[j2], j2))
            inst[i] = j
            waiting[j].append(i)
            if step_end[j] is None:
                start_step(j, t)
            continue
        if j_next < 0:
            break
        t = t_next
        still = []
        for r in running[j_next]:
            gen[r] += 1
            if gen[r] >= output[r]:
                finish[r] = t
            else:
                still.append(r)
        running[j_next] = still
        start_step(j_next, t)
    return finish, inst


def summarize(arrival, output, finish, short_below=800, long_from=1300):
    """Serving metrics of Sec. 5.3 and its appendix: throughput (output tokens / makespan), mean
    latency, and P99 latency of short / medium / long requests by true length
    (nearest-rank percentile)."""
    lat = [f - a for f, a in zip(finish, arrival)]
    span = max(finish) - min(arrival)

    def p99(xs):
        if not xs:
            return float("nan")
        xs = sorted(xs)
        return xs[max(0, math.ceil(0.99 * len(xs)) - 1)]

    cats = {"short": [], "medium": [], "long": []}
    for l, o in zip(lat, output):
        cats["short" if o < short_below else ("long" if o >= long_from else "medium")].append(l)
    return {"throughput_tok_s": sum(output) / span, "mean_latency_s": sum(lat) / len(lat),
            "p99_short_s": p99(cats["short"]), "p99_medium_s": p99(cats["medium"]),
            "p99_long_s": p99(cats["long"]), "n": len(lat)}
