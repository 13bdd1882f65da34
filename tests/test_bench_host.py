"""Host logic of bench.py that its figures rest on: which measured bf16 peak
a tensor fraction is taken against, and the algorithmic FLOP counts of a
static prediction (dense products and the causal attention), each checked
against an independent count."""
import os
import sys

import numpy as np

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402
from paper_2609_01068_gb300 import synth  # noqa: E402

PEAKS = {"hbm_gbs": 6698.5, "bf16": 1950.6, "bf16_sus": 1749.7, "src": "of measured"}


def test_tensor_peak_burst_for_a_short_region_at_full_clock():
    peak, kind = bench.tensor_peak(PEAKS, 300.0, {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []})
    assert peak == PEAKS["bf16"] and kind.startswith("bf16 burst")
    # the power cap flagged while the clock held its maximum: still the burst figure, noted
    peak, kind = bench.tensor_peak(PEAKS, 300.0, {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0,
                                                  "reasons": ["sw_power_cap"]})
    assert peak == PEAKS["bf16"] and "power cap" in kind


def test_tensor_peak_sustained_when_capped_below_max_or_long():
    peak, kind = bench.tensor_peak(PEAKS, 300.0, {"sm_mhz": 1785.0, "sm_max_mhz": 2070.0,
                                                  "reasons": ["sw_power_cap"]})
    assert peak == PEAKS["bf16_sus"] and kind.startswith("bf16 sustained")
    peak, _ = bench.tensor_peak(PEAKS, 2500.0, {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []})
    assert peak == PEAKS["bf16_sus"]


def _causal_pairs(lengths):
    """(query, key) pairs a causal mask keeps, counted one query at a time."""
    n = 0
    for L in lengths:
        for i in range(int(L)):
            n += sum(1 for k in range(int(L)) if k <= i)
    return n


def test_attention_flops_count_causal_pairs():
    rng = np.random.default_rng(3)
    lengths = rng.integers(1, 90, size=7)
    shape = synth.TINY
    r = bench.attention_roofline(shape, lengths, 1.0, PEAKS)
    # QK^T and PV: hd multiply-adds each per kept pair and head
    assert r["flop_per_pass"] == 2 * 2 * shape.head_dim * shape.n_heads * _causal_pairs(lengths)
    assert abs(r["achieved"] - r["flop_per_pass"] / 1e-3 / 1e12) < 1e-12 * max(1.0, r["achieved"])
    assert abs(r["frac_of_burst"] - r["achieved"] / PEAKS["bf16"]) < 1e-15


def _layer_products(shape, gated=False):
    """(N, K) of each per-row matrix product of the draft layer, written out one by one."""
    d, H, KVH, hd, F = shape.d, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn
    prods = [(d, 3 * d),           # FC over the three taps (Eq. 1)
             (H * hd, d),          # q
             (KVH * hd, d),        # k
             (KVH * hd, d),        # v
             (d, H * hd),          # O
             (F, d), (F, d),       # gate, up
             (d, F)]               # down
    if gated:
        prods.append((H * hd, d))  # attention gate
    return prods


def test_whole_layer_flops_match_enumerated_products():
    rng = np.random.default_rng(5)
    lengths = rng.integers(1, 50, size=5)
    for shape in (synth.TINY, synth.LLAMA8B):
        T = int(lengths.sum())
        B = len(lengths)
        dense = sum(2 * T * n * k for n, k in _layer_products(shape))
        widths = (shape.d,) + tuple(shape.head_widths) + (1,)
        head = sum(2 * B * widths[i] * widths[i + 1] for i in range(len(widths) - 1))
        attn = 4 * shape.n_heads * shape.head_dim * _causal_pairs(lengths)
        got = bench.prefill_flops(shape, lengths, B, whole_layer=True)
        assert abs(got - (dense + attn + head)) <= 1e-9 * got, shape.name


def test_pruned_prefill_flops_match_enumerated_products():
    """Keys and values for every row, the rest for the last row of each prompt
    (one query against its prompt's keys)."""
    rng = np.random.default_rng(9)
    lengths = rng.integers(1, 50, size=6)
    shape = synth.LLAMA8B
    T = int(lengths.sum())
    B = len(lengths)
    d, H, KVH, hd, F = shape.d, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn
    every_row = 2 * T * (d * 3 * d + 2 * KVH * hd * d)
    last_rows = 2 * B * (H * hd * d + d * H * hd + 2 * F * d + d * F)
    widths = (d,) + tuple(shape.head_widths) + (1,)
    head = sum(2 * B * widths[i] * widths[i + 1] for i in range(len(widths) - 1))
    attn = 4 * H * hd * int(lengths.sum())  # each last row against all keys of its prompt
    got = bench.prefill_flops(shape, lengths, B, whole_layer=False)
    assert abs(got - (every_row + last_rows + head + attn)) <= 1e-9 * got
