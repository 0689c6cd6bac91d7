"""Pins of the App. A graph statement and the App. C cost model.

  * Theorem 1 is checked by brute force over every layer-shared mask on
    {LT, X, R} in which LT attends X (and shown non-vacuous);
  * the oracle's own block tables are run through the same reachability: the
    paper's beyond mask and the isolated cache are StructCacheable, full
    attention is not, and only the beyond mask carries the instruction to R;
  * the cost model reproduces the one number App. C prints (0.87 x), satisfies
    its monotonicity and ceiling statements, the anchor-overhead identity and
    the printed derivative.
"""
import json
import os

import numpy as np
import pytest

from oracle import cost_model as cm
from oracle import structure as st

GOLD = os.path.join(os.path.dirname(__file__), "golden")


@pytest.mark.parametrize("depth", [2, 3, 4])
def test_theorem_1_by_exhaustion(depth):
    blocks = ("LT", "X", "R")
    n_masks = both = cache_only = reach_only = 0
    for m in st.all_masks(blocks):
        if not m[("LT", "X")]:
            continue
        n_masks += 1
        att = lambda q, k, m=m: m[(q, k)]
        c = st.struct_cacheable(blocks, att, depth)
        r = st.live_text_reachable(blocks, att, depth)
        both += c and r
        cache_only += c and not r
        reach_only += r and not c
    assert n_masks == 256
    assert both == 0
    assert cache_only > 0 and reach_only > 0


def test_theorem_needs_depth_two():
    """With L = 1 LiveTextReachable is void (needs l < m), so the theorem's L >= 2 matters."""
    att = lambda q, k: True
    assert not st.live_text_reachable(("LT", "X", "R"), att, 1)


@pytest.mark.parametrize("depth", [2, 5])
def test_oracle_block_tables_under_app_a(oracle_mod, depth):
    blocks = ("LT", "X", "ST", "R")

    def att(mode):
        return lambda q, k: oracle_mod.block_visible(mode, q, k)

    for mode in ("beyond", "beyond_alt", "isolated"):
        assert st.struct_cacheable(blocks, att(mode), depth), mode
        assert not st.live_text_reachable(blocks, att(mode), depth), mode
    assert not st.struct_cacheable(blocks, att("full"), depth)
    assert st.instruction_reaches_reference(blocks, att("beyond"), depth)
    assert st.instruction_reaches_reference(blocks, att("beyond_alt"), depth)
    assert not st.instruction_reaches_reference(blocks, att("isolated"), depth)


def test_asymptotic_one_reference_printed_value():
    g = json.load(open(os.path.join(GOLD, "cost_model_app_c.json")))["asymptotic_one_reference"]
    r = cm.speedup_asymptotic(g["n_r"], g["s"], g["T"])
    assert round(r, g["printed_decimals"]) == g["printed"]


def test_anchor_overhead_is_prefill_difference():
    for n_r in (256, 4096, 20480, 40960):
        for n_st in (0, 32, 64, 128, 512):
            assert cm.anchor_overhead(n_r, n_st) == cm.c_pre(n_r, n_st) - cm.c_pre(n_r, 0)


def test_speedup_forms_agree_and_monotone_below_ceiling():
    T, S = 40, 4608
    for n_st in (0, 128, 512, S):
        prev = 0.0
        for n_r in range(0, 200_001, 1024):
            r = cm.speedup(n_r, n_st, S, T)
            u = n_r + S
            assert r == pytest.approx(cm.speedup_of_u(u, n_st, S, T), rel=1e-12)
            assert r < T
            assert r > prev
            prev = r
            d = cm.speedup_derivative_u(u, n_st, S, T)
            assert d > 0
            h = 1e-3 * u
            fd = (cm.speedup_of_u(u + h, n_st, S, T) - cm.speedup_of_u(u - h, n_st, S, T)) / (2 * h)
            assert d == pytest.approx(fd, rel=1e-5)


def test_speedup_tends_to_T():
    assert cm.speedup(1e12, 128, 4608, 40) == pytest.approx(40, rel=1e-6)


def test_flops_per_unit():
    assert cm.flops_per_unit(128) == 512 and cm.flops_per_unit(64) == 256
