"""Host logic: the accounting the benchmark reports against the App. C model,
and the seeded input generators."""
import pytest
import torch

import workloads
from oracle import cost_model as cm
from paper_2608_21229_gb300 import accounting as acc


@pytest.mark.parametrize("w", [workloads.TINY, workloads.EDIT_512_2REF, workloads.EDIT_1024_5REF]
                         + list(workloads.SWEEP_1024), ids=lambda w: w.name)
def test_accounting_equals_app_c_model(w):
    r = w.requests[0]
    s = r.n_lt + r.n_x
    assert acc.prefill_units(w.requests) == cm.c_pre(r.n_r, r.n_st)
    assert acc.step_units(w.requests) == cm.c_step(r.n_r, s)
    assert 40 * acc.full_units(w.requests) == cm.c_full(r.n_r, s, 40)
    assert acc.modelled_ratio(w.requests, 40) == pytest.approx(cm.speedup(r.n_r, r.n_st, s, 40), rel=1e-12)
    assert acc.flops(1, 24, 128) == cm.flops_per_unit(128) * 24
    assert acc.prefill_units(w.requests) - acc.prefill_units(
        [workloads.Request(0, r.n_lt, r.n_x, r.n_r)]) == cm.anchor_overhead(r.n_r, r.n_st)


def test_headline_step_flops():
    w = workloads.EDIT_1024_5REF
    f = acc.flops(acc.step_units(w.requests), w.num_heads, w.head_dim)
    assert f == 4 * 128 * 24 * 4608 * (4608 + 20480)
    assert acc.cache_bytes(w.requests, 24, 128) == 2 * 20480 * 24 * 128 * 2


def test_generators_are_deterministic_and_distinct():
    a = workloads.randn_bf16((64, 2, 8), 0, "x")
    b = workloads.randn_bf16((64, 2, 8), 0, "x")
    c = workloads.randn_bf16((64, 2, 8), 0, "y")
    assert a.dtype == torch.bfloat16 and torch.equal(a, b) and not torch.equal(a, c)
    assert abs(float(workloads.randn_bf16((4096, 64), 1, "z").float().std()) - 1.0) < 0.02


def test_workload_shapes():
    w = workloads.RAGGED_4REQ
    assert w.batch == 4 and [r.n_r // 1024 if r.n_x == 1024 else r.n_r // 4096 for r in w.requests] == [1, 3, 5, 8]
    assert w.cu_live[-1] == sum(r.n_lt + r.n_x for r in w.requests)
    q, k, v = workloads.static_qkv(workloads.TINY)
    assert q.shape == (288, 4, 64)


def test_bench_clock_ceilings():
    """The bench line's two clock-based figures: the tensor pipe's ceiling
    (8192 dense bf16 FLOPs per clock per SM) and the exponential floor (one
    ex2 per visible pair at a given rate per clock per SM), at a given clock."""
    import bench

    n = bench.nominal_at_clock(1000.0, 2000.0, 152)
    assert n["tflops"] == pytest.approx(8192 * 152 * 2.0e9 / 1e12) and n["frac"] == pytest.approx(1000.0 / n["tflops"])
    assert bench.nominal_at_clock(1000.0, None, 152) is None
    w = workloads.EDIT_1024_5REF
    exps = acc.step_units(w.requests) * w.num_heads
    f = bench.exp_floor(exps, 1e-3, 2000.0, 152, 32.0)
    assert f["floor_ms"] == pytest.approx(exps / (32 * 152 * 2.0e9) * 1e3)
    assert f["frac_of_step"] == pytest.approx(f["floor_ms"] / 1.0)
    assert bench.exp_floor(exps, 1e-3, 2000.0, 152, 16.0)["floor_ms"] == pytest.approx(2 * f["floor_ms"])
    assert bench.exp_floor(exps, 1e-3, None, 152, 32.0) is None


def test_guard_report_finds_planted_writes():
    """The canary check of tests/test_gpu_canary.py: bytes changed in either
    guard and elements left unwritten are counted (planted on the CPU)."""
    import numpy as np
    import parity_utils as pu

    g, n, pat = 64, 40, 0xA5
    full = np.full(g + n + g, pat, dtype=np.uint8)
    full[g:g + n] = 1                      # every element written
    assert pu.guard_report(full, g, n, 4, pat) == (0, 0, 0)
    full[g - 1] = 0                        # one byte before the buffer
    full[g + n + 5] = 7                    # and one after
    full[g + 8:g + 12] = pat               # one 4-byte element never written
    assert pu.guard_report(full, g, n, 4, pat) == (1, 1, 1)
    full[g + 12] = pat                     # a partly matching element is written
    assert pu.guard_report(full, g, n, 4, pat)[2] == 1
    assert pu.guard_report(full, g, n, 2, pat)[2] == 2
