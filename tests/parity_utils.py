"""Helpers shared by the GPU parity tests: run a workload through the C ABI
(binding in paper_2608_21229_gb300.refcache) and through the CPU oracle on
the same seeded inputs, and compare."""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
import workloads
from paper_2608_21229_gb300 import refcache as rcb

MAX_ABS = 2e-2  # element-wise bound on |gpu - oracle| for unit-variance bf16 inputs
MEAN_ABS = 2e-3  # bound on the mean |gpu - oracle|
LSE_ABS = 2e-3  # bound on |lse_gpu - lse_oracle| (fp32 scores, natural log)


def bits(t: torch.Tensor) -> np.ndarray:
    return workloads.bf16_bits(t.cpu())


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().to(torch.float64).numpy()


class GpuRun:
    """One workload through the library: build of layer 0, one step, outputs on the CPU."""

    def __init__(self, w, mode="beyond", kernel="tcgen05", layer=0, step=0, num_layers=1, static=None, live=None,
                 device="cuda:0", scale=None):
        self.w, self.mode = w, mode
        self.scale = scale  # softmax scale passed to the library (None: 1/sqrt(head_dim))
        rcb.set_kernel(kernel)
        self.seg = rcb.Segments.from_workload(w)
        self.static = static if static is not None else workloads.static_qkv(w, layer)
        self.live = live if live is not None else workloads.live_qkv(w, layer, step)
        dev = torch.device(device)
        H, D = w.num_heads, w.head_dim
        self.cache = rcb.RefCache(self.seg, num_layers=num_layers, mask_mode=mode, device=dev)
        qs, ks, vs = (t.to(dev) for t in self.static)
        ql, kl, vl = (t.to(dev) for t in self.live)
        self.o_static = torch.full((self.seg.static_rows, H, D), float("nan"), dtype=torch.bfloat16, device=dev)
        self.lse_static = torch.full((self.seg.static_rows, H), float("nan"), dtype=torch.float32, device=dev)
        self.o_live = torch.full((self.seg.live_rows, H, D), float("nan"), dtype=torch.bfloat16, device=dev)
        self.lse_live = torch.full((self.seg.live_rows, H), float("nan"), dtype=torch.float32, device=dev)
        self.cache.build(layer, qs, ks, vs, self.o_static, self.lse_static, scale=scale)
        self.cache.step(layer, ql, kl, vl, self.o_live, self.lse_live, scale=scale)
        torch.cuda.synchronize()
        assert rcb.status() == rcb.OK, rcb.last_error()
        self.k_cache, self.v_cache = (t.cpu() for t in self.cache.kv(layer))


def cache_offsets(w, mode):
    off = [0]
    for r in w.requests:
        off.append(off[-1] + r.n_r + (r.n_st if mode == "beyond_alt" else 0))
    return off


def oracle_static_request(w, mode, b, static, scale, pairs=None):
    r = w.requests[b]
    s0 = w.cu_static[b]
    sl = slice(s0, s0 + r.n_static)
    qs, ks, vs = (bits(t)[sl] for t in static)
    return oracle.prefill(qs, ks, vs, r.n_st, r.n_r, mode, scale, pairs)


def oracle_live_request(w, mode, b, static, live, scale, pairs=None):
    """Step rows of request b; the cache comes from the oracle's own prefill."""
    r = w.requests[b]
    s0 = w.cu_static[b]
    sl = slice(s0, s0 + r.n_static)
    kc, vc = oracle.cached_kv(bits(static[1])[sl], bits(static[2])[sl], r.n_st, mode)
    l0 = w.cu_live[b]
    sl = slice(l0, l0 + r.n_live)
    ql, kl, vl = (bits(t)[sl] for t in live)
    return oracle.step(ql, kl, vl, kc, vc, r.n_lt, r.n_x, r.n_st, r.n_r, mode, scale, pairs)


def check_close(gpu_o, ref_o, gpu_lse=None, ref_lse=None, what=""):
    g = np.asarray(gpu_o, np.float64)
    assert np.isfinite(g).all(), f"{what}: non-finite GPU output"
    err = np.abs(g - ref_o)
    assert err.max() <= MAX_ABS, f"{what}: max-abs {err.max():.3e} > {MAX_ABS}"
    assert err.mean() <= MEAN_ABS, f"{what}: mean-abs {err.mean():.3e} > {MEAN_ABS}"
    if gpu_lse is not None:
        le = np.abs(np.asarray(gpu_lse, np.float64) - ref_lse)
        assert le.max() <= LSE_ABS, f"{what}: lse max-abs {le.max():.3e}"
    return float(err.max()), float(err.mean())


def full_compare(run: GpuRun, scale=None):
    """Every output row of both calls against the oracle (at the run's softmax
    scale unless one is given)."""
    w, mode = run.w, run.mode
    scale = scale or getattr(run, "scale", None) or 1.0 / math.sqrt(w.head_dim)
    o_s, l_s, o_l, l_l = f64(run.o_static), f64(run.lse_static), f64(run.o_live), f64(run.lse_live)
    coff = cache_offsets(w, mode)
    for b, r in enumerate(w.requests):
        s0, l0 = w.cu_static[b], w.cu_live[b]
        if r.n_static:
            ref_o, ref_l, kc, vc = oracle_static_request(w, mode, b, run.static, scale)
            check_close(o_s[s0:s0 + r.n_static], ref_o, l_s[s0:s0 + r.n_static], ref_l, f"prefill req {b}")
            np.testing.assert_array_equal(bits(run.k_cache)[coff[b]:coff[b + 1]], kc)
            np.testing.assert_array_equal(bits(run.v_cache)[coff[b]:coff[b + 1]], vc)
        if r.n_live:
            ref_o, ref_l = oracle_live_request(w, mode, b, run.static, run.live, scale)
            check_close(o_l[l0:l0 + r.n_live], ref_o, l_l[l0:l0 + r.n_live], ref_l, f"step req {b}")


def sample_rows(n, rng, extra=24):
    """Tile edges, the ragged tail and random rows of a segment of n rows."""
    if n == 0:
        return np.zeros(0, np.int64)
    edges = {0, 1, 127, 128, 129, 255, 256, 257, n - 129, n - 128, n - 2, n - 1}
    rows = {e for e in edges if 0 <= e < n}
    rows |= set(int(x) for x in rng.integers(0, n, size=min(extra, n)))
    return np.array(sorted(rows), np.int64)


def sampled_compare(run: GpuRun, seed=0, per_request=24, scale=None, heads=None):
    """Sampled (row, head) outputs of both calls against the oracle, computed
    one by one; heads restricts the sampled heads."""
    w, mode = run.w, run.mode
    scale = scale or 1.0 / math.sqrt(w.head_dim)
    rng = np.random.default_rng(seed)
    o_s, l_s, o_l, l_l = f64(run.o_static), f64(run.lse_static), f64(run.o_live), f64(run.lse_live)
    coff = cache_offsets(w, mode)
    for b, r in enumerate(w.requests):
        s0, l0 = w.cu_static[b], w.cu_live[b]
        rows = sample_rows(r.n_static, rng, per_request)
        hs = rng.choice(np.asarray(heads), size=rows.size) if heads is not None else rng.integers(0, w.num_heads, size=rows.size)
        pairs = np.stack([rows, hs], 1).astype(np.int32)
        ref_o, ref_l, kc, vc = oracle_static_request(w, mode, b, run.static, scale, pairs)
        check_close(o_s[s0 + pairs[:, 0], pairs[:, 1]], ref_o, l_s[s0 + pairs[:, 0], pairs[:, 1]], ref_l,
                    f"prefill req {b} (sampled)")
        np.testing.assert_array_equal(bits(run.k_cache)[coff[b]:coff[b + 1]], kc)
        np.testing.assert_array_equal(bits(run.v_cache)[coff[b]:coff[b + 1]], vc)
        rows = sample_rows(r.n_live, rng, per_request)
        hs = rng.choice(np.asarray(heads), size=rows.size) if heads is not None else rng.integers(0, w.num_heads, size=rows.size)
        pairs = np.stack([rows, hs], 1).astype(np.int32)
        ref_o, ref_l = oracle_live_request(w, mode, b, run.static, run.live, scale, pairs)
        check_close(o_l[l0 + pairs[:, 0], pairs[:, 1]], ref_o, l_l[l0 + pairs[:, 0], pairs[:, 1]], ref_l,
                    f"step req {b} (sampled)")


def guard_report(full: np.ndarray, guard: int, n: int, width: int, pattern: int):
    """For a byte buffer laid out as [guard | n bytes of elements of `width`
    bytes | guard], all set to `pattern` before a call: the guard bytes that
    changed before and after the elements, and the elements that still hold
    the pattern in every byte (never written)."""
    before = int((full[:guard] != pattern).sum())
    after = int((full[guard + n:] != pattern).sum())
    words = full[guard:guard + n].reshape(-1, width)
    untouched = int((words == pattern).all(axis=1).sum()) if n else 0
    return before, after, untouched
