"""Failure detection without a GPU fault.

Every wait inside the tcgen05 kernel is bounded.  The library's debug switch
makes the TMA producer skip its first K-tile load (a load that never
arrives), so the consumers' waits run out: the kernel must then set the
device error word (and the launching cache's own word), leave every loop,
free its tensor memory and return, and refcache_status() (and the cache's
refcache_cache_status()) must report REFCACHE_ERR_TIMEOUT -- no trap, no
hang, and the context stays usable for the next, correct call.
"""
import pytest
import torch

import workloads
from paper_2608_21229_gb300 import refcache as rcb

import parity_utils as pu

pytestmark = pytest.mark.gpu


def test_wait_timeout_is_reported_and_context_survives():
    rcb.load()
    rcb.set_kernel("tcgen05")
    w = workloads.TINY
    run = pu.GpuRun(w)  # a normal build + step first
    seg = run.seg
    H, D = w.num_heads, w.head_dim
    ql, kl, vl = (t.cuda() for t in run.live)
    o = torch.zeros(seg.live_rows, H, D, dtype=torch.bfloat16, device="cuda")
    old = rcb.set_wait_timeout_ns(50_000_000)  # 50 ms
    try:
        rcb.debug_skip_first_load(True)
        run.cache.step(0, ql, kl, vl, o)
        assert rcb.status() == rcb.ERR_TIMEOUT
        assert "wait ran out" in rcb.last_error()
        assert rcb.status() == rcb.OK  # the error word was cleared
    finally:
        rcb.debug_skip_first_load(False)
        rcb.set_wait_timeout_ns(old)
    # the context is still usable and correct
    again = pu.GpuRun(w, static=run.static, live=run.live)
    pu.full_compare(again)


@pytest.mark.parametrize("cache_dtype", ["bf16", "fp8"])
def test_pair_kernel_wait_timeout_is_reported_and_context_survives(cache_dtype):
    """The same on the head-dim-128 CTA-pair kernel (its gate, MMA, producer and
    softmax warps in both CTAs, and for the E4M3 cache the query-tile, scale
    ring and row-sum waits): the leader skips its first stage, every wait of
    the pair runs out or sees the abort, and the next call is correct."""
    rcb.load()
    rcb.set_kernel("tcgen05")
    w = workloads.CFG_SMALL
    seg = rcb.Segments.from_workload(w)
    H, D = w.num_heads, w.head_dim
    cache = rcb.RefCache(seg, device="cuda:0", cache_dtype=cache_dtype)
    other = rcb.RefCache(seg, device="cuda:0", cache_dtype=cache_dtype)  # a second cache on the device
    qs, ks, vs = (t.cuda() for t in workloads.static_qkv(w))
    ql, kl, vl = (t.cuda() for t in workloads.live_qkv(w))
    o_s = torch.empty_like(qs)
    cache.build(0, qs, ks, vs, o_s)
    other.build(0, qs, ks, vs, o_s)
    o_ref = torch.empty_like(ql)
    cache.step(0, ql, kl, vl, o_ref)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK and cache.status() == rcb.OK and other.status() == rcb.OK
    o = torch.zeros_like(ql)
    old = rcb.set_wait_timeout_ns(50_000_000)  # 50 ms
    try:
        rcb.debug_skip_first_load(True)
        cache.step(0, ql, kl, vl, o)
        # the fault is this cache's: its own word says so, the other cache's does not
        assert cache.status() == rcb.ERR_TIMEOUT
        assert "this cache" in rcb.last_error()
        assert cache.status() == rcb.OK and other.status() == rcb.OK
        assert rcb.status() == rcb.ERR_TIMEOUT
        assert "wait ran out" in rcb.last_error()
        assert rcb.status() == rcb.OK
    finally:
        rcb.debug_skip_first_load(False)
        rcb.set_wait_timeout_ns(old)
    # the context is still usable: the same step gives the same bytes as before
    o2 = torch.empty_like(ql)
    cache.step(0, ql, kl, vl, o2)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    assert torch.equal(o2.view(torch.int16), o_ref.view(torch.int16))
