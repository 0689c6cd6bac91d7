"""Failure detection without a GPU fault.

Every wait inside the tcgen05 kernel is bounded.  The library's debug switch
makes the TMA producer skip its first K-tile load (a load that never
arrives), so the consumers' waits run out: the kernel must then set the
device error word, leave every loop, free its tensor memory and return, and
refcache_status() must report REFCACHE_ERR_TIMEOUT -- no trap, no hang, and
the context stays usable for the next, correct call.
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
