"""refcache_build_in_slot: the prefill of a layer whose cached rows' K and V
the caller projected straight into the cache slots (Sec. 3.3: only R's K/V
are kept, so they can be written where they are kept); the library reads
them from the slots and launches no cache write.

Checked through the C ABI against the CPU oracle (prefill and the step that
follows, every output row), in the three mask modes, at both head dims, on
both kernel families; the step after an in-slot build equals the step after
refcache_build bit for bit (the cache bytes are the same); repeated calls give
the same bytes and leave the slots untouched.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads
from paper_2608_21229_gb300 import refcache as rcb

import parity_utils as pu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    rcb.load()
    oracle.build()
    yield
    rcb.set_kernel("tcgen05")


def fill_slots(cache, w, mode, static, layer=0):
    """Write every request's cached rows (R, or [ST; R] in the alternative
    reading) into the layer's slots, as a projection writing into the cache
    would."""
    k_slot, v_slot = cache.kv(layer)
    off = pu.cache_offsets(w, mode)
    _, ks, vs = static
    for b, r in enumerate(w.requests):
        s0 = w.cu_static[b]
        keep = 0 if mode == "beyond_alt" else r.n_st
        k_slot[off[b]:off[b + 1]] = ks[s0 + keep:s0 + r.n_static].cuda()
        v_slot[off[b]:off[b + 1]] = vs[s0 + keep:s0 + r.n_static].cuda()


def anchor_kv(w, mode, static):
    """The anchors' K and V, request after request ([sum N_ST, H, d]), or
    None where the slots hold them or there are none."""
    if mode == "beyond_alt" or sum(r.n_st for r in w.requests) == 0:
        return None, None
    _, ks, vs = static
    rows = [(w.cu_static[b], r.n_st) for b, r in enumerate(w.requests)]
    return tuple(torch.cat([t[s0:s0 + n] for s0, n in rows]).cuda() for t in (ks, vs))


class InSlotRun:
    """Layer 0 built in the slot, then one step; outputs on the CPU (the same
    fields as parity_utils.GpuRun, so its comparisons apply)."""

    def __init__(self, w, mode="beyond", kernel="tcgen05"):
        self.w, self.mode = w, mode
        rcb.set_kernel(kernel)
        self.seg = rcb.Segments.from_workload(w)
        self.static = workloads.static_qkv(w)
        self.live = workloads.live_qkv(w)
        H, D = w.num_heads, w.head_dim
        self.cache = rcb.RefCache(self.seg, mask_mode=mode)
        fill_slots(self.cache, w, mode, self.static)
        k0, v0 = (t.clone() for t in self.cache.kv(0))
        ka, va = anchor_kv(w, mode, self.static)
        qs = self.static[0].cuda()
        self.o_static = torch.full((self.seg.static_rows, H, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        self.lse_static = torch.full((self.seg.static_rows, H), float("nan"), dtype=torch.float32, device="cuda")
        self.o_live = torch.full((self.seg.live_rows, H, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        self.lse_live = torch.full((self.seg.live_rows, H), float("nan"), dtype=torch.float32, device="cuda")
        self.cache.build_in_slot(0, qs, ka, va, self.o_static, self.lse_static)
        assert self.cache.built(0)
        ql, kl, vl = (t.cuda() for t in self.live)
        self.cache.step(0, ql, kl, vl, self.o_live, self.lse_live)
        torch.cuda.synchronize()
        assert rcb.status() == rcb.OK, rcb.last_error()
        self.k_cache, self.v_cache = (t.cpu() for t in self.cache.kv(0))
        # the call only reads the slots
        assert torch.equal(self.k_cache.view(torch.int16), k0.cpu().view(torch.int16))
        assert torch.equal(self.v_cache.view(torch.int16), v0.cpu().view(torch.int16))


KERNELS = ["tcgen05", "tcgen05_k128", "mma_sync"]


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("mode", ["beyond", "beyond_alt"])
@pytest.mark.parametrize("w", [workloads.TINY, workloads.EDIT_512_2REF], ids=lambda w: w.name)
def test_build_in_slot_matches_oracle(kernel, mode, w):
    pu.full_compare(InSlotRun(w, mode=mode, kernel=kernel))


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("mode", ["beyond", "beyond_alt", "isolated"])
@pytest.mark.parametrize("head_dim", [64, 128])
def test_build_in_slot_ragged_matches_oracle(kernel, mode, head_dim):
    """Ragged requests with lengths 0, 1, odd and across tile edges, some
    without anchors or without references."""
    rng = np.random.default_rng(31 + head_dim)
    reqs = list(workloads.random_requests(rng, 3, max_len=300))
    reqs.append(workloads.Request(1, 0, 1, 1))
    reqs.append(workloads.Request(0, 0, 0, 5))
    reqs.append(workloads.Request(3, 2, 0, 0))
    if mode == "isolated":
        reqs = [workloads.Request(0, r.n_lt, r.n_x, r.n_r) for r in reqs]
    w = workloads.Workload(f"in_slot_ragged_{head_dim}", 3, head_dim, tuple(reqs), 31)
    pu.full_compare(InSlotRun(w, mode=mode, kernel=kernel))


def test_build_in_slot_sampled_edit1024_5ref():
    run = InSlotRun(workloads.EDIT_1024_5REF)
    pu.sampled_compare(run, seed=41, per_request=32)


@pytest.mark.parametrize("mode", ["beyond", "beyond_alt"])
def test_step_after_build_in_slot_equals_step_after_build(mode):
    """The cache bytes are the same either way, so the step is the same bit for bit."""
    w = workloads.EDIT_512_2REF
    a = InSlotRun(w, mode=mode)
    b = pu.GpuRun(w, mode=mode, static=a.static, live=a.live)
    assert np.array_equal(pu.bits(a.o_live), pu.bits(b.o_live))
    assert np.array_equal(pu.bits(a.k_cache), pu.bits(b.k_cache))
    # the prefill itself is tiled differently (anchors and R apart): equal up to rounding order
    d = np.abs(pu.f64(a.o_static) - pu.f64(b.o_static))
    assert d.max() <= pu.MAX_ABS / 10


def test_build_in_slot_repeats_bytes_and_counts_one_launch():
    w = workloads.RAGGED_4REQ
    seg = rcb.Segments.from_workload(w)
    static = workloads.static_qkv(w)
    cache = rcb.RefCache(seg, num_layers=2)
    fill_slots(cache, w, "beyond", static, layer=1)
    ka, va = anchor_kv(w, "beyond", static)
    qs = static[0].cuda()
    H, D = w.num_heads, w.head_dim
    outs = []
    for _ in range(2):
        o = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device="cuda")
        cache.build_in_slot(1, qs, ka, va, o)
        outs.append(o)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    assert torch.equal(outs[0].view(torch.int16), outs[1].view(torch.int16))
    assert cache.built(1) and not cache.built(0)
    assert cache.launches("build_in_slot") == 1


def test_build_in_slot_refuses_e4m3_cache_and_missing_anchors():
    w = workloads.EDIT_512_2REF
    seg = rcb.Segments.from_workload(w)
    H, D = w.num_heads, w.head_dim
    qs = torch.zeros(seg.static_rows, H, D, dtype=torch.bfloat16, device="cuda")
    o = torch.empty_like(qs)
    f8 = rcb.RefCache(seg, cache_dtype="fp8")
    ka = torch.zeros(w.requests[0].n_st, H, D, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(rcb.RefCacheError) as e:
        f8.build_in_slot(0, qs, ka, ka, o)
    assert e.value.code == rcb.ERR_UNSUPPORTED
    cache = rcb.RefCache(seg)
    rc = rcb.load().refcache_build_in_slot(cache.h, 0, qs.data_ptr(), None, None, o.data_ptr(), None, 0.1, None)
    assert rc == rcb.ERR_INVALID_ARG
    assert not cache.built(0)
