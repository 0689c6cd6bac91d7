"""Guard bytes around every buffer the library writes (a stand-in for a
memory checker, which this pool does not offer).

Each output (O and LSE of refcache_build, refcache_build_in_slot,
step_attention, full_attention and full_attention_noalloc) sits in the middle
of a larger device buffer whose bytes are all set to one pattern, and so does
the cache memory handed to refcache_create.  After the calls:
  - every guard byte before and after each buffer still holds the pattern
    (nothing is written outside the tensors the caller passed);
  - no element of an output still holds the pattern (every row of every item
    was written: a skipped or lost work item would leave it);
  - the inputs are unchanged, byte for byte.
Ragged batches put request ends inside tiles; both head dims and all three
kernels run, and the E4M3 cache for the CTA-pair kernel.
"""
import ctypes

import numpy as np
import pytest
import torch

import workloads
from paper_2608_21229_gb300 import refcache as rcb

import parity_utils as pu

pytestmark = pytest.mark.gpu

GUARD = 1 << 16  # bytes on each side (keeps the inner buffers 256-byte aligned)
PATTERN = 0xA5


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    rcb.load()
    yield
    rcb.set_kernel("tcgen05")


class Guarded:
    """A device buffer of `shape` x `dtype` between two guard regions."""

    def __init__(self, shape, dtype):
        n = int(np.prod(shape)) * torch.tensor([], dtype=dtype).element_size()
        self.n = n
        self.full = torch.full((GUARD + n + GUARD,), PATTERN, dtype=torch.uint8, device="cuda")
        self.t = self.full[GUARD:GUARD + n].view(dtype).view(*shape)

    def check(self, name, written=True):
        before, after, untouched = pu.guard_report(self.full.cpu().numpy(), GUARD, self.n, self.t.element_size(),
                                                   PATTERN)
        assert before == 0, f"{name}: {before} bytes written before the buffer"
        assert after == 0, f"{name}: {after} bytes written after the buffer"
        if written:
            assert untouched == 0, f"{name}: {untouched} elements never written"


def guarded_cache(seg, mask_mode="beyond", cache_dtype="bf16"):
    """A RefCache whose memory is caller-provided, between two guard regions."""
    L = rcb.load()
    flags = rcb.MASK_MODES[mask_mode] | rcb.CACHE_DTYPES[cache_dtype]
    nbytes = L.refcache_bytes(1, flags, ctypes.byref(seg.c))
    assert nbytes > 0
    g = Guarded((nbytes,), torch.uint8)
    c = rcb.RefCache.__new__(rcb.RefCache)
    c.seg, c.num_layers, c.mask_mode, c.cache_dtype = seg, 1, mask_mode, cache_dtype
    c.mem = g.t
    c.h = ctypes.c_void_p()
    rc = L.refcache_create(ctypes.byref(c.h), 1, flags, ctypes.byref(seg.c), ctypes.c_void_p(g.t.data_ptr()), nbytes)
    assert rc == rcb.OK, rcb.last_error()
    return c, g


def ragged(head_dim, seed):
    rng = np.random.default_rng(seed)
    reqs = list(workloads.random_requests(rng, 3, max_len=700))
    reqs.append(workloads.Request(3, 1, 0, 5))
    return workloads.Workload(f"canary_{head_dim}_{seed}", 3, head_dim, tuple(reqs), seed)


def snapshot(ts):
    return [t.clone() for t in ts]


def unchanged(before, after):
    return all(torch.equal(a.view(torch.int16), b.view(torch.int16)) for a, b in zip(before, after))


CASES = [("tcgen05", 128), ("tcgen05_k128", 128), ("mma_sync", 128), ("tcgen05", 64), ("mma_sync", 64)]


@pytest.mark.parametrize("kernel,head_dim", CASES, ids=[f"{k}_d{d}" for k, d in CASES])
def test_writes_stay_inside_the_buffers(kernel, head_dim):
    rcb.set_kernel(kernel)
    w = ragged(head_dim, 70 + head_dim)
    seg = rcb.Segments.from_workload(w)
    H, D = w.num_heads, w.head_dim
    static = [t.cuda() for t in workloads.static_qkv(w)]
    live = [t.cuda() for t in workloads.live_qkv(w)]
    s0, l0 = snapshot(static), snapshot(live)
    cache, cache_g = guarded_cache(seg)
    o_s, lse_s = Guarded((seg.static_rows, H, D), torch.bfloat16), Guarded((seg.static_rows, H), torch.float32)
    o_l, lse_l = Guarded((seg.live_rows, H, D), torch.bfloat16), Guarded((seg.live_rows, H), torch.float32)
    cache.build(0, *static, o_s.t, lse_s.t)
    for _ in range(2):
        cache.step(0, *live, o_l.t, lse_l.t)
    # full attention over the live rows as one ragged batch of their own
    cu = [0] + list(np.cumsum([r.n_live for r in w.requests]))
    o_f, lse_f = Guarded((seg.live_rows, H, D), torch.bfloat16), Guarded((seg.live_rows, H), torch.float32)
    o_n, lse_n = Guarded((seg.live_rows, H, D), torch.bfloat16), Guarded((seg.live_rows, H), torch.float32)
    rcb.full_attention(cu, *live, o_f.t, lse_f.t)
    rcb.full_attention_noalloc(cu, *live, o_n.t, lse_n.t)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK, rcb.last_error()
    for name, g in (("prefill O", o_s), ("prefill LSE", lse_s), ("step O", o_l), ("step LSE", lse_l),
                    ("full O", o_f), ("full LSE", lse_f), ("noalloc O", o_n), ("noalloc LSE", lse_n)):
        g.check(name)
    cache_g.check("cache", written=False)
    assert unchanged(s0, static) and unchanged(l0, live), "an input was modified"
    cache.close()


@pytest.mark.parametrize("head_dim", [64, 128])
def test_in_slot_build_writes_stay_inside(head_dim):
    rcb.set_kernel("tcgen05")
    w = ragged(head_dim, 90 + head_dim)
    seg = rcb.Segments.from_workload(w)
    H, D = w.num_heads, w.head_dim
    qs, ks, vs = (t.cuda() for t in workloads.static_qkv(w))
    cache, cache_g = guarded_cache(seg)
    k_slot, v_slot = cache.kv(0)
    off = 0
    anchors_k, anchors_v = [], []
    for b, r in enumerate(w.requests):
        s0 = seg.cu_static[b]
        k_slot[off:off + r.n_r] = ks[s0 + r.n_st:s0 + r.n_static]
        v_slot[off:off + r.n_r] = vs[s0 + r.n_st:s0 + r.n_static]
        anchors_k.append(ks[s0:s0 + r.n_st])
        anchors_v.append(vs[s0:s0 + r.n_st])
        off += r.n_r
    ka, va = torch.cat(anchors_k).contiguous(), torch.cat(anchors_v).contiguous()
    before = snapshot([qs, ka, va, k_slot, v_slot])
    o, lse = Guarded((seg.static_rows, H, D), torch.bfloat16), Guarded((seg.static_rows, H), torch.float32)
    cache.build_in_slot(0, qs, ka, va, o.t, lse.t)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK, rcb.last_error()
    o.check("in-slot prefill O")
    lse.check("in-slot prefill LSE")
    cache_g.check("cache", written=False)
    assert unchanged(before, [qs, ka, va, k_slot, v_slot]), "an input or a slot was modified"
    cache.close()


def test_e4m3_cache_writes_stay_inside():
    rcb.set_kernel("tcgen05")
    w = ragged(128, 111)
    seg = rcb.Segments.from_workload(w)
    H, D = w.num_heads, w.head_dim
    static = [t.cuda() for t in workloads.static_qkv(w)]
    live = [t.cuda() for t in workloads.live_qkv(w)]
    s0, l0 = snapshot(static), snapshot(live)
    cache, cache_g = guarded_cache(seg, cache_dtype="fp8")
    o_s = Guarded((seg.static_rows, H, D), torch.bfloat16)
    o_l, lse_l = Guarded((seg.live_rows, H, D), torch.bfloat16), Guarded((seg.live_rows, H), torch.float32)
    cache.build(0, *static, o_s.t)
    cache.step(0, *live, o_l.t, lse_l.t)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK, rcb.last_error()
    for name, g in (("prefill O", o_s), ("step O", o_l), ("step LSE", lse_l)):
        g.check(name)
    cache_g.check("cache", written=False)
    assert unchanged(s0, static) and unchanged(l0, live), "an input was modified"
    cache.close()
