"""The E4M3 reference cache (REFCACHE_CACHE_FP8) through the C ABI against the
CPU oracle of ``oracle/fp8.py`` on the same seeded inputs.

Bar: the cache codes and scales bit for bit; every step output within the
oracle's worst-case bound of the bf16 / E4M3 rounding of the softmax weights
(which the oracle does not model) plus FP8_SLACK, and, for requests with at
least FP8_STAT_MIN_KEYS cached keys, within FP8_MAX_ABS / FP8_MEAN_ABS (all
pinned on the CPU by ``test_oracle_fp8.py``); the LSE within the exact path's
bound (the weights' rounding does not enter it); the prefill's outputs equal
the bf16 cache's bit for bit (the same kernel on the same inputs).
"""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads
from oracle import fp8 as ofp8
from paper_2608_21229_gb300 import refcache as rcb

import parity_utils as pu
from test_oracle_fp8 import FP8_MAX_ABS, FP8_MEAN_ABS, FP8_SLACK, FP8_STAT_MIN_KEYS

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    rcb.load()
    oracle.build()
    rcb.set_kernel("tcgen05")
    yield
    rcb.set_kernel("tcgen05")


class Fp8Run:
    """Build of layer 0 and one step on an E4M3 cache; outputs and the cache on the CPU."""

    def __init__(self, w, mode="beyond", layer=0, step=0, static=None):
        self.w, self.mode = w, mode
        self.seg = rcb.Segments.from_workload(w)
        self.static = static if static is not None else workloads.static_qkv(w, layer)
        self.live = workloads.live_qkv(w, layer, step)
        dev = torch.device("cuda:0")
        H, D = w.num_heads, w.head_dim
        self.cache = rcb.RefCache(self.seg, mask_mode=mode, device=dev, cache_dtype="fp8")
        qs, ks, vs = (t.to(dev) for t in self.static)
        ql, kl, vl = (t.to(dev) for t in self.live)
        self.o_static = torch.full((self.seg.static_rows, H, D), float("nan"), dtype=torch.bfloat16, device=dev)
        self.lse_static = torch.full((self.seg.static_rows, H), float("nan"), dtype=torch.float32, device=dev)
        self.o_live = torch.full((self.seg.live_rows, H, D), float("nan"), dtype=torch.bfloat16, device=dev)
        self.lse_live = torch.full((self.seg.live_rows, H), float("nan"), dtype=torch.float32, device=dev)
        self.cache.build(layer, qs, ks, vs, self.o_static, self.lse_static)
        self.cache.step(layer, ql, kl, vl, self.o_live, self.lse_live)
        torch.cuda.synchronize()
        assert rcb.status() == rcb.OK, rcb.last_error()
        k8, vt8, sc = self.cache.fp8(layer)
        self.k8, self.vt8, self.scales = k8.cpu().numpy(), vt8.cpu().numpy(), sc.cpu().numpy()


def cached_rows(w, mode, static, b):
    """Request b's cached K and V (bf16 bits), as the exact oracle's prefill keeps them."""
    r = w.requests[b]
    s0 = w.cu_static[b]
    sl = slice(s0, s0 + r.n_static)
    return oracle.cached_kv(pu.bits(static[1])[sl], pu.bits(static[2])[sl], r.n_st, mode)


def check_cache(run, heads):
    """The E4M3 cache of the given heads, bit for bit against the oracle's quantisation."""
    w, mode = run.w, run.mode
    parts = [cached_rows(w, mode, run.static, b) for b in range(w.batch)]
    lens = [p[0].shape[0] for p in parts]
    kc = np.concatenate([p[0] for p in parts])[:, heads]
    vc = np.concatenate([p[1] for p in parts])[:, heads]
    k8, vt8, sc, off = ofp8.build_fp8_cache(kc, vc, lens)
    np.testing.assert_array_equal(run.k8[:, heads], k8)
    np.testing.assert_array_equal(run.vt8[heads], vt8)
    np.testing.assert_array_equal(run.scales[:, heads, :2], sc)
    # derived columns the kernel reads: log2 s_V and 1 / s_V (0 where s_V = 0)
    sv = sc[..., 1].astype(np.float64)
    nz = sv > 0
    np.testing.assert_allclose(run.scales[:, heads, 2][nz], np.log2(sv[nz]), rtol=0, atol=1e-5)
    np.testing.assert_allclose(run.scales[:, heads, 3][nz], 1.0 / sv[nz], rtol=1e-6)
    assert not run.scales[:, heads, 2:][~nz].any()
    return k8, vt8, sc, off, lens


def check_step(run, heads, rows_per_request=None, seed=0, statistical=True):
    """Step outputs of (row, head) pairs against the FP8 oracle; all rows when
    rows_per_request is None, else tile edges plus that many random rows.  The
    statistical bounds assume that many keys carry the softmax weight
    (statistical=False checks the worst-case bound only)."""
    w = run.w
    scale = 1.0 / math.sqrt(w.head_dim)
    k8, vt8, sc, off, lens = check_cache(run, heads)
    kd, vd = ofp8.dequantized_cache(k8, vt8, sc, off, lens)
    vsc = ofp8.cached_v_scales(sc, off, lens)
    cum = np.concatenate([[0], np.cumsum(lens)])
    o_l, l_l = pu.f64(run.o_live), pu.f64(run.lse_live)
    rng = np.random.default_rng(seed)
    errs = []
    for b, r in enumerate(w.requests):
        if r.n_live == 0:
            continue
        l0 = w.cu_live[b]
        if rows_per_request is None:
            rows = np.arange(r.n_live)
            hj = np.repeat(np.arange(len(heads))[None], rows.size, 0).reshape(-1)
            rows = np.repeat(rows, len(heads))
        else:
            rows = pu.sample_rows(r.n_live, rng, rows_per_request)
            hj = rng.integers(0, len(heads), size=rows.size)
        pairs = np.stack([rows, hj], 1)
        q, k, v = (pu.bits(t)[l0:l0 + r.n_live][:, heads] for t in run.live)
        ref_o, ref_l, bnd = ofp8.step_fp8(q, k, v, kd[cum[b]:cum[b + 1]], vd[cum[b]:cum[b + 1]], scale, pairs,
                                          bound=True, v_scale=vsc[cum[b]:cum[b + 1]])
        hs = np.asarray(heads)[hj]
        g_o = o_l[l0 + rows, hs]
        assert np.isfinite(g_o).all(), f"step req {b}: non-finite output"
        err = np.abs(g_o - ref_o)
        over = err - (bnd + FP8_SLACK)
        assert over.max() <= 0, f"step req {b}: error above the rounding bound by {over.max():.3e}"
        if statistical and lens[b] >= FP8_STAT_MIN_KEYS:
            assert err.max() <= FP8_MAX_ABS, f"step req {b}: max-abs {err.max():.3e}"
            assert err.mean() <= FP8_MEAN_ABS, f"step req {b}: mean-abs {err.mean():.3e}"
        le = np.abs(l_l[l0 + rows, hs] - ref_l)
        assert le.max() <= pu.LSE_ABS, f"step req {b}: lse max-abs {le.max():.3e}"
        errs.append((float(err.max()), float(err.mean())))
    return errs


@pytest.mark.parametrize("mode", ["beyond", "beyond_alt"])
def test_fp8_cfg_small_full_compare(mode):
    w = workloads.CFG_SMALL
    run = Fp8Run(w, mode=mode)
    check_step(run, heads=list(range(w.num_heads)))


@pytest.mark.parametrize("seed", [21, 22])
def test_fp8_ragged_full_compare(seed):
    """Ragged requests: lengths 0, 1, odd and across tile edges; a request with
    no cached rows, one with a 5-row cache, one without live rows."""
    rng = np.random.default_rng(seed)
    reqs = list(workloads.random_requests(rng, 3, max_len=400))
    reqs += [workloads.Request(1, 0, 1, 5), workloads.Request(0, 3, 40, 0), workloads.Request(3, 0, 0, 130)]
    w = workloads.Workload(f"fp8_ragged_{seed}", 3, 128, tuple(reqs), seed)
    run = Fp8Run(w)
    check_step(run, heads=[0, 1, 2])


def test_fp8_prefill_equals_bf16_cache_prefill():
    w = workloads.CFG_SMALL
    run8 = Fp8Run(w)
    run16 = pu.GpuRun(w)
    assert torch.equal(run8.o_static.view(torch.int16), run16.o_static.view(torch.int16))
    assert torch.equal(run8.lse_static.view(torch.int32), run16.lse_static.view(torch.int32))


def test_fp8_edit1024_5ref_sampled():
    """The 1024^2 five-reference step at full size; heads 21-23 run as split items."""
    run = Fp8Run(workloads.EDIT_1024_5REF)
    check_step(run, heads=[0, 7, 21, 23], rows_per_request=40, seed=3)


def test_fp8_cfg_edit1024_5ref_sampled():
    run = Fp8Run(workloads.CFG_1024_5REF)
    check_step(run, heads=[5, 22], rows_per_request=30, seed=4)


def test_fp8_step_refused_on_mma_sync_kernel():
    w = workloads.CFG_SMALL
    seg = rcb.Segments.from_workload(w)
    cache = rcb.RefCache(seg, device="cuda:0", cache_dtype="fp8")
    dev = torch.device("cuda:0")
    qs, ks, vs = (t.to(dev) for t in workloads.static_qkv(w))
    ql, kl, vl = (t.to(dev) for t in workloads.live_qkv(w))
    o_s = torch.empty_like(qs)
    o_l = torch.empty_like(ql)
    cache.build(0, qs, ks, vs, o_s)
    rcb.set_kernel("mma_sync")
    try:
        with pytest.raises(rcb.RefCacheError) as e:
            cache.step(0, ql, kl, vl, o_l)
        assert e.value.code == rcb.ERR_UNSUPPORTED
    finally:
        rcb.set_kernel("tcgen05")
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK


def test_fp8_call_launches():
    w = workloads.EDIT_1024_5REF
    cache = rcb.RefCache(rcb.Segments.from_workload(w), device="cuda:0", cache_dtype="fp8")
    assert cache.launches("build") >= 2  # quantisation + attention (+ combine)
    assert cache.launches("step") >= 1


def test_fp8_layers_are_independent_and_match_single_layer_caches():
    """A three-layer E4M3 cache: each layer built with its own inputs gives the
    same cache bytes and step outputs as a one-layer cache of that layer."""
    w = workloads.CFG_SMALL
    seg = rcb.Segments.from_workload(w)
    dev = torch.device("cuda:0")
    H, D = w.num_heads, w.head_dim
    multi = rcb.RefCache(seg, num_layers=3, device=dev, cache_dtype="fp8")
    outs = {}
    for layer in (2, 0, 1):  # out of order: a layer's build must not touch another's
        qs, ks, vs = (t.to(dev) for t in workloads.static_qkv(w, layer))
        o_s = torch.empty_like(qs)
        multi.build(layer, qs, ks, vs, o_s)
    for layer in range(3):
        ql, kl, vl = (t.to(dev) for t in workloads.live_qkv(w, layer))
        o_l = torch.empty_like(ql)
        multi.step(layer, ql, kl, vl, o_l)
        outs[layer] = o_l
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    for layer in range(3):
        single = rcb.RefCache(seg, num_layers=1, device=dev, cache_dtype="fp8")
        qs, ks, vs = (t.to(dev) for t in workloads.static_qkv(w, layer))
        ql, kl, vl = (t.to(dev) for t in workloads.live_qkv(w, layer))
        o_s, o_l = torch.empty_like(qs), torch.empty_like(ql)
        single.build(0, qs, ks, vs, o_s)
        single.step(0, ql, kl, vl, o_l)
        torch.cuda.synchronize()
        for a, b in zip(multi.fp8(layer), single.fp8(0)):
            assert torch.equal(a, b), f"layer {layer}: cache bytes differ"
        assert torch.equal(outs[layer].view(torch.int16), o_l.view(torch.int16)), f"layer {layer}: outputs differ"


def test_fp8_edit1024_10ref_sampled():
    """The largest reference count of the sweep (40960 cached rows per request)."""
    w = [x for x in workloads.SWEEP_1024 if x.requests[0].n_r == 10 * 4096][0]
    run = Fp8Run(w)
    check_step(run, heads=[3, 22], rows_per_request=24, seed=9)


def test_fp8_rescale_path_full_compare():
    """Cached keys growing tile by tile: the running maximum and the tile scales
    change along the row, so the rescale path and the per-tile weight shifts run."""
    from test_gpu_parity import _growing_keys

    w = workloads.Workload("fp8_growing_keys", 2, 128, (workloads.Request(16, 32, 200, 1500),), 13)
    run = Fp8Run(w, static=_growing_keys(w))
    # the growing keys make every row's softmax peaked (a few keys of the last
    # tiles carry the weight), so the rounding of those weights does not
    # average out: only the worst-case bound applies
    check_step(run, heads=[0, 1], statistical=False)


def test_accessors_refuse_the_other_cache_format():
    w = workloads.CFG_SMALL
    seg = rcb.Segments.from_workload(w)
    c8 = rcb.RefCache(seg, device="cuda:0", cache_dtype="fp8")
    c16 = rcb.RefCache(seg, device="cuda:0")
    with pytest.raises(rcb.RefCacheError) as e:
        c8.kv(0)
    assert e.value.code == rcb.ERR_UNSUPPORTED
    with pytest.raises(rcb.RefCacheError) as e:
        c16.fp8(0)
    assert e.value.code == rcb.ERR_UNSUPPORTED
    with pytest.raises(rcb.RefCacheError) as e:
        c8.fp8(1)  # one layer only
    assert e.value.code == rcb.ERR_INVALID_ARG
    k8, vt8, sc = c8.fp8(0)
    rows_pad = sum((r.n_r + 127) // 128 * 128 for r in w.requests)
    assert k8.shape == (rows_pad, w.num_heads, w.head_dim) and vt8.shape == (w.num_heads, w.head_dim, rows_pad)
    assert sc.shape == (rows_pad // 128, w.num_heads, 4)


def test_fp8_ragged_4req_sampled():
    """The paper-shaped ragged serving batch (four requests, 1 to 8 references)
    on the E4M3 cache, sampled at full size."""
    run = Fp8Run(workloads.RAGGED_4REQ)
    check_step(run, heads=[2, 19], rows_per_request=24, seed=11)


@pytest.mark.parametrize("seed", [31, 32, 33])
def test_fp8_many_ragged_requests(seed):
    """Up to a dozen ragged requests per batch (empty and one-row segments,
    caches across tile edges), every output of two heads against the oracle."""
    rng = np.random.default_rng(seed)
    reqs = list(workloads.random_requests(rng, int(rng.integers(6, 12)), max_len=300))
    reqs.append(workloads.Request(0, 0, 1, 1))
    w = workloads.Workload(f"fp8_many_{seed}", 3, 128, tuple(reqs), seed)
    run = Fp8Run(w)
    check_step(run, heads=[0, 2])
