"""CUDA path (through the C ABI) against the CPU oracle on the same seeded inputs.

Bar: max |gpu - oracle| <= 2e-2 and mean |gpu - oracle| <= 2e-3 for outputs,
|lse| error <= 2e-3; cached K/V and the exact-caching invariant bit for bit.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads
from paper_2608_21229_gb300 import refcache as rcb

import parity_utils as pu

pytestmark = pytest.mark.gpu

KERNELS = ["tcgen05", "tcgen05_k128", "mma_sync"]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    rcb.load()
    oracle.build()
    yield
    rcb.set_kernel("tcgen05")


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("mode", ["beyond", "beyond_alt"])
def test_tiny_full_compare(kernel, mode):
    run = pu.GpuRun(workloads.TINY, mode=mode, kernel=kernel)
    pu.full_compare(run)


@pytest.mark.parametrize("kernel", KERNELS)
def test_tiny_isolated_full_compare(kernel):
    w = workloads.Workload("tiny_isolated", 4, 64, (workloads.Request(0, 64, 256, 256),), 0)
    run = pu.GpuRun(w, mode="isolated", kernel=kernel)
    pu.full_compare(run)


@pytest.mark.parametrize("kernel", KERNELS)
def test_edit512_2ref_full_compare(kernel):
    run = pu.GpuRun(workloads.EDIT_512_2REF, kernel=kernel)
    pu.full_compare(run)


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("mode", ["beyond", "beyond_alt", "isolated"])
@pytest.mark.parametrize("head_dim", [64, 128])
@pytest.mark.parametrize("seed", [11, 12])
def test_ragged_small_full_compare(kernel, mode, head_dim, seed):
    """Several requests with ragged lengths (0, 1, odd, across tile edges)."""
    rng = np.random.default_rng(seed)
    reqs = list(workloads.random_requests(rng, 3, max_len=300))
    reqs.append(workloads.Request(1, 0, 1, 1))
    reqs.append(workloads.Request(0, 0, 0, 5))
    reqs.append(workloads.Request(3, 2, 0, 0))
    if mode == "isolated":
        reqs = [workloads.Request(0, r.n_lt, r.n_x, r.n_r) for r in reqs]
    w = workloads.Workload(f"ragged_small_{seed}", 3, head_dim, tuple(reqs), seed)
    run = pu.GpuRun(w, mode=mode, kernel=kernel)
    pu.full_compare(run)


@pytest.mark.parametrize("kernel", KERNELS)
def test_edit1024_5ref_sampled(kernel):
    run = pu.GpuRun(workloads.EDIT_1024_5REF, kernel=kernel)
    pu.sampled_compare(run, seed=5)


@pytest.mark.parametrize("refs", [1, 2, 8, 10])
def test_sweep_sampled(refs):
    """The reference-scaling sweep at 1024^2 (5 references is the headline
    test above): prefill and step sampled against the oracle."""
    w = [x for x in workloads.SWEEP_1024 if x.requests[0].n_r == refs * 4096][0]
    run = pu.GpuRun(w, kernel="tcgen05")
    pu.sampled_compare(run, seed=refs, per_request=16)


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("mode", ["beyond", "beyond_alt"])
def test_ragged_serving_batch_sampled(kernel, mode):
    run = pu.GpuRun(workloads.RAGGED_4REQ, mode=mode, kernel=kernel)
    pu.sampled_compare(run, seed=7, per_request=16)


@pytest.mark.parametrize("kernel", KERNELS)
def test_exact_caching_invariant_bitwise(kernel):
    """Sec. 3.1 / 3.3: the prefill outputs and the cache bytes do not depend
    on the live inputs; rebuilding after steps with other live data, and on a
    second layer, reproduces them bit for bit."""
    w = workloads.EDIT_512_2REF
    rcb.set_kernel(kernel)
    seg = rcb.Segments.from_workload(w)
    H, D = w.num_heads, w.head_dim
    cache = rcb.RefCache(seg, num_layers=2)
    qs, ks, vs = (t.cuda() for t in workloads.static_qkv(w))
    o1 = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device="cuda")
    o2 = torch.empty_like(o1)
    cache.build(0, qs, ks, vs, o1)
    k0, v0 = (t.clone() for t in cache.kv(0))
    ol = torch.empty(seg.live_rows, H, D, dtype=torch.bfloat16, device="cuda")
    for step in range(3):
        ql, kl, vl = (t.cuda() for t in workloads.live_qkv(w, step=step))
        cache.step(0, ql, kl, vl, ol)
    cache.build(1, qs, ks, vs, o2)
    o3 = torch.empty_like(o1)
    cache.build(0, qs, ks, vs, o3)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
    assert torch.equal(o1.view(torch.int16), o3.view(torch.int16))
    for layer in (0, 1):
        k, v = cache.kv(layer)
        assert torch.equal(k.view(torch.int16), k0.view(torch.int16))
        assert torch.equal(v.view(torch.int16), v0.view(torch.int16))
    # the cache holds exactly the R rows' K and V given (Eq. 2)
    r = w.requests[0]
    assert torch.equal(k0.view(torch.int16), ks[r.n_st:].view(torch.int16))
    assert torch.equal(v0.view(torch.int16), vs[r.n_st:].view(torch.int16))


@pytest.mark.parametrize("kernel", KERNELS)
def test_step_depends_on_cache_not_on_static_inputs(kernel):
    """The step reads K/V of R only from the cache: overwriting the prefill
    input tensors after the build leaves the step output unchanged."""
    w = workloads.TINY
    rcb.set_kernel(kernel)
    seg = rcb.Segments.from_workload(w)
    H, D = w.num_heads, w.head_dim
    cache = rcb.RefCache(seg)
    qs, ks, vs = (t.cuda() for t in workloads.static_qkv(w))
    os_ = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device="cuda")
    cache.build(0, qs, ks, vs, os_)
    ql, kl, vl = (t.cuda() for t in workloads.live_qkv(w))
    a = torch.empty(seg.live_rows, H, D, dtype=torch.bfloat16, device="cuda")
    b = torch.empty_like(a)
    cache.step(0, ql, kl, vl, a)
    ks.normal_()
    vs.normal_()
    cache.step(0, ql, kl, vl, b)
    torch.cuda.synchronize()
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("w", [workloads.TINY, workloads.EDIT_512_2REF], ids=lambda w: w.name)
def test_full_attention_matches_oracle(kernel, w):
    """The full-recompute baseline: every row of [LT; X; R] sees every key (Sec. 3.2)."""
    rcb.set_kernel(kernel)
    r = w.requests[0]
    n = r.n_lt + r.n_x + r.n_r
    H, D = w.num_heads, w.head_dim
    q, k, v = (workloads.randn_bf16((n, H, D), w.seed, f"full_{t}") for t in "qkv")
    o = torch.empty(n, H, D, dtype=torch.bfloat16, device="cuda")
    lse = torch.empty(n, H, dtype=torch.float32, device="cuda")
    rcb.full_attention([0, n], q.cuda(), k.cuda(), v.cuda(), o, lse)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    rng = np.random.default_rng(3)
    rows = pu.sample_rows(n, rng, 64)
    pairs = np.stack([rows, rng.integers(0, H, rows.size)], 1).astype(np.int32)
    ref_o, ref_l = oracle.full(pu.bits(q), pu.bits(k), pu.bits(v), 1 / math.sqrt(D), pairs)
    go = pu.f64(o)[pairs[:, 0], pairs[:, 1]]
    gl = pu.f64(lse)[pairs[:, 0], pairs[:, 1]]
    pu.check_close(go, ref_o, gl, ref_l, "full")


def test_full_attention_sampled_edit1024_5ref():
    """The recompute baseline at the size the benchmark times it: [LT; X; R] of
    the 1024^2, five-reference edit (25,088 rows, 24 heads), every row over
    every key (C_full in App. C).  Rows at the 256-row task edges, the ragged
    tail and random rows, against the oracle one by one."""
    rcb.set_kernel("tcgen05")
    r = workloads.EDIT_1024_5REF.requests[0]
    n = r.n_lt + r.n_x + r.n_r
    H, D = 24, 128
    q, k, v = (workloads.randn_bf16((n, H, D), 2, f"full_{t}") for t in "qkv")
    o = torch.full((n, H, D), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((n, H), float("nan"), dtype=torch.float32, device="cuda")
    rcb.full_attention([0, n], q.cuda(), k.cuda(), v.cuda(), o, lse)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    rng = np.random.default_rng(25088)
    rows = set(int(x) for x in pu.sample_rows(n, rng, 40))
    rows |= {256 * t + e for t in (1, 17, 50, 97) for e in (-1, 0)} | {n - 256, n - 255}
    rows = np.array(sorted(x for x in rows if 0 <= x < n), np.int64)
    pairs = np.stack([rows, rng.integers(0, H, rows.size)], 1).astype(np.int32)
    ref_o, ref_l = oracle.full(pu.bits(q), pu.bits(k), pu.bits(v), 1 / math.sqrt(D), pairs)
    go = pu.f64(o)[pairs[:, 0], pairs[:, 1]]
    gl = pu.f64(lse)[pairs[:, 0], pairs[:, 1]]
    pu.check_close(go, ref_o, gl, ref_l, "full 1024^2 x 5 refs")


def test_kernels_agree_closely():
    """The two kernels compute the same function (different rounding order)."""
    w = workloads.EDIT_512_2REF
    a = pu.GpuRun(w, kernel="tcgen05")
    b = pu.GpuRun(w, kernel="mma_sync", static=a.static, live=a.live)
    d = (pu.f64(a.o_live) - pu.f64(b.o_live))
    assert np.abs(d).max() < 2e-2 and np.abs(d).mean() < 1e-3


def test_not_built_and_bad_args_are_rejected():
    w = workloads.TINY
    seg = rcb.Segments.from_workload(w)
    cache = rcb.RefCache(seg, num_layers=2)
    H, D = w.num_heads, w.head_dim
    ql, kl, vl = (t.cuda() for t in workloads.live_qkv(w))
    o = torch.empty(seg.live_rows, H, D, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(rcb.RefCacheError) as e:
        cache.step(1, ql, kl, vl, o)
    assert e.value.code == rcb.ERR_NOT_BUILT
    qs, ks, vs = (t.cuda() for t in workloads.static_qkv(w))
    os_ = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(rcb.RefCacheError) as e:
        cache.build(0, qs, ks, vs, os_, scale=-1.0)
    assert e.value.code == rcb.ERR_INVALID_ARG
    with pytest.raises(rcb.RefCacheError) as e:
        cache.build(5, qs, ks, vs, os_)
    assert e.value.code == rcb.ERR_INVALID_ARG
    # misaligned base pointer (2-byte offset view)
    flat = torch.empty(seg.static_rows * H * D + 8, dtype=torch.bfloat16, device="cuda")
    mis = flat[1:1 + seg.static_rows * H * D].view(seg.static_rows, H, D)
    with pytest.raises(rcb.RefCacheError) as e:
        cache.build(0, mis, ks, vs, os_)
    assert e.value.code == rcb.ERR_INVALID_ARG
    assert rcb.status() == rcb.OK


# ---------------------------------------------------------------- CFG pair (positive + negative branch)
@pytest.mark.parametrize("kernel", KERNELS)
def test_cfg_small_full_compare(kernel):
    run = pu.GpuRun(workloads.CFG_SMALL, kernel=kernel)
    pu.full_compare(run)


def test_cfg_edit1024_5ref_sampled():
    run = pu.GpuRun(workloads.CFG_1024_5REF, kernel="tcgen05")
    pu.sampled_compare(run, seed=9, per_request=24)


@pytest.mark.parametrize("w", [workloads.CFG_SMALL, workloads.CFG_1024_5REF], ids=lambda w: w.name)
def test_cfg_pair_equals_branches_run_alone(w):
    """Both branches in one launch give what each branch gives alone.  The
    prefill (outputs, LSE and cache) bit for bit: its items are never split,
    so a request's static block does not depend on what else is in the batch
    (Sec. 3.3).  The step: most outputs bit for bit and every output within a
    tenth of the parity bar (a step launch splits the items of its last round
    by key range, and which items those are depends on the launch's item
    count; each part rounds P against its own running maximum)."""
    pair = pu.GpuRun(w, kernel="tcgen05")
    for b, r in enumerate(w.requests):
        single = workloads.Workload(f"{w.name}_branch{b}", w.num_heads, w.head_dim, (r,), w.seed)
        s0, l0 = w.cu_static[b], w.cu_live[b]
        static = tuple(t[s0:s0 + r.n_static] for t in pair.static)
        live = tuple(t[l0:l0 + r.n_live] for t in pair.live)
        alone = pu.GpuRun(single, kernel="tcgen05", static=static, live=live)
        assert np.array_equal(pu.bits(pair.o_static[s0:s0 + r.n_static]), pu.bits(alone.o_static))
        ls_pair = pair.lse_static[s0:s0 + r.n_static].cpu().view(torch.int32)
        assert torch.equal(ls_pair, alone.lse_static.cpu().view(torch.int32))
        got, ref = pair.o_live[l0:l0 + r.n_live], alone.o_live
        g, a = pu.f64(got), pu.f64(ref)
        assert np.max(np.abs(g - a)) <= pu.MAX_ABS / 10
        assert np.mean(pu.bits(got) == pu.bits(ref)) > 0.5
        c0 = pu.cache_offsets(w, "beyond")[b]
        assert np.array_equal(pu.bits(alone.k_cache), pu.bits(pair.k_cache[c0:c0 + r.n_r]))
        assert np.array_equal(pu.bits(alone.v_cache), pu.bits(pair.v_cache[c0:c0 + r.n_r]))


# ---------------------------------------------------------------- split items (last round of the persistent grid)
def test_split_tail_items_sampled():
    """The last round of items of a step launch is split by key range into
    parts merged by a combine kernel; on the headline case those are items of
    the last heads (head-major order)."""
    run = pu.GpuRun(workloads.EDIT_1024_5REF, kernel="tcgen05")
    pu.sampled_compare(run, seed=21, per_request=64, heads=[21, 22, 23])


def test_split_tail_items_cfg_pair_sampled():
    run = pu.GpuRun(workloads.CFG_1024_5REF, kernel="tcgen05")
    pu.sampled_compare(run, seed=22, per_request=32, heads=[22, 23])


def test_call_launch_counts():
    """Kernels per call: attention (+ cache copy for the build) (+ combine when
    the device's plan split the step's last round; the headline step's 432
    items do not fill 76 CTA pairs evenly, so it is split on a GB300; the
    prefill is never split)."""
    w = workloads.EDIT_1024_5REF
    seg = rcb.Segments.from_workload(w)
    cache = rcb.RefCache(seg, num_layers=1, mask_mode="beyond")
    rcb.set_kernel("tcgen05")
    assert cache.launches("step") in (1, 2)
    assert cache.launches("build") == 2
    rcb.set_kernel("mma_sync")
    assert cache.launches("step") == 1 and cache.launches("build") == 2
    rcb.set_kernel("tcgen05")
    tiny = rcb.RefCache(rcb.Segments.from_workload(workloads.TINY), num_layers=1, mask_mode="beyond")
    assert tiny.launches("step") == 1 and tiny.launches("build") == 2


def _growing_keys(w, growth=0.5):
    """Seeded inputs whose cached keys grow tile by tile (rows of key tile t of
    R scaled by 1 + growth * t), so that a row's running maximum rises by more
    than 2^8 several times after its first tile and the rescale path runs."""
    qs, ks, vs = workloads.static_qkv(w)
    ks = ks.float()
    for b, r in enumerate(w.requests):
        r0 = w.cu_static[b] + r.n_st
        t = torch.arange(r.n_r, dtype=torch.float32) // 128
        ks[r0:r0 + r.n_r] *= (1.0 + growth * t)[:, None, None]
    return qs, ks.to(torch.bfloat16), vs


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("head_dim", [64, 128])
def test_rescale_path_full_compare(kernel, head_dim):
    w = workloads.Workload(f"growing_keys_d{head_dim}", 2, head_dim, (workloads.Request(16, 32, 200, 1500),), 13)
    run = pu.GpuRun(w, kernel=kernel, static=_growing_keys(w))
    pu.full_compare(run)


@pytest.mark.parametrize("kernel,head_dim", [("tcgen05", 128), ("tcgen05_k128", 128), ("tcgen05", 64)])
def test_many_requests_full_compare(kernel, head_dim):
    """40 requests of uneven lengths (up to about 660 live and 600 cached rows) on 8 heads:
    hundreds of work items of different sizes, several per CTA pair, handed
    out by the work counter longest first; every output row compared with the
    oracle."""
    rng = np.random.default_rng(2024 + head_dim)
    reqs = list(workloads.random_requests(rng, 40, max_len=600))
    w = workloads.Workload(f"many_requests_{head_dim}", 8, head_dim, tuple(reqs), 17)
    run = pu.GpuRun(w, mode="beyond", kernel=kernel)
    pu.full_compare(run)


def test_split_tail_items_full_compare():
    """A step whose items all fall in the last round and are long enough to
    split: one request of 768 live rows over 3000 cached rows on 8 heads is
    24 items of 20 key tiles, each split into parts that run on separate CTA
    pairs and are merged by the combine kernel; every output row against the
    oracle, and the cache and prefill as well."""
    w = workloads.Workload("split_tail_768x3000", 8, 128, (workloads.Request(64, 256, 512, 3000),), 19)
    run = pu.GpuRun(w, mode="beyond", kernel="tcgen05")
    pu.full_compare(run)


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("head_dim", [64, 128])
@pytest.mark.parametrize("scale", [0.02, 0.3, 1.0])
def test_softmax_scale_full_compare(kernel, head_dim, scale):
    """Softmax scales other than 1/sqrt(d): nearly uniform weights (0.02) and
    nearly one-hot rows whose running maximum moves often (1.0: scaled scores
    with a standard deviation of sqrt(d)); prefill, cache and step against the
    oracle at the same scale."""
    rng = np.random.default_rng(int(scale * 1000) + head_dim)
    reqs = list(workloads.random_requests(rng, 3, max_len=500))
    w = workloads.Workload(f"scale_{scale}_{head_dim}", 3, head_dim, tuple(reqs), 23)
    run = pu.GpuRun(w, mode="beyond", kernel=kernel, scale=scale)
    pu.full_compare(run)


@pytest.mark.parametrize("head_dim", [64, 128])
def test_layers_keep_their_own_cache(head_dim):
    """Four layers of one cache built from layer-specific inputs (in the order
    2, 0, 3, 1), then one step of every layer: each step is compared with the
    oracle on that layer's own static and live inputs, and each slot holds
    that layer's reference K/V bit for bit."""
    rng = np.random.default_rng(40 + head_dim)
    reqs = list(workloads.random_requests(rng, 3, max_len=400))
    w = workloads.Workload(f"layers_{head_dim}", 3, head_dim, tuple(reqs), 29)
    seg = rcb.Segments.from_workload(w)
    H, D = w.num_heads, w.head_dim
    rcb.set_kernel("tcgen05")
    cache = rcb.RefCache(seg, num_layers=4)
    static = {l: workloads.static_qkv(w, l) for l in range(4)}
    live = {l: workloads.live_qkv(w, l, step=l) for l in range(4)}
    for l in (2, 0, 3, 1):
        o = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device="cuda")
        cache.build(l, *(t.cuda() for t in static[l]), o)
    outs = {}
    for l in range(4):
        outs[l] = torch.full((seg.live_rows, H, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        cache.step(l, *(t.cuda() for t in live[l]), outs[l])
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    scale = 1.0 / np.sqrt(D)
    coff = pu.cache_offsets(w, "beyond")
    for l in range(4):
        k_slot, v_slot = (pu.bits(t) for t in cache.kv(l))
        o = pu.f64(outs[l])
        for b, r in enumerate(w.requests):
            ref, _ = pu.oracle_live_request(w, "beyond", b, static[l], live[l], scale)
            l0 = w.cu_live[b]
            err = np.abs(o[l0:l0 + r.n_live] - ref)
            assert err.size == 0 or (err.max() <= pu.MAX_ABS and err.mean() <= pu.MEAN_ABS), (l, b)
            s0 = w.cu_static[b]
            k_ref = pu.bits(static[l][1])[s0 + r.n_st:s0 + r.n_static]
            v_ref = pu.bits(static[l][2])[s0 + r.n_st:s0 + r.n_static]
            assert np.array_equal(k_slot[coff[b]:coff[b + 1]], k_ref) and np.array_equal(v_slot[coff[b]:coff[b + 1]], v_ref), (l, b)
