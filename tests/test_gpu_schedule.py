"""Work distribution of the CTA-pair kernel (head dim 128).

Items are handed out through a work counter: the CTA pair that is free takes
the next item of the list, so which pair computes an item changes from launch
to launch, while each item's arithmetic does not.  The last pair to finish
resets the counter for the next launch.  Checked through the C ABI:
  - outputs and LSE equal, bit for bit, those of the same call with items in
    the static order (full_attention_noalloc keeps it), on ragged batches;
  - launches with more items than CTA pairs and with fewer, interleaved on one
    stream and across two caches, repeat their bytes (an unreset counter
    would skip items and leave the NaN the outputs are filled with);
  - two caches (each with its own counter) driven at the same time on two
    streams give the bytes of the same calls made one after the other;
  - 240 launches of four kinds in rotation, with no host synchronisation
    between them, all repeat the bytes of the first call of their kind;
  - the same holds for the E4M3 cache's kernel.
"""
import numpy as np
import pytest
import torch

import workloads
from paper_2608_21229_gb300 import refcache as rcb

import parity_utils as pu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    rcb.load()
    rcb.set_kernel("tcgen05")
    yield
    rcb.set_kernel("tcgen05")


def _qkv(lengths, H, seed):
    g = torch.Generator().manual_seed(seed)
    rows = sum(lengths)
    q, k, v = (torch.randn(rows, H, 128, generator=g).to(torch.bfloat16).cuda() for _ in range(3))
    cu = [0]
    for n in lengths:
        cu.append(cu[-1] + n)
    return cu, q, k, v


def _full(fn, cu, q, k, v):
    o = torch.full_like(q, float("nan"))
    lse = torch.full((q.shape[0], q.shape[1]), float("nan"), dtype=torch.float32, device="cuda")
    fn(cu, q, k, v, o, lse)
    return o, lse


def _bits(o, lse):
    return pu.bits(o.cpu()), lse.cpu().numpy().view(np.int32)


BIG = ([5000, 777, 2300, 1], 8, 1)  # 33 tasks x 8 heads: more items than CTA pairs
SMALL = ([300], 2, 2)                # 4 items: fewer than CTA pairs


@pytest.mark.parametrize("case", [BIG, SMALL], ids=["more_items_than_pairs", "fewer_items_than_pairs"])
def test_outputs_do_not_depend_on_which_pair_takes_an_item(case):
    cu, q, k, v = _qkv(*case)
    a = _bits(*_full(rcb.full_attention, cu, q, k, v))
    b = _bits(*_full(rcb.full_attention_noalloc, cu, q, k, v))
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    assert not np.isnan(pu.f64(_full(rcb.full_attention, cu, q, k, v)[0])).any()


def test_counter_resets_between_launches_of_different_sizes():
    big, small = _qkv(*BIG), _qkv(*SMALL)
    ref = {n: _bits(*_full(rcb.full_attention_noalloc, *x)) for n, x in (("big", big), ("small", small))}
    for name in ("big", "small", "big", "small", "small", "big"):
        got = _bits(*_full(rcb.full_attention, *(big if name == "big" else small)))
        assert np.array_equal(got[0], ref[name][0]) and np.array_equal(got[1], ref[name][1]), name
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK


def _cache_run(w, cache_dtype="bf16"):
    seg = rcb.Segments.from_workload(w)
    cache = rcb.RefCache(seg, cache_dtype=cache_dtype)
    H, D = w.num_heads, w.head_dim
    static = [t.cuda() for t in workloads.static_qkv(w)]
    live = [t.cuda() for t in workloads.live_qkv(w)]
    o_s = torch.full((seg.static_rows, H, D), float("nan"), dtype=torch.bfloat16, device="cuda")
    cache.build(0, *static, o_s)

    def step():
        o = torch.full((seg.live_rows, H, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        cache.step(0, *live, o)
        return o

    return cache, o_s, step


def test_two_caches_interleaved_repeat_their_bytes():
    """Two caches on one stream (each with its own counter), steps and
    prefills interleaved: every repeat gives the first call's bytes."""
    a_cache, a_pre, a_step = _cache_run(workloads.EDIT_512_2REF)
    b_cache, b_pre, b_step = _cache_run(workloads.RAGGED_4REQ)
    first = {"a": pu.bits(a_step().cpu()), "b": pu.bits(b_step().cpu())}
    for name in ("b", "a", "a", "b", "a"):
        got = pu.bits((a_step if name == "a" else b_step)().cpu())
        assert np.array_equal(got, first[name]), name
    # a second prefill of each cache between steps
    pre2 = torch.full_like(a_pre, float("nan"))
    w = workloads.EDIT_512_2REF
    a_cache.build(0, *[t.cuda() for t in workloads.static_qkv(w)], pre2)
    assert np.array_equal(pu.bits(pre2.cpu()), pu.bits(a_pre.cpu()))
    assert np.array_equal(pu.bits(b_step().cpu()), first["b"])
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    assert a_cache.status() == rcb.OK and b_cache.status() == rcb.OK


def test_e4m3_cache_step_repeats_its_bytes():
    cache, _, step = _cache_run(workloads.EDIT_512_2REF, cache_dtype="fp8")
    first = pu.bits(step().cpu())
    assert not np.isnan(pu.f64(step())).any()
    for _ in range(3):
        assert np.array_equal(pu.bits(step().cpu()), first)
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK


def test_two_caches_on_two_streams_at_once():
    """Each cache has its own work counter, so launches of two caches may run
    at the same time on two streams; their outputs equal those of the same
    calls made one after the other."""
    runs = {}
    for name, w in (("a", workloads.EDIT_512_2REF), ("b", workloads.RAGGED_4REQ)):
        cache, _, step = _cache_run(w)
        runs[name] = (cache, step, pu.bits(step().cpu()))
    torch.cuda.synchronize()
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    outs = {"a": [], "b": []}
    for _ in range(3):
        for name, s in (("a", sa), ("b", sb)):
            with torch.cuda.stream(s):
                outs[name].append(runs[name][1]())
    torch.cuda.synchronize()
    assert rcb.status() == rcb.OK
    for name in ("a", "b"):
        assert runs[name][0].status() == rcb.OK
        for o in outs[name]:
            assert np.array_equal(pu.bits(o.cpu()), runs[name][2]), name


def test_counter_survives_many_launches():
    """Many launches back to back with no host synchronisation between them:
    steps of two caches and full attention of two sizes in a fixed rotation,
    every output checked against the first call of its kind, bit for bit."""
    a_cache, _, a_step = _cache_run(workloads.EDIT_512_2REF)
    b_cache, _, b_step = _cache_run(workloads.RAGGED_4REQ)
    big, small = _qkv(*BIG), _qkv(*SMALL)
    calls = {
        "a": a_step,
        "b": b_step,
        "big": lambda: _full(rcb.full_attention, *big)[0],
        "small": lambda: _full(rcb.full_attention, *small)[0],
    }
    first = {k: pu.bits(f().cpu()) for k, f in calls.items()}
    outs = []
    for i in range(60):
        for k in ("a", "big", "b", "small") if i % 2 == 0 else ("small", "b", "a", "big"):
            outs.append((k, calls[k]()))
        if len(outs) >= 40:  # compare in batches to bound the memory held
            torch.cuda.synchronize()
            for k, o in outs:
                assert np.array_equal(pu.bits(o.cpu()), first[k]), k
            outs = []
    torch.cuda.synchronize()
    for k, o in outs:
        assert np.array_equal(pu.bits(o.cpu()), first[k]), k
    assert rcb.status() == rcb.OK
    assert a_cache.status() == rcb.OK and b_cache.status() == rcb.OK
