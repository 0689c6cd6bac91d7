"""step_attention inside a CUDA graph: a serving loop can capture the
per-step call once (after a first call on the device has set the kernels'
attributes) and replay it; the replay must give the same bytes as a direct
call, for both cache formats."""
import pytest
import torch

import workloads
from paper_2608_21229_gb300 import refcache as rcb

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("cache_dtype", ["bf16", "fp8"])
def test_step_attention_replays_from_a_cuda_graph(cache_dtype):
    rcb.load()
    rcb.set_kernel("tcgen05")
    w = workloads.EDIT_512_2REF
    seg = rcb.Segments.from_workload(w)
    dev = torch.device("cuda:0")
    cache = rcb.RefCache(seg, device=dev, cache_dtype=cache_dtype)
    qs, ks, vs = (t.to(dev) for t in workloads.static_qkv(w))
    cache.build(0, qs, ks, vs, torch.empty_like(qs))
    lives = [tuple(t.to(dev) for t in workloads.live_qkv(w, step=i)) for i in range(2)]
    ql, kl, vl = (t.clone() for t in lives[0])  # the graph's fixed input buffers
    o_direct = torch.empty_like(ql)
    cache.step(0, ql, kl, vl, o_direct)  # first call: attributes set outside the capture
    torch.cuda.synchronize()
    o_graph = torch.zeros_like(ql)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        cache.step(0, ql, kl, vl, o_graph)
    for i in (1, 0):  # new inputs copied into the captured buffers, then replay
        for dst, src in zip((ql, kl, vl), lives[i]):
            dst.copy_(src)
        g.replay()
        torch.cuda.synchronize()
        ref = torch.empty_like(ql)
        cache.step(0, *lives[i], ref)
        torch.cuda.synchronize()
        assert torch.equal(o_graph.view(torch.int16), ref.view(torch.int16)), f"replay {i} differs"
    assert rcb.status() == rcb.OK
