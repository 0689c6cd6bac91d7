"""full_attention_noalloc: the entry point for callers that may not allocate
device memory (for example under an allocator that forbids cudaMalloc after
start-up).  Its work list lives in the library's static device memory.

Checked through the C ABI, on two calls in a row (the static array is reused
by the second): against the allocating full_attention on the same inputs bit
for bit (both build the same work items in the same order and launch the same
kernel, so a corrupted work list shows up as a changed bit), and against the
CPU oracle on sampled rows; at both head dims, where one work item covers 128
and 256 query rows.  Oversized inputs are refused at both head dims.  This
file is collected last so that a failure here leaves every other test already
run; it also passes alone in a fresh process.
"""
import ctypes
import math

import numpy as np
import pytest
import torch

import oracle
import workloads
from paper_2608_21229_gb300 import refcache as rcb

import parity_utils as pu

pytestmark = pytest.mark.gpu


def _call_noalloc(lib, cu, q, k, v, o, lse, scale):
    H, D = q.shape[1:]
    arr = (ctypes.c_int32 * len(cu))(*cu)
    return lib.full_attention_noalloc(len(cu) - 1, H, D, arr, q.data_ptr(), k.data_ptr(), v.data_ptr(),
                                      o.data_ptr(), lse.data_ptr(), scale,
                                      torch.cuda.current_stream().cuda_stream)


def _bits_equal(a: torch.Tensor, b: torch.Tensor) -> bool:
    view = torch.int16 if a.dtype == torch.bfloat16 else torch.int32
    return torch.equal(a.view(view), b.view(view))


@pytest.mark.parametrize("kernel", ["tcgen05", "mma_sync"])
@pytest.mark.parametrize("head_dim", [64, 128])
def test_noalloc_matches_full_attention_twice(kernel, head_dim):
    lib = rcb.load()
    oracle.build()
    rcb.set_kernel(kernel)
    try:
        H, D = 8, head_dim
        cu = [0, 1000, 3329, 3330, 3700]  # ragged requests, one of a single row
        n = cu[-1]
        q, k, v = (workloads.randn_bf16((n, H, D), 21, f"noalloc_{t}").cuda() for t in "qkv")
        o_ref = torch.full((n, H, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        lse_ref = torch.full((n, H), float("nan"), dtype=torch.float32, device="cuda")
        rcb.full_attention(cu, q, k, v, o_ref, lse_ref)
        scale = 1.0 / math.sqrt(D)
        rng = np.random.default_rng(D)
        for call in range(2):
            o = torch.full_like(o_ref, float("nan"))
            lse = torch.full_like(lse_ref, float("nan"))
            assert _call_noalloc(lib, cu, q, k, v, o, lse, scale) == rcb.OK, rcb.last_error()
            torch.cuda.synchronize()
            assert rcb.status() == rcb.OK
            assert _bits_equal(o, o_ref), f"call {call}: outputs differ from full_attention"
            assert _bits_equal(lse, lse_ref), f"call {call}: LSE differs from full_attention"
        # and the outputs themselves against the oracle, request by request
        for b in range(len(cu) - 1):
            s0, nb = cu[b], cu[b + 1] - cu[b]
            rows = pu.sample_rows(nb, rng, 12)
            pairs = np.stack([rows, rng.integers(0, H, rows.size)], 1).astype(np.int32)
            sl = slice(s0, s0 + nb)
            ref_o, ref_l = oracle.full(pu.bits(q[sl]), pu.bits(k[sl]), pu.bits(v[sl]), scale, pairs)
            pu.check_close(pu.f64(o[sl])[pairs[:, 0], pairs[:, 1]], ref_o,
                           pu.f64(lse[sl])[pairs[:, 0], pairs[:, 1]], ref_l, f"noalloc request {b}")
    finally:
        rcb.set_kernel("tcgen05")


@pytest.mark.parametrize("head_dim", [64, 128])
def test_noalloc_rejects_inputs_beyond_its_limit(head_dim):
    """One work item (256 query rows at either head dim) more than the static
    array holds is refused.  The tensors are NULL, so that no kernel could run
    even if the limit check let the call through (the pointer check would
    refuse it next)."""
    lib = rcb.load()
    rows = rcb.NOALLOC_MAX_TASKS * 256 + 1
    cu = (ctypes.c_int32 * 2)(0, rows)
    rc = lib.full_attention_noalloc(1, 1, head_dim, cu, None, None, None, None, None, 0.125, None)
    assert rc == rcb.ERR_INVALID_ARG
    assert "static limit" in rcb.last_error()
    # exactly at the limit the same call passes the limit check and stops at the NULL pointers
    cu_at = (ctypes.c_int32 * 2)(0, rcb.NOALLOC_MAX_TASKS * 256)
    assert lib.full_attention_noalloc(1, 1, head_dim, cu_at, None, None, None, None, None, 0.125, None) == rcb.ERR_INVALID_ARG
    assert "static limit" not in rcb.last_error()
