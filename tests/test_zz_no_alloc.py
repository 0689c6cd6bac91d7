"""full_attention_noalloc: the entry point for callers that may not allocate
device memory (for example under an allocator that forbids cudaMalloc after
start-up).  Its work list lives in the library's static device memory.

Checked through the C ABI against the allocating full_attention on the same
inputs, on two calls in a row (the static array is reused by the second), in
the tolerance of the other parity tests; and oversized inputs are refused.
This file is collected last so that a failure here leaves every other test
already run; it also passes alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

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


@pytest.mark.parametrize("kernel", ["tcgen05", "mma_sync"])
def test_noalloc_matches_full_attention_twice(kernel):
    lib = rcb.load()
    rcb.set_kernel(kernel)
    try:
        H, D = 8, 128
        cu = [0, 1000, 3329, 3330, 3700]  # ragged requests, one of a single row
        n = cu[-1]
        q, k, v = (workloads.randn_bf16((n, H, D), 21, f"noalloc_{t}").cuda() for t in "qkv")
        o_ref = torch.empty(n, H, D, dtype=torch.bfloat16, device="cuda")
        lse_ref = torch.empty(n, H, dtype=torch.float32, device="cuda")
        rcb.full_attention(cu, q, k, v, o_ref, lse_ref)
        scale = 1.0 / np.sqrt(D)
        for _ in range(2):
            o = torch.full_like(o_ref, float("nan"))
            lse = torch.full_like(lse_ref, float("nan"))
            assert _call_noalloc(lib, cu, q, k, v, o, lse, scale) == rcb.OK, rcb.last_error()
            torch.cuda.synchronize()
            assert rcb.status() == rcb.OK
            pu.check_close(pu.f64(o), pu.f64(o_ref), pu.f64(lse), pu.f64(lse_ref), "noalloc vs full_attention")
    finally:
        rcb.set_kernel("tcgen05")


def test_noalloc_rejects_inputs_beyond_its_limit():
    lib = rcb.load()
    rows = (rcb.NOALLOC_MAX_TASKS + 1) * 128
    cu = (ctypes.c_int32 * 2)(0, rows)
    q = torch.empty(16, dtype=torch.bfloat16, device="cuda")
    rc = lib.full_attention_noalloc(1, 1, 64, cu, q.data_ptr(), q.data_ptr(), q.data_ptr(), q.data_ptr(), None,
                                    0.125, None)
    assert rc == rcb.ERR_INVALID_ARG
    assert "static limit" in rcb.last_error()
