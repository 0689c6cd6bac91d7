"""Host-side checks of the C ABI that need no GPU: the library builds and
loads, exports every symbol include/refcache.h declares, and its argument
checks reject bad segment tables before touching a device."""
import ctypes
import os
import re
import subprocess

import pytest

import workloads
from paper_2608_21229_gb300 import accounting
from paper_2608_21229_gb300 import build as cbuild
from paper_2608_21229_gb300 import refcache as rcb

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    cbuild.build()
    return rcb.load()


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "refcache.h")).read()
    return sorted(set(re.findall(r"REFCACHE_API\s+[\w\s\*]+?\b(\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    syms = declared_symbols()
    for name in ("refcache_create", "refcache_build", "step_attention", "full_attention", "refcache_status"):
        assert name in syms
    assert set(syms) == set(rcb.EXPORTED)


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", cbuild.LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    missing = [s for s in declared_symbols() if s not in exported]
    assert not missing, missing
    for s in declared_symbols():
        assert hasattr(lib, s)
    assert "sm_103a" in rcb.version()


def test_library_is_built_for_sm103a_only():
    cmd = cbuild.nvcc_cmd("x.so")
    assert "arch=compute_103a,code=sm_103a" in cmd and cmd.count("-gencode") == 1


def seg_of(w, **kw):
    d = dict(num_heads=w.num_heads, head_dim=w.head_dim, cu_live=w.cu_live, cu_static=w.cu_static,
             n_anchor=w.n_anchor, n_instr=w.n_instr)
    d.update(kw)
    return rcb.Segments(**d)


@pytest.mark.parametrize("w", [workloads.TINY, workloads.EDIT_1024_5REF, workloads.RAGGED_4REQ],
                         ids=lambda w: w.name)
@pytest.mark.parametrize("mode", ["beyond", "beyond_alt"])
def test_cache_bytes_cover_the_slots(lib, w, mode):
    s = seg_of(w)
    layers = 3
    n = lib.refcache_bytes(layers, rcb.MASK_MODES[mode], ctypes.byref(s.c))
    slots = layers * accounting.cache_bytes(w.requests, w.num_heads, w.head_dim, mode)
    assert slots <= n <= slots + 64 * 1024


@pytest.mark.parametrize("bad", [
    dict(cu_live=[0, 10, 5]),
    dict(cu_static=[1, 20]),
    dict(n_anchor=[10 ** 6]),
    dict(n_anchor=[-1]),
    dict(head_dim=96),
    dict(num_heads=0),
    dict(n_instr=[10 ** 6]),
])
def test_bad_segment_tables_are_rejected_on_the_host(lib, bad):
    w = workloads.TINY
    base = dict(cu_live=[0, 320], cu_static=[0, 288], n_anchor=[32])
    base.update(bad)
    s = seg_of(w, **base)
    assert lib.refcache_bytes(1, 0, ctypes.byref(s.c)) == 0
    h = ctypes.c_void_p()
    rc = lib.refcache_create(ctypes.byref(h), 1, 0, ctypes.byref(s.c), None, 0)
    assert rc in (rcb.ERR_INVALID_ARG, rcb.ERR_UNSUPPORTED)
    assert not h.value
    assert rcb.last_error()


def test_isolated_mode_requires_zero_anchors(lib):
    s = seg_of(workloads.TINY)
    assert lib.refcache_bytes(1, rcb.MASK_MODES["isolated"], ctypes.byref(s.c)) == 0
    s0 = seg_of(workloads.TINY, n_anchor=[0])
    assert lib.refcache_bytes(1, rcb.MASK_MODES["isolated"], ctypes.byref(s0.c)) > 0


def test_unknown_mode_and_kernel_rejected(lib):
    s = seg_of(workloads.TINY)
    assert lib.refcache_bytes(1, 7, ctypes.byref(s.c)) == 0
    assert lib.refcache_set_kernel(9) == rcb.ERR_INVALID_ARG
    assert lib.refcache_set_kernel(0) in (0, 1)


def test_full_attention_rejects_bad_args_without_a_device(lib):
    cu = (ctypes.c_int32 * 2)(0, 16)
    assert lib.full_attention(1, 4, 96, cu, None, None, None, None, None, 0.1, None) == rcb.ERR_UNSUPPORTED
    assert lib.full_attention(1, 4, 64, cu, None, None, None, None, None, 0.1, None) == rcb.ERR_INVALID_ARG
    assert lib.full_attention(0, 4, 64, cu, None, None, None, None, None, 0.1, None) == rcb.ERR_INVALID_ARG
    assert lib.full_attention(1, 4, 64, cu, None, None, None, None, None, float("nan"), None) == rcb.ERR_INVALID_ARG


def test_binding_fails_loudly_without_library(tmp_path):
    with pytest.raises(RuntimeError, match="not built"):
        saved = rcb._lib
        rcb._lib = None
        try:
            rcb.load(str(tmp_path / "missing.so"))
        finally:
            rcb._lib = saved


@pytest.mark.parametrize("w", [workloads.EDIT_1024_5REF, workloads.RAGGED_4REQ, workloads.CFG_SMALL],
                         ids=lambda w: w.name)
@pytest.mark.parametrize("mode", ["beyond", "beyond_alt"])
def test_fp8_cache_bytes_follow_the_padded_layout(lib, w, mode):
    """E4M3 cache: per layer the K codes and the transposed V codes of every
    request's cached rows padded to 128, and (s_K, s_V) per tile and head."""
    s = seg_of(w)
    layers = 2
    flags = rcb.MASK_MODES[mode] | rcb.CACHE_DTYPES["fp8"]
    n = lib.refcache_bytes(layers, flags, ctypes.byref(s.c))
    rows_pad = sum((r.n_r + (r.n_st if mode == "beyond_alt" else 0) + 127) // 128 * 128 for r in w.requests)
    align = lambda x: (x + 255) // 256 * 256  # noqa: E731
    per_layer = 2 * align(rows_pad * w.num_heads * w.head_dim) + align(rows_pad // 128 * w.num_heads * 16)
    assert layers * per_layer <= n <= layers * per_layer + 64 * 1024
    bf16 = lib.refcache_bytes(layers, rcb.MASK_MODES[mode], ctypes.byref(s.c))
    assert n < 0.6 * bf16  # about half the bytes of the bf16 cache


def test_fp8_cache_needs_head_dim_128(lib):
    s = seg_of(workloads.TINY)  # head_dim 64
    assert lib.refcache_bytes(1, rcb.CACHE_DTYPES["fp8"], ctypes.byref(s.c)) == 0
    h = ctypes.c_void_p()
    assert lib.refcache_create(ctypes.byref(h), 1, rcb.CACHE_DTYPES["fp8"], ctypes.byref(s.c), None, 0) == \
        rcb.ERR_UNSUPPORTED
