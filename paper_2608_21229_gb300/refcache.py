"""Thin ctypes binding of librefcache.so (include/refcache.h).

Argument marshalling only: torch tensors are passed as raw device pointers,
the current torch stream as the CUDA stream.  Every attention step runs in the
library's CUDA kernels; when the library is missing this module raises, it
never falls back to another implementation.
"""
from __future__ import annotations

import ctypes
import math
import os
from typing import Optional, Sequence

from . import build as _build

OK = 0
ERR_INVALID_ARG = -1
ERR_UNSUPPORTED = -2
ERR_NOT_BUILT = -3
ERR_CUDA = -4
ERR_OOM = -5
ERR_TIMEOUT = -6

MASK_MODES = {"beyond": 0, "beyond_alt": 1, "isolated": 2}
KERNELS = {"tcgen05": 0, "mma_sync": 1, "tcgen05_k128": 2}
CACHE_DTYPES = {"bf16": 0, "fp8": 0x100}  # REFCACHE_CACHE_FP8: E4M3 codes with per-tile scales

EXPORTED = (
    "refcache_bytes", "refcache_create", "refcache_destroy", "refcache_kv_ptr", "refcache_layer_built",
    "refcache_build", "step_attention", "full_attention", "refcache_status", "refcache_set_wait_timeout_ns",
    "refcache_set_kernel", "refcache_debug_skip_first_load", "refcache_last_error", "refcache_version",
    "full_attention_noalloc", "refcache_call_launches", "refcache_fp8_ptr", "refcache_build_in_slot",
    "refcache_cache_status", "refcache_ex2_rate",
)
NOALLOC_MAX_TASKS = 16384


class RefCacheError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"refcache error {code}: {msg}")
        self.code = code


class _Segments(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int32), ("num_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("cu_live", ctypes.POINTER(ctypes.c_int32)), ("cu_static", ctypes.POINTER(ctypes.c_int32)),
        ("n_anchor", ctypes.POINTER(ctypes.c_int32)), ("n_instr", ctypes.POINTER(ctypes.c_int32)),
    ]


_lib = None


def lib_path() -> str:
    return _build.LIB_PATH


def load(path: Optional[str] = None):
    """Load the CUDA library.  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or lib_path()
    if not os.path.exists(path):
        raise RuntimeError(f"CUDA library not built ({path} missing): run __graft_entry__.build() "
                           "or python -m paper_2608_21229_gb300.build")
    L = ctypes.CDLL(path)
    vp, i32, i64, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float
    segp = ctypes.POINTER(_Segments)
    L.refcache_bytes.argtypes = [i32, i32, segp]
    L.refcache_bytes.restype = ctypes.c_size_t
    L.refcache_create.argtypes = [ctypes.POINTER(vp), i32, i32, segp, vp, ctypes.c_size_t]
    L.refcache_destroy.argtypes = [vp]
    L.refcache_destroy.restype = None
    L.refcache_kv_ptr.argtypes = [vp, i32, ctypes.POINTER(vp), ctypes.POINTER(vp), ctypes.POINTER(i64)]
    L.refcache_fp8_ptr.argtypes = [vp, i32, ctypes.POINTER(vp), ctypes.POINTER(vp), ctypes.POINTER(vp),
                                   ctypes.POINTER(i64)]
    L.refcache_layer_built.argtypes = [vp, i32]
    L.refcache_call_launches.argtypes = [vp, i32]
    L.refcache_build.argtypes = [vp, i32, vp, vp, vp, vp, vp, f32, vp]
    L.refcache_build_in_slot.argtypes = [vp, i32, vp, vp, vp, vp, vp, f32, vp]
    L.step_attention.argtypes = [vp, i32, vp, vp, vp, vp, vp, f32, vp]
    L.full_attention.argtypes = [i32, i32, i32, ctypes.POINTER(ctypes.c_int32), vp, vp, vp, vp, vp, f32, vp]
    L.full_attention_noalloc.argtypes = [i32, i32, i32, ctypes.POINTER(ctypes.c_int32), vp, vp, vp, vp, vp, f32,
                                         vp]
    L.refcache_status.argtypes = [vp]
    L.refcache_cache_status.argtypes = [vp, vp]
    L.refcache_set_wait_timeout_ns.argtypes = [ctypes.c_uint64]
    L.refcache_set_wait_timeout_ns.restype = ctypes.c_uint64
    L.refcache_set_kernel.argtypes = [i32]
    L.refcache_debug_skip_first_load.argtypes = [i32]
    L.refcache_ex2_rate.argtypes = [ctypes.POINTER(ctypes.c_double), vp]
    L.refcache_debug_skip_first_load.restype = None
    L.refcache_last_error.argtypes = [ctypes.c_char_p, ctypes.c_size_t]
    L.refcache_version.restype = ctypes.c_char_p
    for name in EXPORTED:
        getattr(L, name)
    _lib = L
    return L


def last_error() -> str:
    buf = ctypes.create_string_buffer(1024)
    load().refcache_last_error(buf, len(buf))
    return buf.value.decode(errors="replace")


def _check(code: int):
    if code != OK:
        raise RefCacheError(code, last_error())


def _arr(vals: Optional[Sequence[int]]):
    if vals is None:
        return None
    return (ctypes.c_int32 * len(vals))(*[int(v) for v in vals])


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("tensor must live on the GPU")
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    import torch

    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _check_thd(name, t, rows, H, D):
    import torch

    if t is None:
        raise ValueError(f"{name} is required")
    if t.dtype != torch.bfloat16 or tuple(t.shape) != (rows, H, D):
        raise ValueError(f"{name}: expected bf16 [{rows}, {H}, {D}], got {t.dtype} {tuple(t.shape)}")


def set_kernel(name: str) -> str:
    old = load().refcache_set_kernel(KERNELS[name])
    _check(0 if old >= 0 else old)
    return {v: k for k, v in KERNELS.items()}[old]


def set_wait_timeout_ns(ns: int) -> int:
    return int(load().refcache_set_wait_timeout_ns(int(ns)))


def debug_skip_first_load(on: bool = True) -> None:
    load().refcache_debug_skip_first_load(1 if on else 0)


def status(stream=None) -> int:
    """Synchronise the stream and return the device error word as a status code."""
    return int(load().refcache_status(_stream(stream)))


def ex2_rate(stream=None) -> float:
    """Exponentials (ex2.approx.f32) per clock per SM measured on the current
    device by the library's probe kernel."""
    v = ctypes.c_double(0.0)
    _check(load().refcache_ex2_rate(ctypes.byref(v), _stream(stream)))
    return float(v.value)


def version() -> str:
    return load().refcache_version().decode()


def default_scale(head_dim: int) -> float:
    return 1.0 / math.sqrt(head_dim)


class Segments:
    """Host segment table (refcache_segments_t)."""

    def __init__(self, num_heads, head_dim, cu_live, cu_static, n_anchor, n_instr=None):
        self.num_heads, self.head_dim = int(num_heads), int(head_dim)
        self.cu_live, self.cu_static = list(cu_live), list(cu_static)
        self.n_anchor = list(n_anchor)
        self.n_instr = None if n_instr is None else list(n_instr)
        self.batch = len(self.n_anchor)
        self._keep = [_arr(self.cu_live), _arr(self.cu_static), _arr(self.n_anchor), _arr(self.n_instr)]
        self.c = _Segments(self.batch, self.num_heads, self.head_dim, *self._keep)

    @classmethod
    def from_workload(cls, w):
        return cls(w.num_heads, w.head_dim, w.cu_live, w.cu_static, w.n_anchor, w.n_instr)

    @property
    def live_rows(self):
        return self.cu_live[-1]

    @property
    def static_rows(self):
        return self.cu_static[-1]


class RefCache:
    """The persistent per-layer reference K/V cache (refcache_t).

    Device memory for the cache comes from torch (one uint8 tensor) and is
    handed to refcache_create, so the library itself allocates nothing.
    """

    def __init__(self, seg: Segments, num_layers: int = 1, mask_mode: str = "beyond", device=None,
                 cache_dtype: str = "bf16"):
        import torch

        L = load()
        self.seg, self.num_layers, self.mask_mode = seg, int(num_layers), mask_mode
        self.cache_dtype = cache_dtype
        flags = MASK_MODES[mask_mode] | CACHE_DTYPES[cache_dtype]
        nbytes = L.refcache_bytes(self.num_layers, flags, ctypes.byref(seg.c))
        if nbytes == 0:
            # the planner rejected the arguments: surface its message
            h = ctypes.c_void_p()
            _check(L.refcache_create(ctypes.byref(h), self.num_layers, flags, ctypes.byref(seg.c),
                                     ctypes.c_void_p(1), 0))
        device = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
        self.mem = torch.empty(nbytes, dtype=torch.uint8, device=device)
        self.h = ctypes.c_void_p()
        with torch.cuda.device(device):
            _check(L.refcache_create(ctypes.byref(self.h), self.num_layers, flags, ctypes.byref(seg.c),
                                     ctypes.c_void_p(self.mem.data_ptr()), nbytes))

    def close(self):
        if getattr(self, "h", None) is not None and self.h.value:
            load().refcache_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def kv(self, layer: int):
        """(K slot, V slot) of a layer as bf16 [cache_rows, H, D] views of the cache memory."""
        import torch

        k, v, rows = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_int64()
        _check(load().refcache_kv_ptr(self.h, layer, ctypes.byref(k), ctypes.byref(v), ctypes.byref(rows)))
        H, D = self.seg.num_heads, self.seg.head_dim
        n = rows.value * H * D * 2
        base = self.mem.data_ptr()

        def view(p):
            off = p.value - base
            return self.mem[off:off + n].view(torch.bfloat16).view(rows.value, H, D)

        return view(k), view(v)

    def fp8(self, layer: int):
        """E4M3 cache of a layer as views of the cache memory: (K codes uint8
        [rows_pad, H, D], V codes uint8 [H, D, rows_pad], scales float32
        [rows_pad / 128, H, 4] = (s_K, s_V, log2 s_V, 1 / s_V))."""
        import torch

        k, v, sc, rows = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_int64()
        _check(load().refcache_fp8_ptr(self.h, layer, ctypes.byref(k), ctypes.byref(v), ctypes.byref(sc),
                                       ctypes.byref(rows)))
        H, D, n = self.seg.num_heads, self.seg.head_dim, rows.value
        base = self.mem.data_ptr()

        def view(p, nbytes):
            off = p.value - base
            return self.mem[off:off + nbytes]

        return (view(k, n * H * D).view(n, H, D), view(v, n * H * D).view(H, D, n),
                view(sc, (n // 128) * H * 16).view(torch.float32).view(n // 128, H, 4))

    def status(self, stream=None) -> int:
        """Synchronise the stream and return (and clear) this cache's own error
        word as a status code: a bounded wait of one of its launches ran out."""
        return int(load().refcache_cache_status(self.h, _stream(stream)))

    def built(self, layer: int) -> bool:
        r = load().refcache_layer_built(self.h, layer)
        _check(0 if r >= 0 else r)
        return bool(r)

    def launches(self, call: str) -> int:
        """Kernels one build ('build'), step ('step') or in-slot build ('build_in_slot') call launches."""
        r = load().refcache_call_launches(self.h, {"build": 0, "step": 1, "build_in_slot": 2}[call])
        _check(0 if r >= 0 else r)
        return int(r)

    def build(self, layer, q, k, v, o, lse=None, scale=None, stream=None):
        H, D, n = self.seg.num_heads, self.seg.head_dim, self.seg.static_rows
        for name, t in (("q", q), ("k", k), ("v", v), ("o", o)):
            _check_thd(name, t, n, H, D)
        scale = default_scale(D) if scale is None else scale
        _check(load().refcache_build(self.h, layer, _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), scale,
                                     _stream(stream)))

    def build_in_slot(self, layer, q, k_anchor, v_anchor, o, lse=None, scale=None, stream=None):
        """The prefill of a layer whose cached rows' K/V the caller already
        wrote into the slots (``kv(layer)``); the anchors' K/V are passed apart
        as [sum n_anchor, H, D] (None when there are none, or in the
        alternative anchor reading, whose slots hold them)."""
        H, D, n = self.seg.num_heads, self.seg.head_dim, self.seg.static_rows
        for name, t in (("q", q), ("o", o)):
            _check_thd(name, t, n, H, D)
        n_a = sum(self.seg.n_anchor) if self.mask_mode != "beyond_alt" else 0
        if n_a:
            for name, t in (("k_anchor", k_anchor), ("v_anchor", v_anchor)):
                _check_thd(name, t, n_a, H, D)
        else:
            k_anchor = v_anchor = None
        scale = default_scale(D) if scale is None else scale
        _check(load().refcache_build_in_slot(self.h, layer, _ptr(q), _ptr(k_anchor), _ptr(v_anchor), _ptr(o),
                                             _ptr(lse), scale, _stream(stream)))

    def step(self, layer, q, k, v, o, lse=None, scale=None, stream=None):
        H, D, n = self.seg.num_heads, self.seg.head_dim, self.seg.live_rows
        for name, t in (("q", q), ("k", k), ("v", v), ("o", o)):
            _check_thd(name, t, n, H, D)
        scale = default_scale(D) if scale is None else scale
        _check(load().step_attention(self.h, layer, _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), scale,
                                     _stream(stream)))


def full_attention(cu_seqlens, q, k, v, o, lse=None, scale=None, stream=None):
    rows, H, D = q.shape
    cu = list(cu_seqlens)
    for name, t in (("q", q), ("k", k), ("v", v), ("o", o)):
        _check_thd(name, t, cu[-1], H, D)
    scale = default_scale(D) if scale is None else scale
    _check(load().full_attention(len(cu) - 1, H, D, _arr(cu), _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse),
                                 scale, _stream(stream)))


def full_attention_noalloc(cu_seqlens, q, k, v, o, lse=None, scale=None, stream=None):
    """full_attention whose work list sits in the library's static device
    memory: the call allocates no device memory (see include/refcache.h)."""
    rows, H, D = q.shape
    cu = list(cu_seqlens)
    for name, t in (("q", q), ("k", k), ("v", v), ("o", o)):
        _check_thd(name, t, cu[-1], H, D)
    scale = default_scale(D) if scale is None else scale
    _check(load().full_attention_noalloc(len(cu) - 1, H, D, _arr(cu), _ptr(q), _ptr(k), _ptr(v), _ptr(o),
                                         _ptr(lse), scale, _stream(stream)))
