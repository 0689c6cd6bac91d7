"""Beyond-mask joint attention with exact reference K/V caching on GB300.

The library (csrc/, built into _build/librefcache.so) implements the per-step
masked joint attention of an in-context diffusion transformer with static
text anchors: ``RefCache.build`` (the one-shot [ST; R] prefill that fills the
per-layer reference K/V cache), ``RefCache.step`` (live [LT; X_t] rows over
their own keys and the cache) and ``full_attention`` (the full recompute
baseline).  ``refcache`` is the ctypes binding of the C ABI in
include/refcache.h.
"""
from . import accounting
from .refcache import (KERNELS, MASK_MODES, RefCache, RefCacheError, Segments, full_attention, load,
                       set_kernel, set_wait_timeout_ns, status, version)

__all__ = ["accounting", "KERNELS", "MASK_MODES", "RefCache", "RefCacheError", "Segments", "full_attention",
           "load", "set_kernel", "set_wait_timeout_ns", "status", "version"]
