"""CPU oracle for the beyond-mask joint attention -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline /
reference leg may import this package.  The library under
``paper_2608_21229_gb300`` never imports it, and this package imports nothing
from the library.

Contents:
  * ``oracle.c`` (compiled here with gcc): the plain fp64 definition of masked
    softmax attention over one request's joint sequence [LT; X_t; ST; R]
    (Sec. 3.3), plus a brute-force explicit-mask variant;
  * ``structure``: the layered dependency graph of App. A (reachability,
    StructCacheable, LiveTextReachable, Theorem 1);
  * ``cost_model``: the interaction-count model of App. C.

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
against closed forms, a library routine, brute force and the paper's printed
numbers; none is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

MODES = {"beyond": 0, "beyond_alt": 1, "isolated": 2, "full": 3}
BLOCKS = ("LT", "X", "ST", "R")


def build(force: bool = False) -> str:
    """Compile oracle.c into oracle/_build/liboracle.so (gcc, OpenMP).

    ``-ffp-contract=off`` keeps every multiply and add as written, so the
    result does not depend on whether the host compiler fuses them.
    """
    os.makedirs(_BUILD, exist_ok=True)
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-fPIC",
           "-shared", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            path = build()
            L = ctypes.CDLL(path)
            u16p = ctypes.POINTER(ctypes.c_uint16)
            dp = ctypes.POINTER(ctypes.c_double)
            L.oracle_block_visible.argtypes = [ctypes.c_int] * 3
            L.oracle_block_visible.restype = ctypes.c_int
            L.oracle_max_threads.restype = ctypes.c_int
            L.oracle_set_threads.argtypes = [ctypes.c_int]
            L.oracle_attention_explicit_mask.argtypes = [
                u16p, u16p, u16p, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                ctypes.POINTER(ctypes.c_ubyte), ctypes.c_double, dp, dp]
            L.oracle_attention_explicit_mask.restype = ctypes.c_int
            L.oracle_joint_attention.argtypes = [
                u16p, u16p, u16p, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double,
                ctypes.POINTER(ctypes.c_int32), ctypes.c_long, dp, dp]
            L.oracle_joint_attention.restype = ctypes.c_int
            _lib = L
    return _lib


def _u16(a):
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError("oracle inputs are raw bf16 bit patterns (uint16)")
    return a


def _ptr(a, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def block_visible(mode: str, q_block: str, k_block: str) -> bool:
    r = lib().oracle_block_visible(MODES[mode], BLOCKS.index(q_block), BLOCKS.index(k_block))
    if r < 0:
        raise ValueError("bad mode or block")
    return bool(r)


def max_threads() -> int:
    return int(lib().oracle_max_threads())


def set_threads(n: int) -> None:
    lib().oracle_set_threads(int(n))


def attention_explicit_mask(q, k, v, mask, scale):
    """Brute force: q [nq,H,d], k/v [nk,H,d] bf16 bits; mask [nq,nk] bool or None.

    Returns (out [nq,H,d] fp64, lse [nq,H] fp64).
    """
    q, k, v = _u16(q), _u16(k), _u16(v)
    nq, H, d = q.shape
    nk = k.shape[0]
    out = np.zeros((nq, H, d), np.float64)
    lse = np.zeros((nq, H), np.float64)
    mp = None
    if mask is not None:
        m = np.ascontiguousarray(mask, dtype=np.uint8)
        assert m.shape == (nq, nk)
        mp = _ptr(m, ctypes.c_ubyte)
    rc = lib().oracle_attention_explicit_mask(
        _ptr(q, ctypes.c_uint16), _ptr(k, ctypes.c_uint16), _ptr(v, ctypes.c_uint16),
        nq, nk, H, d, mp, float(scale), _ptr(out, ctypes.c_double), _ptr(lse, ctypes.c_double))
    if rc != 0:
        raise RuntimeError(f"oracle_attention_explicit_mask failed: {rc}")
    return out, lse


def joint_attention(q, k, v, n_lt, n_x, n_st, n_r, mode, scale, pairs=None):
    """One request's joint sequence [LT; X; ST; R] (Sec. 3.3), bf16 bits.

    Without ``pairs``: returns (out [N,H,d], lse [N,H]).  With ``pairs`` (an
    int array of (row, head)): returns (out [P,d], lse [P]).
    """
    q, k, v = _u16(q), _u16(k), _u16(v)
    n, H, d = q.shape
    assert n == n_lt + n_x + n_st + n_r and k.shape == q.shape and v.shape == q.shape
    if pairs is None:
        out = np.zeros((n, H, d), np.float64)
        lse = np.zeros((n, H), np.float64)
        pp, npairs = None, 0
    else:
        pairs = np.ascontiguousarray(pairs, dtype=np.int32).reshape(-1, 2)
        npairs = pairs.shape[0]
        out = np.zeros((npairs, d), np.float64)
        lse = np.zeros((npairs,), np.float64)
        if npairs == 0:
            return out, lse
        pp = _ptr(pairs, ctypes.c_int32)
    rc = lib().oracle_joint_attention(
        _ptr(q, ctypes.c_uint16), _ptr(k, ctypes.c_uint16), _ptr(v, ctypes.c_uint16),
        n_lt, n_x, n_st, n_r, H, d, MODES[mode], float(scale), pp, npairs,
        _ptr(out, ctypes.c_double), _ptr(lse, ctypes.c_double))
    if rc != 0:
        raise RuntimeError(f"oracle_joint_attention failed: {rc}")
    return out, lse


def prefill(q_s, k_s, v_s, n_st, n_r, mode, scale, pairs=None):
    """The static block [ST; R] of one request, evaluated once (Sec. 3.3).

    Inputs are that request's [ST; R] rows.  Returns the outputs of the ST and
    R rows and the cache contents, which are the R rows' K and V themselves
    (Eq. 2): (out, lse, k_cache, v_cache).  In the alternative anchor reading
    the cache also keeps the anchors' K and V, so it is the whole [ST; R].
    """
    out, lse = joint_attention(q_s, k_s, v_s, 0, 0, n_st, n_r, mode, scale, pairs)
    k_c, v_c = cached_kv(k_s, v_s, n_st, mode)
    return out, lse, k_c, v_c


def cached_kv(k_s, v_s, n_st, mode):
    """What the static pass keeps (Sec. 3.3): the R rows' K and V, Eq. 2 -- plus
    the anchors' rows in the alternative anchor reading."""
    keep = 0 if mode == "beyond_alt" else n_st
    return np.array(k_s[keep:], copy=True), np.array(v_s[keep:], copy=True)


def step_inputs(q_l, k_l, v_l, k_cache, v_cache, n_lt, n_x, n_st, n_r, mode):
    """The joint sequence [LT; X_t; ST; R] of one denoising step (Sec. 3.3
    order), with the ST/R keys and values taken from the cache.  Queries of the
    ST and R rows are zero placeholders (those rows are not computed in a
    step); in the paper's mask the anchors' K/V are not cached and not
    visible to live rows, so their slots hold zeros."""
    q_l, k_l, v_l = _u16(q_l), _u16(k_l), _u16(v_l)
    H, d = q_l.shape[1:]
    assert q_l.shape[0] == n_lt + n_x
    if mode == "beyond_alt":
        assert k_cache.shape[0] == n_st + n_r
        k_st, v_st = k_cache[:n_st], v_cache[:n_st]
        k_r, v_r = k_cache[n_st:], v_cache[n_st:]
    else:
        assert k_cache.shape[0] == n_r
        k_st = np.zeros((n_st, H, d), np.uint16)
        v_st = np.zeros((n_st, H, d), np.uint16)
        k_r, v_r = k_cache, v_cache
    q = np.concatenate([q_l, np.zeros((n_st + n_r, H, d), np.uint16)])
    k = np.concatenate([k_l, k_st, k_r])
    v = np.concatenate([v_l, v_st, v_r])
    return q, k, v


def step(q_l, k_l, v_l, k_cache, v_cache, n_lt, n_x, n_st, n_r, mode, scale, pairs=None):
    """One denoising step for one request (App. C "Derivation").

    The live rows [LT; X_t] query the joint sequence whose ST/R keys come from
    the cache (``step_inputs``).  ``k_cache``/``v_cache`` hold R (or [ST; R] in
    the alternative anchor reading).  Returns (out, lse) of the live rows:
    [n_live, H, d] / [n_live, H], or per pair with ``pairs``.
    """
    q, k, v = step_inputs(q_l, k_l, v_l, k_cache, v_cache, n_lt, n_x, n_st, n_r, mode)
    H, d = q.shape[1:]
    n_live = n_lt + n_x
    if pairs is None:
        pairs = np.array([(i, h) for i in range(n_live) for h in range(H)], np.int32).reshape(-1, 2)
        out, lse = joint_attention(q, k, v, n_lt, n_x, n_st, n_r, mode, scale, pairs)
        return out.reshape(n_live, H, d), lse.reshape(n_live, H)
    pairs = np.asarray(pairs, np.int32).reshape(-1, 2)
    assert (pairs[:, 0] < n_live).all()
    return joint_attention(q, k, v, n_lt, n_x, n_st, n_r, mode, scale, pairs)


def full(q, k, v, scale, pairs=None):
    """Full attention over one request's whole sequence (all keys visible)."""
    n = q.shape[0]
    return joint_attention(q, k, v, 0, n, 0, 0, "full", scale, pairs)
