"""CPU oracle of the FP8 reference cache -- TEST INFRASTRUCTURE ONLY.

The paper's cache is exact reuse: the cached K and V are the reference rows'
own bf16 values (Sec. 3.3, Eq. 2).  This module defines an explicitly
approximate variant of it that stores the cached rows in the OCP FP8 E4M3
format with one fp32 scale per tile, and the attention of a denoising step
over that cache.  It is plain numpy, written from the format's definition and
the quantisation rule below; nothing here is shared with the CUDA path.

Quantisation rule (per block of values x, bf16 inputs widened to fp32):
    amax  = max |x| over the block                      (fp32)
    s     = amax / 448          (fp32 division, round to nearest even)
    inv   = 448 / amax, or 0 when amax = 0              (fp32 division)
    code  = E4M3(fp32(x * inv))  (fp32 product, then round to nearest even,
                                  saturating at +-448)
    value = s * decode(code)
Blocks:
  * cached K and V: one block per (tile of 128 cached rows of one request,
    head), i.e. 128 x head_dim values; each request's cached rows are padded
    to a whole number of tiles, pad rows hold code 0;
  * queries of a step: one block per (query row, head), i.e. head_dim values.
The step then attends the live keys with the live rows' exact bf16 queries,
keys and values, and the cached keys with the dequantised queries, keys and
values, in one softmax (App. C's step: live rows over [LT; X_t; R]), in fp64.

Stored layout of one layer's cache (the format the CUDA cache must reproduce
byte for byte):
  * k8      uint8 [rows_pad, H, d]    E4M3 codes, rows in cache order
  * vt8     uint8 [H, d, rows_pad]    E4M3 codes of V, transposed per head
  * scales  float32 [rows_pad / 128, H, 2]  (s_K, s_V) of each tile and head
where request b's cached rows start at row seg_off[b] (a multiple of 128).

Parity status: pinned by ``tests/test_oracle_fp8.py`` (every E4M3 code against
the format's closed forms and a library decoder, the encoder against a
library encoder and against brute-force nearest-value search, and the
quantised step against the exact oracle where the quantisation is lossless).
"""
from __future__ import annotations

import numpy as np

TILE = 128
E4M3_MAX = 448.0


def bf16_to_f32(bits):
    """bf16 bit patterns (uint16) -> float32 values (exact)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def e4m3_decode(codes):
    """E4M3 codes -> float64 values.

    Format (OCP FP8 E4M3, "fn" variant): 1 sign bit, 4 exponent bits with bias
    7, 3 mantissa bits; exponent field 0 is subnormal (m / 8 * 2^-6); there is
    no infinity and the all-ones pattern S.1111.111 is NaN, so the largest
    finite magnitude is 1.75 * 2^8 = 448.
    """
    c = np.asarray(codes, dtype=np.uint8).astype(np.int64)
    sign = np.where(c & 0x80, -1.0, 1.0)
    e = (c >> 3) & 0xF
    m = c & 0x7
    sub = m.astype(np.float64) * 2.0 ** -9
    nor = (1.0 + m / 8.0) * np.exp2(e.astype(np.float64) - 7.0)
    val = np.where(e == 0, sub, nor)
    val = np.where((e == 0xF) & (m == 0x7), np.nan, val)
    return sign * val


def e4m3_encode(x):
    """float32 values -> E4M3 codes, round to nearest (ties to even mantissa),
    magnitudes above 448 saturate to 448, NaN -> 0x7F.  Every step is exact in
    float64, which holds any float32 value."""
    x = np.asarray(x, dtype=np.float32).astype(np.float64)
    out = np.zeros(x.shape, dtype=np.uint8)
    sign = np.signbit(x).astype(np.uint8) << 7
    a = np.abs(x)
    nan = np.isnan(a)
    a = np.where(nan, 0.0, a)
    # subnormal range (below 2^-6): multiples of 2^-9, rounded half to even;
    # 8 * 2^-9 = 2^-6 is code 0x08, the smallest normal, so the carry is exact
    small = a < 2.0 ** -6
    q_sub = np.rint(a / 2.0 ** -9).astype(np.int64)
    # normal range: a = 2^e (1 + f), f rounded to eighths, half to even
    with np.errstate(divide="ignore"):
        e = np.floor(np.log2(np.where(small, 1.0, a))).astype(np.int64)
    # log2 of a float64 can be off by one ulp near a power of two: fix e so
    # that 2^e <= a < 2^(e+1) holds exactly
    e = np.where(np.exp2(e.astype(np.float64)) > a, e - 1, e)
    e = np.where(np.exp2((e + 1).astype(np.float64)) <= a, e + 1, e)
    frac = a / np.exp2(e.astype(np.float64)) - 1.0      # exact: a is a float32
    m = np.rint(frac * 8.0).astype(np.int64)
    e = np.where(m == 8, e + 1, e)
    m = np.where(m == 8, 0, m)
    code_n = ((e + 7) << 3) | m
    # saturate: anything that rounds above 448 (exponent > 8, or 8 with m = 7)
    code_n = np.where((e > 8) | ((e == 8) & (m == 7)), 0x7E, code_n)
    code = np.where(small, q_sub, code_n).astype(np.uint8)
    out = code | sign
    out = np.where(nan, np.uint8(0x7F), out)
    return out.astype(np.uint8)


def quantize_block(x_f32):
    """One block (any shape) of float32 values -> (codes, scale) by the rule in
    the module docstring."""
    x = np.asarray(x_f32, dtype=np.float32)
    amax = np.float32(np.max(np.abs(x))) if x.size else np.float32(0.0)
    s = np.float32(amax / np.float32(E4M3_MAX))
    inv = np.float32(np.float32(E4M3_MAX) / amax) if amax > 0 else np.float32(0.0)
    codes = e4m3_encode((x * inv).astype(np.float32))
    return codes, s


def cache_layout(cached_rows_per_request):
    """Padded row offsets of each request's cached rows: (seg_off[b], rows_pad)."""
    off, pos = [], 0
    for n in cached_rows_per_request:
        off.append(pos)
        pos += (int(n) + TILE - 1) // TILE * TILE
    return off, pos


def build_fp8_cache(k_cached, v_cached, cached_rows_per_request):
    """Quantise one layer's cached K/V (bf16 bits [sum n_b, H, d], requests back
    to back) into (k8, vt8, scales, seg_off)."""
    k = bf16_to_f32(k_cached)
    v = bf16_to_f32(v_cached)
    _, H, d = k.shape
    seg_off, rows_pad = cache_layout(cached_rows_per_request)
    k8 = np.zeros((rows_pad, H, d), np.uint8)
    vt8 = np.zeros((H, d, rows_pad), np.uint8)
    scales = np.zeros((rows_pad // TILE, H, 2), np.float32)
    src = 0
    for b, n in enumerate(cached_rows_per_request):
        for t0 in range(0, n, TILE):
            rows = min(TILE, n - t0)
            dst = seg_off[b] + t0
            tile = dst // TILE
            for h in range(H):
                ck, sk = quantize_block(k[src + t0:src + t0 + rows, h, :])
                cv, sv = quantize_block(v[src + t0:src + t0 + rows, h, :])
                k8[dst:dst + rows, h, :] = ck
                vt8[h, :, dst:dst + rows] = cv.T
                scales[tile, h] = (sk, sv)
        src += n
    return k8, vt8, scales, seg_off


def dequantized_cache(k8, vt8, scales, seg_off, cached_rows_per_request):
    """The values the quantised cache stands for: (K, V) float64 [sum n_b, H, d]."""
    H, d = k8.shape[1], k8.shape[2]
    ks, vs = [], []
    for b, n in enumerate(cached_rows_per_request):
        rows = np.arange(seg_off[b], seg_off[b] + n)
        tiles = rows // TILE
        sk = scales[tiles, :, 0].astype(np.float64)[:, :, None]
        sv = scales[tiles, :, 1].astype(np.float64)[:, :, None]
        ks.append(sk * e4m3_decode(k8[rows]))
        vs.append(sv * e4m3_decode(np.transpose(vt8[:, :, rows], (2, 0, 1))))
    if not ks:
        return np.zeros((0, H, d)), np.zeros((0, H, d))
    return np.concatenate(ks), np.concatenate(vs)


def cached_v_scales(scales, seg_off, cached_rows_per_request):
    """s_V of the tile each cached row belongs to: float64 [sum n_b, H]."""
    out = []
    for b, n in enumerate(cached_rows_per_request):
        rows = np.arange(seg_off[b], seg_off[b] + n)
        out.append(scales[rows // TILE, :, 1].astype(np.float64))
    if not out:
        return np.zeros((0, scales.shape[1]))
    return np.concatenate(out)


def quantize_queries(q_bits):
    """Per (row, head) quantisation of the step's queries: (codes [n, H, d], s [n, H])."""
    q = bf16_to_f32(q_bits)
    n, H, d = q.shape
    codes = np.zeros((n, H, d), np.uint8)
    s = np.zeros((n, H), np.float32)
    for i in range(n):
        for h in range(H):
            codes[i, h], s[i, h] = quantize_block(q[i, h])
    return codes, s


def step_fp8(q_l, k_l, v_l, k_cache_deq, v_cache_deq, scale, pairs, bound=False, v_scale=None):
    """One request's step over the quantised cache, for the (live row, head)
    pairs given: returns (out [P, d], lse [P]) in fp64.

    Keys are the request's live rows (exact bf16 Q, K, V) followed by its
    cached rows (dequantised K, V; each query row dequantised from its own
    per-row E4M3 block); one softmax over all of them with the scores scaled
    by ``scale``.  Every live row sees every key of its request (the mask of
    App. C's step for live rows, with the cache holding R or [ST; R]).

    With ``bound``, also returns [P, d] worst-case bounds of what rounding
    the softmax weights adds to each output under the variant's weight rule;
    ``v_scale`` [n_cached, H] then gives s_V of each cached row's tile
    (``cached_v_scales``).  The rule: with u = score x log2(e), s_ref the V
    scale of one cached tile of the request, delta_t = log2(s_V,t / s_ref) and
    m a running maximum of u (live keys) and u + delta_t (cached keys), a
    cached key's weight exp2(u + delta_t - m) is stored as E4M3 and multiplies
    its V code, a live key's weight exp2(u - m) / s_ref is stored as bf16 and
    multiplies its V, the sum is scaled by s_ref and divided by
    l = sum exp2(u - m); the output is rounded to bf16.  Then, with
    w_k = exp(s_k - max) and den = sum w_k:
      * an E4M3 weight is off by at most 2^-4 of itself (normal range) plus
        half the subnormal step, 2^-10.  The relative part maps to
        2^-4 w_k |v_kc| / den.  The absolute part maps to
        2^-10 (s_ref / s_V,t) 2^(m - M) |v_kc| / den, M the largest u; m - M
        is at most max_t delta_t, so the factor is at most s_V,max / s_V,t
        (s_ref cancels; s_V,max = the largest V scale of the request's
        cached tiles);
      * a bf16 weight is off by at most 2^-9 of itself: 2^-9 w_k |v_kc| / den;
      * the bf16 output by half an ulp, 2^-9 |o_c|, doubled for margin:
        bound_c = (sum_cache (2^-4 w_k + 2^-10 s_V,max / s_V,t(k)) |v_kc|
                   + sum_live 2^-9 w_k |v_kc|) / den + 2^-8 |o_c|
    (a tile with s_V = 0 holds V = 0 and adds nothing).
    """
    if bound and v_scale is None:
        raise ValueError("the weight-rounding bound needs the cached rows' V tile scales (v_scale)")
    qf = bf16_to_f32(q_l).astype(np.float64)
    kf = bf16_to_f32(k_l).astype(np.float64)
    vf = bf16_to_f32(v_l).astype(np.float64)
    pairs = np.asarray(pairs, np.int64).reshape(-1, 2)
    d = qf.shape[2]
    out = np.zeros((len(pairs), d))
    lse = np.zeros(len(pairs))
    bnd = np.zeros((len(pairs), d))
    n_live = kf.shape[0]
    for p, (i, h) in enumerate(pairs):
        s_live = kf[:, h, :] @ qf[i, h]
        if k_cache_deq.shape[0]:
            codes, sq = quantize_block(bf16_to_f32(q_l[i, h]))
            q_deq = float(sq) * e4m3_decode(codes)
            s_cache = k_cache_deq[:, h, :] @ q_deq
        else:
            s_cache = np.zeros(0)
        sc = np.concatenate([s_live, s_cache]) * scale
        vals = np.concatenate([vf[:, h, :], v_cache_deq[:, h, :]])
        m = sc.max()
        w = np.exp(sc - m)
        den = w.sum()
        out[p] = (w @ vals) / den
        lse[p] = m + np.log(den)
        if bound:
            av = np.abs(vals)
            sv = v_scale[:, h]
            ratio = np.where(sv > 0, (sv.max() if sv.size else 0.0) / np.where(sv > 0, sv, 1.0), 0.0)
            bnd[p] = ((2.0 ** -4 * w[n_live:] + 2.0 ** -10 * ratio) @ av[n_live:]
                      + 2.0 ** -9 * w[:n_live] @ av[:n_live]) / den + 2.0 ** -8 * np.abs(out[p])
    if bound:
        return out, lse, bnd
    return out, lse
