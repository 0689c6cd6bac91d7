"""Pins of the FP8 reference-cache oracle (``oracle/fp8.py``) against things
other than itself:

  * the E4M3 format's closed forms (named codes, monotone order, the
    subnormal step) and a library decoder/encoder (torch.float8_e4m3fn);
  * brute force: the encoder returns the nearest representable value, ties
    to the even mantissa, checked by exhaustive search over all 256 codes;
  * the quantisation rule's invariants: the block maximum maps to +-448, the
    relative error of a normal-range value is at most 2^-4;
  * the exact oracle (oracle.c): where every quantised value is already on
    the E4M3 grid with a power-of-two scale the quantisation is lossless, and
    the FP8 step must equal the exact step;
  * the parity tolerance of the CUDA path (which also rounds the softmax
    weights of cached keys to E4M3 and those of live keys to bf16): the error
    that rounding adds is simulated here on the test shapes and must stay
    well inside the tolerance the GPU tests use.
"""
import numpy as np
import pytest
import torch

import workloads
from oracle import fp8

# Tolerance of the CUDA FP8-cache path against this oracle (tests/test_gpu_fp8.py):
# every output within the oracle's worst-case weight-rounding bound (plus
# FP8_SLACK for fp32 arithmetic), and for requests with at least
# FP8_STAT_MIN_KEYS cached keys, where the rounding errors average out, the
# statistical bounds below (simulated here on such shapes).
FP8_MAX_ABS = 3e-2
FP8_MEAN_ABS = 4e-3
FP8_SLACK = 1e-3
FP8_STAT_MIN_KEYS = 384


def test_named_codes_decode_to_closed_forms():
    named = {0x00: 0.0, 0x01: 2.0 ** -9, 0x07: 7 * 2.0 ** -9, 0x08: 2.0 ** -6, 0x38: 1.0, 0x3F: 1.875,
             0x40: 2.0, 0x77: 240.0, 0x7E: 448.0, 0x80: -0.0, 0xB8: -1.0, 0xFE: -448.0}
    for c, v in named.items():
        assert fp8.e4m3_decode(np.uint8(c)) == v, hex(c)
    assert np.isnan(fp8.e4m3_decode(np.uint8(0x7F))) and np.isnan(fp8.e4m3_decode(np.uint8(0xFF)))
    pos = fp8.e4m3_decode(np.arange(0x7F, dtype=np.uint8))
    assert np.all(np.diff(pos) > 0)  # codes 0x00..0x7E are increasing
    # subnormal step 2^-9 continues into the first binade without a gap
    assert np.allclose(np.diff(pos[:16]), 2.0 ** -9)


def test_decode_matches_library_for_all_codes():
    codes = torch.arange(256, dtype=torch.int32).to(torch.uint8)
    lib = codes.view(torch.float8_e4m3fn).to(torch.float64).numpy()
    ours = fp8.e4m3_decode(codes.numpy())
    assert np.array_equal(np.isnan(lib), np.isnan(ours))
    ok = ~np.isnan(lib)
    assert np.array_equal(lib[ok], ours[ok])


def test_encode_round_trips_every_finite_code():
    codes = np.array([c for c in range(256) if c not in (0x7F, 0xFF)], np.uint8)
    vals = fp8.e4m3_decode(codes).astype(np.float32)
    back = fp8.e4m3_encode(vals)
    # -0.0 encodes to 0x80 and +0.0 to 0x00, so every code comes back
    assert np.array_equal(back, codes)


def _brute_force_encode(x):
    grid_codes = np.arange(0x7F, dtype=np.uint8)
    grid = fp8.e4m3_decode(grid_codes)
    out = []
    for v in np.asarray(x, np.float64):
        a = min(abs(v), 448.0)
        dist = np.abs(grid - a)
        best = np.flatnonzero(dist == dist.min())
        c = int(grid_codes[best[0]]) if len(best) == 1 else int([b for b in grid_codes[best] if b % 2 == 0][0])
        out.append(c | (0x80 if np.signbit(v) else 0))
    return np.array(out, np.uint8)


def test_encode_is_nearest_value_ties_to_even():
    rng = np.random.default_rng(11)
    grid = fp8.e4m3_decode(np.arange(0x7F, dtype=np.uint8))
    mids = ((grid[:-1] + grid[1:]) / 2).astype(np.float32)  # exact ties (all representable in fp32)
    rand = (rng.standard_normal(3000) * np.exp2(rng.integers(-12, 9, 3000))).astype(np.float32)
    x = np.concatenate([mids, -mids, rand, np.float32([449.0, 464.0, 1e6, -1e9])])
    assert np.array_equal(fp8.e4m3_encode(x), _brute_force_encode(x))


def test_encode_matches_library_in_range():
    rng = np.random.default_rng(12)
    x = (rng.standard_normal(20000) * np.exp2(rng.integers(-14, 8, 20000))).astype(np.float32)
    x = np.clip(x, -448, 448)
    lib = torch.from_numpy(x).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(fp8.e4m3_encode(x), lib)


def test_quantize_block_rule():
    rng = np.random.default_rng(13)
    x = rng.standard_normal((128, 64)).astype(np.float32)
    codes, s = fp8.quantize_block(x)
    assert s == np.float32(np.float32(np.abs(x).max()) / np.float32(448.0))
    i = np.unravel_index(np.argmax(np.abs(x)), x.shape)
    assert codes[i] in (0x7E, 0xFE)
    deq = float(s) * fp8.e4m3_decode(codes)
    normal = np.abs(x) * (448.0 / np.abs(x).max()) >= 2.0 ** -6
    rel = np.abs(deq - x)[normal] / np.abs(x)[normal]
    assert rel.max() <= 2.0 ** -4 * (1 + 1e-6)
    z, sz = fp8.quantize_block(np.zeros((4, 4), np.float32))
    assert sz == 0 and not z.any()


def _grid_values(rng, shape, blocks_axis_sizes):
    """bf16 bit patterns whose values are 2^-6 x E4M3 values with |code value| <= 16,
    plus one +-448 x 2^-6 element per quantisation block (so every block's scale
    is exactly 2^-6 and the quantisation is lossless)."""
    small = np.array([c for c in range(0x00, 0x5B)], np.uint8)  # decoded magnitudes <= 16
    codes = rng.choice(small, size=shape) | (rng.integers(0, 2, size=shape).astype(np.uint8) << 7)
    vals = fp8.e4m3_decode(codes) * 2.0 ** -6
    blocks_axis_sizes(vals, rng)
    t = torch.from_numpy(vals.astype(np.float32)).to(torch.bfloat16)
    assert torch.equal(t.to(torch.float64), torch.from_numpy(vals))  # exactly representable in bf16
    return workloads.bf16_bits(t)


def _big_per_tile(seg_lens):
    def put(vals, rng):
        H, d = vals.shape[1], vals.shape[2]
        src = 0
        for n in seg_lens:
            for t0 in range(0, n, fp8.TILE):
                rows = min(fp8.TILE, n - t0)
                for h in range(H):
                    r = src + t0 + int(rng.integers(0, rows))
                    vals[r, h, int(rng.integers(0, d))] = 448.0 * 2.0 ** -6 * (1 if rng.random() < 0.5 else -1)
            src += n
    return put


def _big_per_row(vals, rng):
    n, H, d = vals.shape
    for i in range(n):
        for h in range(H):
            vals[i, h, int(rng.integers(0, d))] = 448.0 * 2.0 ** -6 * (1 if rng.random() < 0.5 else -1)


def test_cache_layout_and_lossless_round_trip():
    rng = np.random.default_rng(14)
    seg = [300, 0, 128, 5]
    H, d = 3, 128
    k = _grid_values(rng, (sum(seg), H, d), _big_per_tile(seg))
    v = _grid_values(rng, (sum(seg), H, d), _big_per_tile(seg))
    k8, vt8, scales, seg_off = fp8.build_fp8_cache(k, v, seg)
    assert seg_off == [0, 384, 384, 512] and k8.shape == (640, H, d) and vt8.shape == (H, d, 640)
    assert np.all(scales[[0, 1, 2, 3, 4]] == np.float32(2.0 ** -6))
    kd, vd = fp8.dequantized_cache(k8, vt8, scales, seg_off, seg)
    assert np.array_equal(kd, fp8.bf16_to_f32(k).astype(np.float64))
    assert np.array_equal(vd, fp8.bf16_to_f32(v).astype(np.float64))
    # pad rows of every tile hold code 0
    for lo, hi in ((300, 384), (512 + 5, 640)):
        assert not k8[lo:hi].any() and not vt8[:, :, lo:hi].any()


@pytest.mark.parametrize("mode", ["beyond", "beyond_alt"])
def test_lossless_fp8_step_equals_exact_step(oracle_mod, mode):
    """Grid-valued inputs: the quantised step must reproduce the exact oracle."""
    rng = np.random.default_rng(15 if mode == "beyond" else 16)
    n_st, n_lt, n_x, n_r = 7, 9, 150, 260
    H, d = 2, 128
    cached = n_st + n_r if mode == "beyond_alt" else n_r
    q_l = _grid_values(rng, (n_lt + n_x, H, d), _big_per_row)
    k_l = _grid_values(rng, (n_lt + n_x, H, d), _big_per_row)
    v_l = _grid_values(rng, (n_lt + n_x, H, d), _big_per_row)
    k_c = _grid_values(rng, (cached, H, d), _big_per_tile([cached]))
    v_c = _grid_values(rng, (cached, H, d), _big_per_tile([cached]))
    scale = 1.0 / np.sqrt(d)
    k8, vt8, scales, off = fp8.build_fp8_cache(k_c, v_c, [cached])
    kd, vd = fp8.dequantized_cache(k8, vt8, scales, off, [cached])
    pairs = np.array([(i, h) for i in range(0, n_lt + n_x, 7) for h in range(H)])
    o8, l8 = fp8.step_fp8(q_l, k_l, v_l, kd, vd, scale, pairs)
    o, l = oracle_mod.step(q_l, k_l, v_l, k_c, v_c, n_lt, n_x, n_st, n_r, mode, scale, pairs)
    np.testing.assert_allclose(o8, o, rtol=0, atol=1e-12)
    np.testing.assert_allclose(l8, l, rtol=0, atol=1e-12)


def _fp8_case(seed, n_live, n_cached, H=2, d=128):
    rng = np.random.default_rng(seed)
    bits = lambda n: workloads.bf16_bits(torch.from_numpy(rng.standard_normal((n, H, d)).astype(np.float32))  # noqa: E731
                                         .to(torch.bfloat16))
    q_l, k_l, v_l, k_c, v_c = bits(n_live), bits(n_live), bits(n_live), bits(n_cached), bits(n_cached)
    k8, vt8, sc, off = fp8.build_fp8_cache(k_c, v_c, [n_cached])
    kd, vd = fp8.dequantized_cache(k8, vt8, sc, off, [n_cached])
    return q_l, k_l, v_l, k_c, v_c, kd, vd, fp8.cached_v_scales(sc, off, [n_cached])


def test_fp8_step_close_to_exact_step(oracle_mod):
    """The approximation itself: N(0,1) inputs, error of the quantised step."""
    q_l, k_l, v_l, k_c, v_c, kd, vd, _ = _fp8_case(17, 96, 700)
    pairs = np.array([(i, h) for i in range(0, 96, 5) for h in range(2)])
    scale = 1.0 / np.sqrt(128)
    o8, l8 = fp8.step_fp8(q_l, k_l, v_l, kd, vd, scale, pairs)
    o, l = oracle_mod.step(q_l, k_l, v_l, k_c, v_c, 0, 96, 0, 700, "beyond", scale, pairs)
    err = np.abs(o8 - o)
    assert err.max() < 2e-2 and err.mean() < 2e-3
    assert np.abs(l8 - l).max() < 2e-2


def _weights_rounded(q_l, k_l, v_l, kd, vd, vsc, scale, pairs, lag=0.0):
    """The CUDA path's extra rounding, simulated by the variant's weight rule
    (reading R12): scores in log2 units u, s_ref = the first cached tile's V
    scale, delta = log2(s_V,t / s_ref) per cached tile, m = max over the live
    u and the cached u + delta, lowered by ``lag`` (the running maximum may
    trail the true one by up to 8 before a rescale); cached weights
    exp2(u + delta - m) rounded to E4M3 times the V codes, live weights
    exp2(u - m) / s_ref rounded to bf16 times V, the sum times s_ref over the
    unrounded l = sum exp2(u - m)."""
    qf = fp8.bf16_to_f32(q_l).astype(np.float64)
    kf = fp8.bf16_to_f32(k_l).astype(np.float64)
    vf = fp8.bf16_to_f32(v_l).astype(np.float64)
    out = np.zeros((len(pairs), qf.shape[2]))
    n_live = kf.shape[0]
    for p, (i, h) in enumerate(pairs):
        codes, sq = fp8.quantize_block(fp8.bf16_to_f32(q_l[i, h]))
        u = np.concatenate([kf[:, h] @ qf[i, h], kd[:, h] @ (float(sq) * fp8.e4m3_decode(codes))]) * scale
        u = u * np.log2(np.e)
        sv = vsc[:, h]
        s_ref = sv[0] if sv.size and sv[0] > 0 else 1.0
        delta = np.where(sv > 0, np.log2(np.where(sv > 0, sv, 1.0) / s_ref), 0.0)
        m = max(u[:n_live].max(initial=-np.inf), (u[n_live:] + delta).max(initial=-np.inf)) - lag
        l = np.exp2(u - m).sum()
        w_live = np.exp2(u[:n_live] - m) / s_ref
        w_live = torch.from_numpy(w_live.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
        w_cache = fp8.e4m3_decode(fp8.e4m3_encode(np.exp2(u[n_live:] + delta - m).astype(np.float32)))
        codes_v = np.where(sv[:, None] > 0, vd[:, h] / np.where(sv > 0, sv, 1.0)[:, None], 0.0)
        out[p] = s_ref * (w_live @ vf[:, h] + w_cache @ codes_v) / l
    return out


def test_weight_rounding_bound_on_few_keys():
    """With a handful of keys the statistical tolerance does not apply; the
    worst-case bound must still hold, and be reached within a factor of ten."""
    worst = 0.0
    for seed in range(6):
        q_l, k_l, v_l, k_c, v_c, kd, vd, vsc = _fp8_case(40 + seed, 2, 5)
        pairs = np.array([(i, h) for i in range(2) for h in range(2)])
        o8, _, bnd = fp8.step_fp8(q_l, k_l, v_l, kd, vd, 1.0 / np.sqrt(128), pairs, bound=True, v_scale=vsc)
        sim = _weights_rounded(q_l, k_l, v_l, kd, vd, vsc, 1.0 / np.sqrt(128), pairs)
        err = np.abs(sim - o8)
        assert np.all(err <= bnd)
        worst = max(worst, float((err / bnd).max()))
    assert worst > 0.1


@pytest.mark.parametrize("n_live,n_cached", [(64, 400), (96, 1024), (300, 2048)])
def test_gpu_fp8_tolerance_covers_weight_rounding(n_live, n_cached):
    q_l, k_l, v_l, k_c, v_c, kd, vd, vsc = _fp8_case(18 + n_cached, n_live, n_cached)
    pairs = np.array([(i, h) for i in range(0, n_live, 3) for h in range(2)])
    scale = 1.0 / np.sqrt(128)
    o8, _, bnd = fp8.step_fp8(q_l, k_l, v_l, kd, vd, scale, pairs, bound=True, v_scale=vsc)
    sim = _weights_rounded(q_l, k_l, v_l, kd, vd, vsc, scale, pairs)
    err = np.abs(sim - o8)
    assert np.all(err <= bnd)  # the analytic worst case holds
    lagged = _weights_rounded(q_l, k_l, v_l, kd, vd, vsc, scale, pairs, lag=8.0)
    assert np.all(np.abs(lagged - o8) <= bnd)  # and with the running maximum trailing by 2^8
    # the rounding error must sit well inside the tolerance (margin for fp32
    # arithmetic, the bf16 output and rows the sample did not draw)
    assert err.max() < FP8_MAX_ABS / 2
    assert err.mean() < FP8_MEAN_ABS / 2


@pytest.mark.parametrize("first_tile_gain", [1.0 / 16, 16.0])
def test_weight_rounding_bound_with_uneven_v_scales(first_tile_gain):
    """V tiles whose scales differ by 16x (the first tile, whose scale is
    s_ref, the smallest or the largest): the bound's absolute term, which
    scales with s_V,max / s_V,t, must still cover the variant's rounding, with
    the running maximum exact or trailing by 2^8."""
    rng = np.random.default_rng(77 if first_tile_gain < 1 else 78)
    H, d, n_live, n_cached = 2, 128, 24, 3 * fp8.TILE
    bits = lambda x: workloads.bf16_bits(torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16))  # noqa: E731
    q_l, k_l, v_l = (bits(rng.standard_normal((n_live, H, d))) for _ in range(3))
    k_c = bits(2.0 * rng.standard_normal((n_cached, H, d)))  # peaked softmax: many subnormal weights
    v = rng.standard_normal((n_cached, H, d))
    v[:fp8.TILE] *= first_tile_gain
    v_c = bits(v)
    k8, vt8, sc, off = fp8.build_fp8_cache(k_c, v_c, [n_cached])
    kd, vd = fp8.dequantized_cache(k8, vt8, sc, off, [n_cached])
    vsc = fp8.cached_v_scales(sc, off, [n_cached])
    pairs = np.array([(i, h) for i in range(0, n_live, 2) for h in range(H)])
    scale = 1.0 / np.sqrt(d)
    o8, _, bnd = fp8.step_fp8(q_l, k_l, v_l, kd, vd, scale, pairs, bound=True, v_scale=vsc)
    for lag in (0.0, 8.0):
        sim = _weights_rounded(q_l, k_l, v_l, kd, vd, vsc, scale, pairs, lag=lag)
        assert np.all(np.abs(sim - o8) <= bnd), f"lag {lag}"
