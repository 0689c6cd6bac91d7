"""Pins of the CPU oracle against things other than itself.

  * a library routine: torch's scaled_dot_product_attention in float64
    (the all-visible mask must reduce to standard softmax attention);
  * closed forms: with scale 0 every row returns the mean of the values it can
    see, so the visible set itself is checked; a single visible key returns
    that key's value; the LSE equals scipy's logsumexp of the scores;
  * the paper's block visibility (golden text restated from Sec. 3.3);
  * brute force with an explicit N x N mask on tiny ragged inputs;
  * the exact-caching invariant of Sec. 3.1 / 3.3: reference-row outputs and
    cached K/V do not change, bit for bit, when LT/X inputs change.
"""
import numpy as np
import pytest
import torch
from scipy.special import logsumexp

import workloads

BLOCKS = ("LT", "X", "ST", "R")
MODES = ("beyond", "beyond_alt", "isolated", "full")


def rand_bits(rng, shape):
    x = torch.from_numpy(rng.standard_normal(shape).astype(np.float32)).to(torch.bfloat16)
    return workloads.bf16_bits(x)


def to_f64(bits):
    return torch.from_numpy(bits.astype(np.int16)).view(torch.bfloat16).to(torch.float64)


def explicit_mask(rel, mode, n_lt, n_x, n_st, n_r):
    lens = (n_lt, n_x, n_st, n_r)
    blk = np.concatenate([np.full(n, i, np.int64) for i, n in enumerate(lens)])
    n = blk.size
    m = np.zeros((n, n), bool)
    for i in range(n):
        for j in range(n):
            m[i, j] = rel[(mode, BLOCKS[blk[i]], BLOCKS[blk[j]])]
    return m


def sdpa64(q, k, v, mask, scale):
    """torch SDPA in float64, heads first; rows without a visible key -> 0."""
    Q, K, V = (to_f64(a).permute(1, 0, 2) for a in (q, k, v))
    am = None if mask is None else torch.from_numpy(mask)
    o = torch.nn.functional.scaled_dot_product_attention(Q, K, V, attn_mask=am, scale=scale)
    return o.permute(1, 0, 2).numpy()


def test_block_table_matches_paper(oracle_mod, paper_relations):
    for (mode, qb, kb), bit in paper_relations.items():
        assert oracle_mod.block_visible(mode, qb, kb) == bit, (mode, qb, kb)


@pytest.mark.parametrize("H,d,n", [(1, 8, 1), (2, 16, 7), (3, 64, 33), (2, 128, 70)])
def test_all_visible_equals_standard_attention(oracle_mod, H, d, n):
    rng = np.random.default_rng(n)
    q, k, v = (rand_bits(rng, (n, H, d)) for _ in range(3))
    scale = 1.0 / np.sqrt(d)
    out, lse = oracle_mod.full(q, k, v, scale)
    ref = sdpa64(q, k, v, None, scale)
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)
    s = np.einsum("ihc,jhc->hij", to_f64(q).numpy(), to_f64(k).numpy()) * scale
    np.testing.assert_allclose(lse, logsumexp(s, axis=2).T, rtol=0, atol=1e-12)


@pytest.mark.parametrize("mode", ["beyond", "beyond_alt", "isolated", "full"])
def test_explicit_mask_brute_force_matches_library(oracle_mod, paper_relations, mode):
    rng = np.random.default_rng(7)
    n_lt, n_x, n_st, n_r = 5, 9, (3 if mode in ("beyond", "beyond_alt") else 0), 11
    n = n_lt + n_x + n_st + n_r
    H, d = 2, 32
    q, k, v = (rand_bits(rng, (n, H, d)) for _ in range(3))
    m = explicit_mask(paper_relations, mode, n_lt, n_x, n_st, n_r)
    out, _ = oracle_mod.attention_explicit_mask(q, k, v, m, 0.125)
    np.testing.assert_allclose(out, sdpa64(q, k, v, m, 0.125), rtol=0, atol=1e-12)


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("seed", range(6))
def test_joint_matches_explicit_mask_on_ragged_tiny(oracle_mod, paper_relations, mode, seed):
    rng = np.random.default_rng(100 + seed)
    lens = [int(x) for x in rng.integers(0, 9, size=4)]
    lens[3] = max(lens[3], 1)
    if mode in ("isolated", "full"):
        lens[2] = 0
    n_lt, n_x, n_st, n_r = lens
    n = sum(lens)
    H, d = 2, 16
    q, k, v = (rand_bits(rng, (n, H, d)) for _ in range(3))
    m = explicit_mask(paper_relations, mode, *lens)
    out_j, lse_j = oracle_mod.joint_attention(q, k, v, *lens, mode, 0.25)
    out_b, lse_b = oracle_mod.attention_explicit_mask(q, k, v, m, 0.25)
    np.testing.assert_array_equal(out_j, out_b)
    np.testing.assert_array_equal(lse_j, lse_b)


@pytest.mark.parametrize("mode", MODES)
def test_scale_zero_returns_mean_of_visible_values(oracle_mod, paper_relations, mode):
    """Closed form: with zero scores the softmax is uniform over visible keys."""
    rng = np.random.default_rng(3)
    lens = (4, 6, 0 if mode in ("isolated", "full") else 3, 5)
    n = sum(lens)
    H, d = 3, 8
    q, k, v = (rand_bits(rng, (n, H, d)) for _ in range(3))
    out, lse = oracle_mod.joint_attention(q, k, v, *lens, mode, 0.0)
    m = explicit_mask(paper_relations, mode, *lens)
    vf = to_f64(v).numpy()
    for i in range(n):
        vis = np.nonzero(m[i])[0]
        np.testing.assert_allclose(out[i], vf[vis].mean(axis=0), rtol=0, atol=1e-14)
        np.testing.assert_allclose(lse[i], np.log(len(vis)), rtol=0, atol=1e-14)


def test_single_visible_key_returns_its_value(oracle_mod):
    rng = np.random.default_rng(4)
    H, d, nq, nk = 2, 16, 5, 9
    q, = (rand_bits(rng, (nq, H, d)),)
    k, v = rand_bits(rng, (nk, H, d)), rand_bits(rng, (nk, H, d))
    m = np.zeros((nq, nk), bool)
    for i in range(nq):
        m[i, (3 * i + 1) % nk] = True
    out, _ = oracle_mod.attention_explicit_mask(q, k, v, m, 0.3)
    vf = to_f64(v).numpy()
    for i in range(nq):
        np.testing.assert_array_equal(out[i], vf[(3 * i + 1) % nk])


def test_row_without_visible_key_is_zero_with_minus_inf_lse(oracle_mod):
    rng = np.random.default_rng(5)
    q, k, v = (rand_bits(rng, (3, 1, 8)) for _ in range(3))
    m = np.ones((3, 3), bool)
    m[1] = False
    out, lse = oracle_mod.attention_explicit_mask(q, k, v, m, 1.0)
    assert (out[1] == 0).all() and np.isneginf(lse[1]).all()
    assert np.isfinite(lse[0]).all()


def test_key_permutation_invariance(oracle_mod):
    rng = np.random.default_rng(6)
    H, d, n = 2, 32, 40
    q, k, v = (rand_bits(rng, (n, H, d)) for _ in range(3))
    perm = rng.permutation(n)
    a, la = oracle_mod.attention_explicit_mask(q, k, v, None, 0.2)
    b, lb = oracle_mod.attention_explicit_mask(q, k[perm], v[perm], None, 0.2)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-13)
    np.testing.assert_allclose(la, lb, rtol=0, atol=1e-13)


@pytest.mark.parametrize("mode", ["beyond", "beyond_alt", "isolated"])
def test_exact_caching_invariant(oracle_mod, mode):
    """Sec. 3.1 / 3.3: with LT and X_t inputs changed, every ST and R row
    output is bit-identical and every LT/X row changes."""
    rng = np.random.default_rng(8)
    lens = (7, 13, 0 if mode == "isolated" else 5, 17)
    n_lt, n_x, n_st, n_r = lens
    n, H, d = sum(lens), 2, 32
    q, k, v = (rand_bits(rng, (n, H, d)) for _ in range(3))
    q2, k2, v2 = q.copy(), k.copy(), v.copy()
    live = slice(0, n_lt + n_x)
    for a in (q2, k2, v2):
        a[live] = rand_bits(rng, a[live].shape)
    o1, l1 = oracle_mod.joint_attention(q, k, v, *lens, mode, 0.177)
    o2, l2 = oracle_mod.joint_attention(q2, k2, v2, *lens, mode, 0.177)
    st_r = slice(n_lt + n_x, n)
    np.testing.assert_array_equal(o1[st_r], o2[st_r])
    np.testing.assert_array_equal(l1[st_r], l2[st_r])
    assert (np.abs(o1[live] - o2[live]).max(axis=(1, 2)) > 0).all()


@pytest.mark.parametrize("mode", ["beyond", "beyond_alt", "isolated"])
def test_prefill_cache_and_step_agree_with_joint(oracle_mod, mode):
    """(c) cached K/V equal the reference K/V given; the prefill rows and the
    step rows computed from the cache equal the joint sequence's rows."""
    rng = np.random.default_rng(9)
    n_lt, n_x, n_st, n_r = 6, 10, (0 if mode == "isolated" else 4), 12
    H, d = 2, 16
    n = n_lt + n_x + n_st + n_r
    q, k, v = (rand_bits(rng, (n, H, d)) for _ in range(3))
    s0 = n_lt + n_x
    o_p, l_p, kc, vc = oracle_mod.prefill(q[s0:], k[s0:], v[s0:], n_st, n_r, mode, 0.3)
    keep = 0 if mode == "beyond_alt" else n_st
    np.testing.assert_array_equal(kc, k[s0 + keep:])
    np.testing.assert_array_equal(vc, v[s0 + keep:])
    o_j, l_j = oracle_mod.joint_attention(q, k, v, n_lt, n_x, n_st, n_r, mode, 0.3)
    np.testing.assert_array_equal(o_p, o_j[s0:])
    np.testing.assert_array_equal(l_p, l_j[s0:])
    o_s, l_s = oracle_mod.step(q[:s0], k[:s0], v[:s0], kc, vc, n_lt, n_x, n_st, n_r, mode, 0.3)
    np.testing.assert_array_equal(o_s, o_j[:s0])
    np.testing.assert_array_equal(l_s, l_j[:s0])


def test_sampled_pairs_equal_full_computation(oracle_mod):
    rng = np.random.default_rng(10)
    lens = (5, 9, 3, 11)
    n, H, d = sum(lens), 3, 16
    q, k, v = (rand_bits(rng, (n, H, d)) for _ in range(3))
    o, l = oracle_mod.joint_attention(q, k, v, *lens, "beyond", 0.25)
    pairs = np.array([(i, h) for i in range(0, n, 3) for h in range(H)], np.int32)
    po, pl = oracle_mod.joint_attention(q, k, v, *lens, "beyond", 0.25, pairs=pairs)
    np.testing.assert_array_equal(po, o[pairs[:, 0], pairs[:, 1]])
    np.testing.assert_array_equal(pl, l[pairs[:, 0], pairs[:, 1]])
