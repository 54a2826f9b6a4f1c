"""Pins of the float64 attention-budget oracle (Sec. 4.2, Table tab:attn-budget).

Checked against closed forms (uniform scores, a dominating key, two keys)
and against verify_attention -- itself pinned to torch's float64
scaled_dot_product_attention -- with one-hot segment indicators as values.
"""
import numpy as np
import pytest

import oracle


def _case(rng, B, R, Hq, Hkv, D, prefix, n_vis, cap):
    q = rng.standard_normal((B, R, Hq, D))
    k = rng.standard_normal((B, Hkv, cap, D))
    return q, k, np.asarray(prefix) + R, np.asarray(n_vis)


def test_masses_sum_to_one_and_are_nonnegative():
    rng = np.random.default_rng(1)
    q, k, lens, nv = _case(rng, 2, 4, 4, 2, 16, [20, 7], [12, 0], 40)
    mass, ent = oracle.attention_budget(q, k, lens, nv)
    assert np.allclose(mass.sum(-1), 1.0, atol=1e-12)
    assert (mass >= 0).all() and ((ent >= 0) & (ent <= 1 + 1e-12)).all()


def test_uniform_scores_give_segment_sizes_and_entropy_one():
    # q = 0: every visible key scores 0, so the softmax is uniform
    B, R, Hq, Hkv, D, L, nv = 1, 3, 2, 1, 8, 10, 6
    q = np.zeros((B, R, Hq, D))
    k = np.random.default_rng(2).standard_normal((B, Hkv, L + R, D))
    mass, ent = oracle.attention_budget(q, k, [L + R], [nv])
    for i in range(R):
        n = L + i + 1
        assert np.allclose(mass[0, i, :, 0], nv / n)
        assert np.allclose(mass[0, i, :, 1], (L - nv) / n)
        assert np.allclose(mass[0, i, :, 2], (i + 1) / n)
        assert np.allclose(ent[0, i], 1.0)


def test_dominating_key_takes_all_mass_and_zero_entropy():
    rng = np.random.default_rng(3)
    B, R, Hq, Hkv, D, L, nv = 1, 2, 1, 1, 16, 12, 5
    q = rng.standard_normal((B, R, Hq, D))
    k = rng.standard_normal((B, Hkv, L + R, D)) * 0.01
    # key 8 (trajectory / text segment) aligned with both rows' queries, scores ~ +400
    k[0, 0, 8] = 50.0 * (q[0, 0, 0] + q[0, 1, 0])
    mass, ent = oracle.attention_budget(q, k, [L + R], [nv])
    assert np.allclose(mass[0, :, 0, 1], 1.0, atol=1e-9)
    assert np.allclose(ent[0, :, 0], 0.0, atol=1e-6)


def test_two_nonvisual_keys_binary_entropy():
    # prefix = 1 text key, R = 1: the non-visual keys are that key and the row
    # itself; entropy = binary entropy of their renormalised weights / ln 2
    rng = np.random.default_rng(4)
    D = 8
    q = rng.standard_normal((1, 1, 1, D))
    k = rng.standard_normal((1, 1, 4, D))
    nv = 0
    mass, ent = oracle.attention_budget(q, k, [2], [nv])
    s = np.array([k[0, 0, 0] @ q[0, 0, 0], k[0, 0, 1] @ q[0, 0, 0]]) / np.sqrt(D)
    p = np.exp(s - s.max())
    p /= p.sum()
    h2 = -(p * np.log(p)).sum() / np.log(2)
    assert np.isclose(ent[0, 0, 0], h2, atol=1e-12)
    assert np.isclose(mass[0, 0, 0, 1], p[0]) and np.isclose(mass[0, 0, 0, 2], p[1])


def test_masses_equal_attention_with_indicator_values():
    # verify_attention with v[n] = one-hot(segment of key n) returns the masses
    rng = np.random.default_rng(5)
    B, R, Hq, Hkv, D = 2, 5, 4, 2, 16
    prefix, nvis, cap = [30, 11], [17, 11], 40
    q, k, lens, nv = _case(rng, B, R, Hq, Hkv, D, prefix, nvis, cap)
    v = np.zeros((B, Hkv, cap, D))
    for b in range(B):
        v[b, :, :nvis[b], 0] = 1.0
        v[b, :, nvis[b]:prefix[b], 1] = 1.0
        v[b, :, prefix[b]:, 2] = 1.0
    mass, _ = oracle.attention_budget(q, k, lens, nv)
    out = oracle.verify_attention(q, k, v, lens)
    assert np.allclose(out[..., :3], mass, atol=1e-12)


@pytest.mark.parametrize("bad", [-1, 31])
def test_visual_count_outside_the_prefix_is_rejected(bad):
    q = np.zeros((1, 1, 1, 4))
    k = np.zeros((1, 1, 40, 4))
    with pytest.raises(ValueError):
        oracle.attention_budget(q, k, [31], [bad])
