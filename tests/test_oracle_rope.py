"""Pins of the float64 RoPE / M-RoPE / FlatRoPE oracle (Sec. 3.3, Sec. 4.2).

Each check is a fact the paper or plain mathematics fixes, chosen so that a
wrong sign, a wrong pairing, a wrong frequency exponent or a wrong axis
assignment fails at least one of them.
"""
import math

import numpy as np
import pytest

import oracle


def test_closed_form_d4_base4():
    # D = 4, base 4: theta = (4^0, 4^(-2/4)) = (1, 1/2). At m = 1 the pairs
    # (x0, x1) = (1, 0) and (x2, x3) = (0, 1) rotate by 1 rad and 0.5 rad:
    # (1, 0) -> (cos 1, sin 1) and (0, 1) -> (-sin 0.5, cos 0.5).
    x = np.array([1.0, 0.0, 0.0, 1.0])
    want = np.array([math.cos(1.0), math.sin(1.0), -math.sin(0.5), math.cos(0.5)])
    np.testing.assert_allclose(oracle.rope_1d(x, 1, 4.0), want, rtol=0, atol=1e-15)
    got = oracle.mrope_apply(x, np.array([1, 1, 1]), (1, 1, 0), 0, 4.0)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-15)


def test_closed_form_d4_base100_pos3():
    # base 100: theta = (1, 100^(-1/2)) = (1, 0.1); m = 3 -> angles 3 and 0.3.
    x = np.array([0.5, -2.0, 3.0, 0.25])
    a0, a1 = 3.0, 0.3
    want = np.array([
        0.5 * math.cos(a0) + 2.0 * math.sin(a0),
        0.5 * math.sin(a0) - 2.0 * math.cos(a0),
        3.0 * math.cos(a1) - 0.25 * math.sin(a1),
        3.0 * math.sin(a1) + 0.25 * math.cos(a1),
    ])
    np.testing.assert_allclose(oracle.rope_1d(x, 3, 100.0), want, rtol=0, atol=1e-14)
    for sec, inter in [((2, 0, 0), 0), ((0, 1, 1), 0), ((1, 1, 0), 1)]:
        got = oracle.mrope_apply(x, np.array([3, 3, 3]), sec, inter, 100.0)
        np.testing.assert_allclose(got, want, rtol=0, atol=1e-14)


def test_frequency_schedule_values():
    # theta_d = b^(-2d/h): for h = 8, b = 10000 the schedule is 1, 0.1, 0.01, 0.001.
    np.testing.assert_allclose(oracle.rope_frequencies(8, 10000.0),
                               [1.0, 0.1, 0.01, 0.001], rtol=1e-15)


@pytest.mark.parametrize("inter,expected_axes", [
    (0, [0, 1, 1, 2, 2, 2]),       # blocked, sections (1, 2, 3)
    (1, [0, 1, 2, 0, 1, 2]),       # interleaved: d mod 3
])
def test_axis_assignment_and_support(inter, expected_axes):
    assert list(oracle.axis_assignment(12, (1, 2, 3), inter)) == expected_axes
    rng = np.random.default_rng(0)
    x = rng.standard_normal(12)
    for axis in range(3):
        pos = np.zeros(3, dtype=np.int64)
        pos[axis] = 5
        y = oracle.mrope_apply(x, pos, (1, 2, 3), inter, 10000.0)
        for d in range(6):
            moved = not np.array_equal(y[2 * d:2 * d + 2], x[2 * d:2 * d + 2])
            assert moved == (expected_axes[d] == axis), (axis, d)


def test_position_zero_is_identity():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((3, 5, 128))
    y = oracle.mrope_apply(x, np.zeros((3, 1, 3)), (16, 24, 24), 0, 1e6)
    assert np.array_equal(x, y)


@pytest.mark.parametrize("D,sec", [(64, (8, 12, 12)), (128, (16, 24, 24))])
@pytest.mark.parametrize("inter", [0, 1])
@pytest.mark.parametrize("base", [1e4, 1e6])
def test_mrope_reduces_to_1d_when_coordinates_equal(D, sec, inter, base):
    # Sec. 3.3 / Sec. 4.2: with m^T = m^H = m^W = m, M-RoPE equals 1D RoPE;
    # the 1D side is the explicit block-diagonal matrix of Eq. rope-1d.
    rng = np.random.default_rng(2)
    for m in [0, 1, 7, 544, 4103, 16400]:
        x = rng.standard_normal((4, D))
        got = oracle.mrope_apply(x, np.array([m, m, m]), sec, inter, base)
        np.testing.assert_allclose(got, oracle.rope_1d(x, m, base), rtol=0, atol=1e-12)


def test_rotation_is_orthogonal_and_composes():
    for m1, m2 in [(3, 4), (100, 27), (4000, 96)]:
        r1 = oracle.rope_1d_matrix(m1, 16, 1e6)
        r2 = oracle.rope_1d_matrix(m2, 16, 1e6)
        np.testing.assert_allclose(r1.T @ r1, np.eye(16), atol=1e-13)
        np.testing.assert_allclose(r1 @ r2, oracle.rope_1d_matrix(m1 + m2, 16, 1e6), atol=1e-10)
        assert abs(np.linalg.det(r1) - 1.0) < 1e-12


def test_pair_norms_preserved():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((2, 8, 4, 128))
    pos = rng.integers(0, 20000, size=(2, 8, 1, 3))
    y = oracle.mrope_apply(x, pos, (16, 24, 24), 0, 1e6)
    nx = x[..., 0::2] ** 2 + x[..., 1::2] ** 2
    ny = y[..., 0::2] ** 2 + y[..., 1::2] ** 2
    np.testing.assert_allclose(ny, nx, rtol=1e-12)


@pytest.mark.parametrize("inter", [0, 1])
def test_scores_depend_only_on_relative_position_per_axis(inter):
    # Sec. 4.2 ("Why mirroring is harmful", FlatRoPE (ii)): after rotation the
    # score q.k depends on the coordinate difference of each axis only, so a
    # common shift of one axis leaves it unchanged.
    rng = np.random.default_rng(4)
    q, k = rng.standard_normal(128), rng.standard_normal(128)
    pq, pk = np.array([2, 13, 7]), np.array([0, 4, 30])
    sec = (16, 24, 24)
    base_score = oracle.mrope_apply(q, pq, sec, inter, 1e6) @ oracle.mrope_apply(k, pk, sec, inter, 1e6)
    for axis in range(3):
        for c in [1, 17, 999]:
            sh = np.zeros(3, dtype=np.int64)
            sh[axis] = c
            s = oracle.mrope_apply(q, pq + sh, sec, inter, 1e6) @ oracle.mrope_apply(k, pk + sh, sec, inter, 1e6)
            assert abs(s - base_score) < 1e-10 * max(1.0, abs(base_score))
    # shifting only the query's W coordinate moves the score
    sh = np.array([0, 0, 1])
    s = oracle.mrope_apply(q, pq + sh, sec, inter, 1e6) @ oracle.mrope_apply(k, pk, sec, inter, 1e6)
    assert abs(s - base_score) > 1e-6


def test_flatrope_ignores_section_layout():
    # Sec. 4.2, FlatRoPE (i): with p_T = p_H = p_W = m the section sizes and the
    # interleaved flag are irrelevant, so all layouts agree exactly.
    rng = np.random.default_rng(5)
    x = rng.standard_normal((7, 16, 128))
    pos = oracle.flatrope_positions(np.arange(4096, 4103))[:, None, :]
    ref = oracle.mrope_apply(x, pos, (16, 24, 24), 0, 1e6)
    for sec, inter in [((64, 0, 0), 0), ((0, 0, 64), 0), ((20, 22, 22), 1), ((16, 24, 24), 1)]:
        assert np.array_equal(oracle.mrope_apply(x, pos, sec, inter, 1e6), ref)


def test_sections_must_sum_to_half_dim():
    with pytest.raises(ValueError):
        oracle.axis_assignment(128, (16, 24, 23), 0)
