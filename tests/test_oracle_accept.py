"""Pins of the float64 acceptance oracles.

Greedy (Eqs. verify, accept, commit): constructed cases with known answers and
a brute-force sequential scan. Sampling (Leviathan/Chen, cited in Sec. 1-2):
exact enumeration on a 5-token vocabulary against the theorem that the
emitted token is distributed as the target's p, plus limiting cases.
"""
import numpy as np
import pytest

import oracle


def _scan_argmax(row):
    # sequential strict-greater scan: keeps the first of equal maxima
    best, idx = -np.inf, -1
    for i, x in enumerate(row):
        if x > best:
            best, idx = x, i
    return idx


def test_argmax_matches_sequential_scan_with_ties():
    rng = np.random.default_rng(20)
    for _ in range(200):
        row = rng.integers(-3, 4, size=rng.integers(1, 40)).astype(np.float64)
        assert oracle.argmax_lowest(row) == _scan_argmax(row)


def test_signed_zero_is_a_tie():
    row = np.array([-1.0, -0.0, 0.0, -2.0])
    assert oracle.argmax_lowest(row) == 1
    row = np.array([0.0, -0.0])
    assert oracle.argmax_lowest(row) == 0


def test_identical_drafts_commit_k_plus_one():
    rng = np.random.default_rng(21)
    B, K, V = 3, 7, 50
    logits = rng.standard_normal((B, K + 1, V))
    star = logits.argmax(axis=-1)
    n_emit, tokens, r_star = oracle.accept_greedy(logits, star[:, :K])
    assert list(n_emit) == [K + 1] * B
    assert np.array_equal(tokens, star)
    assert np.array_equal(r_star, star)


@pytest.mark.parametrize("ell", range(0, 8))
def test_exact_prefix_length(ell):
    rng = np.random.default_rng(22 + ell)
    K, V = 7, 30
    logits = rng.standard_normal((1, K + 1, V))
    star = logits[0].argmax(axis=-1)
    draft = star[:K].copy()
    if ell < K:
        draft[ell] = (star[ell] + 1) % V
        draft[ell + 1:] = rng.integers(0, V, size=K - ell - 1)
    n_emit, tokens, _ = oracle.accept_greedy(logits, draft[None])
    assert n_emit[0] == ell + 1
    assert list(tokens[0, :ell]) == list(draft[:ell])
    assert tokens[0, ell] == star[ell]
    assert all(t == -1 for t in tokens[0, ell + 1:])


def test_first_mismatch_emits_target_argmax():
    logits = np.zeros((1, 3, 5))
    logits[0, 0, 3] = 1.0
    logits[0, 1, 1] = 1.0
    logits[0, 2, 4] = 1.0
    n_emit, tokens, _ = oracle.accept_greedy(logits, np.array([[2, 1]]))
    assert n_emit[0] == 1 and tokens[0, 0] == 3 and list(tokens[0, 1:]) == [-1, -1]


def test_tied_maxima_resolve_to_lowest_index():
    logits = np.zeros((1, 2, 6))
    logits[0, 0, [2, 4, 5]] = 3.0
    logits[0, 1, [0, 1]] = 1.5
    n_emit, tokens, r_star = oracle.accept_greedy(logits, np.array([[2]]))
    assert list(r_star[0]) == [2, 0]
    assert n_emit[0] == 2 and list(tokens[0]) == [2, 0]
    n_emit, tokens, _ = oracle.accept_greedy(logits, np.array([[4]]))
    assert n_emit[0] == 1 and tokens[0, 0] == 2


def test_k_zero_is_plain_argmax():
    logits = np.array([[[0.1, 0.7, -0.2, 0.7]]])
    n_emit, tokens, _ = oracle.accept_greedy(logits, np.zeros((1, 0), dtype=np.int64))
    assert n_emit[0] == 1 and tokens[0, 0] == 1


# ---------------------------------------------------------------- sampling

def _softmax(z, T):
    e = np.exp((z - z.max()) / T)
    return e / e.sum()


def _enumerate_k1(z_t, z_d, T, N):
    """Output distribution of one draft position + bonus/residual draw, with the
    draft token enumerated (weight q(x)) and both uniforms on an N x N midpoint grid."""
    V = z_t.shape[-1]
    q = _softmax(z_d[0], T)
    grid = (np.arange(N) + 0.5) / N
    u0, u1 = np.meshgrid(grid, grid, indexing="ij")
    u = np.stack([u0.ravel(), u1.ravel()], axis=1)
    n = u.shape[0]
    dist = np.zeros(V)
    accept = 0.0
    for x in range(V):
        zt = np.broadcast_to(z_t, (n,) + z_t.shape)
        zd = np.broadcast_to(z_d, (n,) + z_d.shape)
        n_emit, tokens, _ = oracle.accept_sample(zt, zd, np.full((n, 1), x), u, T)
        out = np.where(n_emit == 2, tokens[:, 0], tokens[:, 0])
        counts = np.bincount(out, minlength=V) / n
        dist += q[x] * counts
        accept += q[x] * np.mean(n_emit == 2)
    return dist, accept


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_first_token_is_distributed_as_target_exact_enumeration(seed):
    # Leviathan/Chen: the first emitted token has law p_0 whatever q is, and the
    # acceptance rate is sum_v min(p, q).
    rng = np.random.default_rng(30 + seed)
    V, T, N = 5, 0.8, 96
    z_t = rng.standard_normal((2, V)) * 1.5
    z_d = rng.standard_normal((1, V)) * 1.5
    dist, acc = _enumerate_k1(z_t, z_d, T, N)
    p = _softmax(z_t[0], T)
    q = _softmax(z_d[0], T)
    np.testing.assert_allclose(dist, p, atol=2.0 / N + 1e-6)
    assert abs(acc - np.minimum(p, q).sum()) <= 1.0 / N + 1e-6


def test_bonus_token_follows_last_target_row():
    # When the draft is accepted the second token is drawn from p_1: with q
    # equal to p_0 every draft is accepted, and the bonus law is p_1.
    rng = np.random.default_rng(40)
    V, T, N = 5, 1.0, 200
    z_t = rng.standard_normal((2, V))
    z_d = z_t[:1].copy()
    u = np.stack([np.full(N, 0.999), (np.arange(N) + 0.5) / N], axis=1)
    n_emit, tokens, _ = oracle.accept_sample(np.broadcast_to(z_t, (N, 2, V)),
                                             np.broadcast_to(z_d, (N, 1, V)),
                                             np.full((N, 1), 2), u, T)
    assert np.all(n_emit == 2) and np.all(tokens[:, 0] == 2)
    freq = np.bincount(tokens[:, 1], minlength=V) / N
    np.testing.assert_allclose(freq, _softmax(z_t[1], T), atol=1.0 / N + 1e-9)


def test_two_positions_joint_law():
    # K = 2 with fixed per-position distributions: the first two emitted tokens
    # (when present) follow p_0 then p_1 given the first was the draft.
    rng = np.random.default_rng(41)
    V, T, N = 5, 0.7, 24
    z_t = rng.standard_normal((3, V))
    z_d = rng.standard_normal((2, V))
    q0, q1 = _softmax(z_d[0], T), _softmax(z_d[1], T)
    p0 = _softmax(z_t[0], T)
    grid = (np.arange(N) + 0.5) / N
    g = np.stack(np.meshgrid(grid, grid, grid, indexing="ij"), axis=-1).reshape(-1, 3)
    n = g.shape[0]
    first = np.zeros(V)
    for x0 in range(V):
        for x1 in range(V):
            w = q0[x0] * q1[x1]
            n_emit, tokens, _ = oracle.accept_sample(np.broadcast_to(z_t, (n, 3, V)),
                                                     np.broadcast_to(z_d, (n, 2, V)),
                                                     np.tile([x0, x1], (n, 1)), g, T)
            first += w * np.bincount(tokens[:, 0], minlength=V) / n
    np.testing.assert_allclose(first, p0, atol=2.0 / N + 1e-6)


def test_equal_distributions_always_accept():
    rng = np.random.default_rng(42)
    B, K, V = 16, 4, 9
    z = rng.standard_normal((B, K + 1, V))
    draft = rng.integers(0, V, size=(B, K))
    u = rng.random((B, K + 1))
    n_emit, tokens, _ = oracle.accept_sample(z, z[:, :K], draft, u, 0.9)
    assert np.all(n_emit == K + 1)
    assert np.array_equal(tokens[:, :K], draft)


def test_low_temperature_agrees_with_greedy():
    # As T -> 0, q is one-hot at argmax z_D, so the proposal is that argmax;
    # p is one-hot at argmax z_T, so the draft is kept iff it is the target's
    # argmax, and the residual (p - q)+ is one-hot at the target's argmax.
    rng = np.random.default_rng(43)
    B, K, V = 12, 5, 40
    z_t = rng.standard_normal((B, K + 1, V))
    z_d = z_t[:, :K] + 0.3 * rng.standard_normal((B, K, V))
    draft = z_d.argmax(-1)
    u = rng.random((B, K + 1))
    n_s, t_s, _ = oracle.accept_sample(z_t, z_d, draft, u, 1e-3)
    assert len(set(n_s.tolist())) > 1
    n_g, t_g, _ = oracle.accept_greedy(z_t, draft)
    assert np.array_equal(n_s, n_g) and np.array_equal(t_s, t_g)


def test_margins_reported_per_decision():
    rng = np.random.default_rng(44)
    z_t = rng.standard_normal((2, 4, 11))
    z_d = rng.standard_normal((2, 3, 11))
    n_emit, _, margins = oracle.accept_sample(z_t, z_d, rng.integers(0, 11, (2, 3)),
                                              rng.random((2, 4)), 1.0)
    for b in range(2):
        # one margin per acceptance test taken plus one for the final draw
        assert len(margins[b]) == min(int(n_emit[b]), 3) + 1
        assert all(m >= 0 for m in margins[b])


def test_inverse_cdf_takes_first_cumulative_sum_strictly_above():
    # Reading of the inverse-CDF draw: the smallest v whose cumulative weight is
    # strictly greater than u * total. With four equal logits p = 1/4 exactly,
    # so u = 0.25 sits on the first step and must yield token 1.
    z = np.zeros((1, 2, 4))
    for u_k, want in [(0.0, 0), (0.25, 1), (0.5, 2), (0.7499, 2), (0.75, 3), (0.999, 3)]:
        n_emit, tokens, _ = oracle.accept_sample(z, z[:, :1], np.array([[1]]),
                                                 np.array([[0.5, u_k]]), 1.0)
        assert n_emit[0] == 2 and tokens[0, 0] == 1 and tokens[0, 1] == want, u_k
