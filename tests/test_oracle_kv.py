"""Pins of the KV-cache append / rollback oracle (Eq. commit)."""
import numpy as np
import pytest

import oracle


def test_append_writes_rows_at_length_and_advances():
    rng = np.random.default_rng(50)
    B, H, cap, D, R = 2, 3, 12, 4, 3
    k = rng.standard_normal((B, H, cap, D))
    v = rng.standard_normal((B, H, cap, D))
    lens = np.array([2, 7])
    kn = rng.standard_normal((B, R, H, D))
    vn = rng.standard_normal((B, R, H, D))
    k2, v2, l2 = oracle.kv_append(k, v, lens, kn, vn)
    assert list(l2) == [5, 10]
    shadow_k, shadow_v = k.copy(), v.copy()
    for b in range(B):
        for i in range(R):
            shadow_k[b, :, lens[b] + i] = kn[b, i]
            shadow_v[b, :, lens[b] + i] = vn[b, i]
    assert np.array_equal(k2, shadow_k) and np.array_equal(v2, shadow_v)


def test_append_beyond_capacity_is_refused():
    k = np.zeros((1, 1, 4, 2))
    with pytest.raises(ValueError):
        oracle.kv_append(k, k, np.array([2]), np.zeros((1, 3, 1, 2)), np.zeros((1, 3, 1, 2)))


def test_rollback_semantics():
    lens = np.array([12, 20, 9])
    assert list(oracle.kv_rollback(lens, [4, 4, 4], 4)) == [12, 20, 9]   # no-op
    assert list(oracle.kv_rollback(lens, [0, 0, 0], 4)) == [8, 16, 5]    # pre-append
    assert list(oracle.kv_rollback(lens, [1, 3, 2], 4)) == [9, 19, 7]
    with pytest.raises(ValueError):
        oracle.kv_rollback(lens, [5, 0, 0], 4)
    with pytest.raises(ValueError):
        oracle.kv_rollback(lens, [-1, 0, 0], 4)
