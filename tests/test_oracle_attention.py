"""Pins of the float64 verify-attention oracle (Eq. verify, Sec. 3.2).

The oracle is checked against torch's float64 scaled_dot_product_attention
(a library routine) with a causal mask built here from the reading "row i
sees keys 0 .. L_b + i", and against special cases with closed-form answers.
"""
import numpy as np
import pytest
import torch

import oracle


def _random_case(rng, B, R, Hq, Hkv, D, prefix, cap):
    q = rng.standard_normal((B, R, Hq, D))
    k = rng.standard_normal((B, Hkv, cap, D))
    v = rng.standard_normal((B, Hkv, cap, D))
    lens = np.asarray(prefix) + R
    return q, k, v, lens


def _sdpa_reference(q, k, v, lens):
    B, R, Hq, D = q.shape
    Hkv = k.shape[1]
    G = Hq // Hkv
    out = np.zeros_like(q)
    for b in range(B):
        n = int(lens[b])
        L = n - R
        qt = torch.from_numpy(q[b]).permute(1, 0, 2)                     # [Hq, R, D]
        kt = torch.from_numpy(k[b, :, :n]).repeat_interleave(G, dim=0)   # [Hq, n, D]
        vt = torch.from_numpy(v[b, :, :n]).repeat_interleave(G, dim=0)
        mask = torch.zeros(R, n, dtype=torch.bool)
        for i in range(R):
            mask[i, :L + i + 1] = True
        o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask)
        out[b] = o.permute(1, 0, 2).numpy()
    return out


@pytest.mark.parametrize("B,R,Hq,Hkv,D,prefix", [
    (1, 5, 4, 1, 64, [37]),
    (2, 8, 8, 2, 32, [100, 61]),
    (3, 1, 4, 4, 16, [0, 5, 12]),       # K = 0 (plain decode), G = 1 (MHA)
    (2, 17, 4, 1, 16, [3, 40]),         # K = 16
])
def test_matches_torch_sdpa_float64(B, R, Hq, Hkv, D, prefix):
    rng = np.random.default_rng(10)
    q, k, v, lens = _random_case(rng, B, R, Hq, Hkv, D, prefix, max(prefix) + R + 3)
    got = oracle.verify_attention(q, k, v, lens)
    np.testing.assert_allclose(got, _sdpa_reference(q, k, v, lens), rtol=0, atol=1e-12)


def test_single_key_returns_its_value():
    rng = np.random.default_rng(11)
    q, k, v, lens = _random_case(rng, 1, 1, 4, 2, 32, [0], 4)
    got = oracle.verify_attention(q, k, v, lens)
    for h in range(4):
        np.testing.assert_allclose(got[0, 0, h], v[0, h // 2, 0], rtol=0, atol=1e-15)


def test_identical_keys_give_mean_of_visible_values():
    rng = np.random.default_rng(12)
    R, L = 4, 9
    q, k, v, lens = _random_case(rng, 1, R, 2, 1, 16, [L], L + R)
    k[:] = k[0, 0, 0]
    got = oracle.verify_attention(q, k, v, lens)
    for i in range(R):
        want = v[0, 0, :L + i + 1].mean(axis=0)
        np.testing.assert_allclose(got[0, i, 0], want, rtol=0, atol=1e-13)


def test_rows_never_see_later_keys_or_the_cache_tail():
    rng = np.random.default_rng(13)
    R, L, cap = 5, 20, 40
    q, k, v, lens = _random_case(rng, 1, R, 4, 2, 16, [L], cap)
    ref = oracle.verify_attention(q, k, v, lens)
    k2, v2 = k.copy(), v.copy()
    k2[:, :, L + R:] = 1e3          # beyond len
    v2[:, :, L + R:] = -1e3
    np.testing.assert_allclose(oracle.verify_attention(q, k2, v2, lens), ref, rtol=0, atol=0)
    k3, v3 = k.copy(), v.copy()
    k3[:, :, L + 2:] *= 5.0         # rows 0 and 1 see keys <= L + 1 only
    v3[:, :, L + 2:] += 7.0
    got = oracle.verify_attention(q, k3, v3, lens)
    np.testing.assert_allclose(got[:, :2], ref[:, :2], rtol=0, atol=0)
    assert not np.allclose(got[:, 2:], ref[:, 2:])


def test_ragged_batch_equals_separate_scenes():
    rng = np.random.default_rng(14)
    R = 3
    q, k, v, lens = _random_case(rng, 3, R, 4, 2, 16, [5, 30, 17], 40)
    got = oracle.verify_attention(q, k, v, lens)
    for b in range(3):
        one = oracle.verify_attention(q[b:b + 1], k[b:b + 1], v[b:b + 1], lens[b:b + 1])
        np.testing.assert_allclose(got[b:b + 1], one, rtol=0, atol=0)


def test_decode_row_equals_full_attention():
    # K = 0: one row at position L sees all L + 1 keys, i.e. unmasked attention.
    rng = np.random.default_rng(15)
    q, k, v, lens = _random_case(rng, 1, 1, 2, 1, 16, [50], 51)
    got = oracle.verify_attention(q, k, v, lens)
    qt = torch.from_numpy(q[0]).permute(1, 0, 2)
    kt = torch.from_numpy(k[0]).repeat_interleave(2, dim=0)
    vt = torch.from_numpy(v[0]).repeat_interleave(2, dim=0)
    want = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt).permute(1, 0, 2).numpy()
    np.testing.assert_allclose(got[0], want, rtol=0, atol=1e-12)


def test_explicit_scale_is_used():
    rng = np.random.default_rng(16)
    q, k, v, lens = _random_case(rng, 1, 2, 2, 1, 16, [6], 8)
    a = oracle.verify_attention(q, k, v, lens, scale=0.5)
    b = oracle.verify_attention(q * (0.5 * 4.0), k, v, lens)   # default 1/sqrt(16) = 1/4
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-13)


def test_block_mask_is_unmasked_attention_over_all_rows():
    # the block mask: every new row sees the prefix and all R new rows
    rng = np.random.default_rng(21)
    q, k, v, lens = _random_case(rng, 2, 6, 4, 2, 16, [13, 0], 24)
    out = oracle.verify_attention(q, k, v, lens, block=True)
    B, R, Hq, D = q.shape
    G = Hq // k.shape[1]
    for b in range(B):
        n = int(lens[b])
        qt = torch.from_numpy(q[b]).permute(1, 0, 2)
        kt = torch.from_numpy(k[b, :, :n]).repeat_interleave(G, dim=0)
        vt = torch.from_numpy(v[b, :, :n]).repeat_interleave(G, dim=0)
        ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt).permute(1, 0, 2).numpy()
        assert np.allclose(out[b], ref, atol=1e-12)
    # the last row sees the same keys under both masks
    causal = oracle.verify_attention(q, k, v, lens)
    assert np.allclose(out[:, -1], causal[:, -1], atol=1e-12)
    assert not np.allclose(out[:, 0], causal[:, 0])
