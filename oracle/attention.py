"""Causal GQA attention of the K+1 verify rows, float64 (test infrastructure, oracle only).

Sec. 3.2, Eq. verify: the target scores the K draft tokens in one batched
forward; the distribution at draft position j conditions on the committed
prefix r_{1:t} and the earlier drafts r^_{<j}. Inside each attention layer
that is one causally masked attention of R = K + 1 new query rows against
the cached prefix plus the R new rows.

Readings taken where the paper is silent:
  * R = K + 1 rows: [last committed token, r^_1 .. r^_K]. Row K's output
    supplies the bonus token of Eq. commit when all K drafts match.
  * The cache holds L_b prefix tokens; after the append it holds
    len_b = L_b + R keys. Row i (0-based) is the token at position L_b + i
    and sees keys 0 .. L_b + i. K = 0 (R = 1) is ordinary decode.
  * Softmax scale 1/sqrt(D) unless the caller gives one.
  * Grouped-query attention with contiguous groups: q head h reads KV head
    floor(h / G), G = Hq / Hkv.
  * Block mask (block=True): the variant of the block-diffusion drafts
    (Sec. 5, "Targets and drafts": a block of K = 16 tokens proposed at
    once), where every new row also sees the new rows after it: row i sees
    keys 0 .. L_b + R - 1.

Parity: pinned (tests/test_oracle_attention.py) against torch's float64
scaled_dot_product_attention with an explicitly built causal mask, and by the
special cases one key -> v, identical keys -> mean of V, R = 1 -> plain
decode, and the per-scene independence of a ragged batch; the block mask
against scaled_dot_product_attention without a mask.
"""

import numpy as np


def verify_attention(q, k_cache, v_cache, lens, scale=None, block=False):
    """o[b, i, h] = softmax_n(q[b, i, h] . k[b, g, n] * scale) v[b, g, n], n <= L_b + i
    (n < L_b + R with block=True).

    q:        [B, R, Hq, D]        float64 (rotated query rows)
    k_cache:  [B, Hkv, cap, D]     float64
    v_cache:  [B, Hkv, cap, D]     float64
    lens:     [B] ints             keys valid per scene, R new rows included
    returns   [B, R, Hq, D]        float64
    """
    q = np.asarray(q, dtype=np.float64)
    k_cache = np.asarray(k_cache, dtype=np.float64)
    v_cache = np.asarray(v_cache, dtype=np.float64)
    b_n, r_n, hq, d = q.shape
    hkv = k_cache.shape[1]
    if hq % hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    group = hq // hkv
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    out = np.zeros_like(q)
    for b in range(b_n):
        n_keys = int(lens[b])
        prefix = n_keys - r_n
        if prefix < 0:
            raise ValueError("lens[b] must count the R new rows")
        # visible[i, n]: row i (position prefix + i) sees key n <= prefix + i
        rows = np.arange(r_n)[:, None]
        keys = np.arange(n_keys)[None, :]
        visible = keys <= prefix + rows if not block else np.ones((r_n, n_keys), dtype=bool)
        for h in range(hq):
            g = h // group
            k = k_cache[b, g, :n_keys]
            v = v_cache[b, g, :n_keys]
            s = (q[b, :, h, :] @ k.T) * scale
            s = np.where(visible, s, -np.inf)
            s = s - s.max(axis=1, keepdims=True)
            p = np.exp(s)
            p = p / p.sum(axis=1, keepdims=True)
            out[b, :, h, :] = p @ v
    return out
