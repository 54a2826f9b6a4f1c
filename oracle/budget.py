"""Attention budget of the verify rows, float64 (test infrastructure, oracle only).

Sec. 4.2 ("Empirical confirmation") and Table tab:attn-budget: how a query
row's attention mass divides among the visual tokens, the trajectory / text
tokens of the prompt and the tokens generated in this step, and how spread
the attention is among the non-visual tokens.

Readings taken where the paper is silent (it gives the table, not formulas):
  * Keys visible to row i of scene b are 0 .. L_b + i (L_b = lens[b] - R), as
    in verify_attention. Segments: visual = [0, n_visual[b]), trajectory and
    prompt text = [n_visual[b], L_b), generated = [L_b, L_b + i] (the new
    rows up to the row itself).
  * mass[seg] = sum over the segment's keys of the row's softmax weights
    (scores q . k * scale); the three masses sum to 1.
  * entropy = H(p') / ln(N'): p' the softmax weights restricted to the
    non-visual keys (trajectory / text and generated) and renormalised, N'
    their number, H in nats. 0 when N' <= 1.
The table reports these averaged over heads; this returns them per
(scene, row, head).

Parity: pinned (tests/test_oracle_budget.py) by the masses summing to 1,
uniform scores giving masses proportional to segment sizes and entropy 1,
a dominating key giving mass 1 on its segment and entropy 0, the closed-form
binary entropy of two non-visual keys, and by verify_attention (itself
pinned to torch's float64 scaled_dot_product_attention) with one-hot segment
indicators as values, whose output is the mass vector.
"""

import numpy as np


def attention_budget(q, k_cache, lens, n_visual, scale=None):
    """Per (scene, row, head): segment masses and the normalised entropy.

    q:        [B, R, Hq, D]     float64 (rotated query rows)
    k_cache:  [B, Hkv, cap, D]  float64
    lens:     [B] ints          keys valid per scene, the R new rows included
    n_visual: [B] ints          visual keys at the front of the prefix
    returns   mass [B, R, Hq, 3] (visual, trajectory / text, generated),
              entropy [B, R, Hq]
    """
    q = np.asarray(q, dtype=np.float64)
    k_cache = np.asarray(k_cache, dtype=np.float64)
    b_n, r_n, hq, d = q.shape
    hkv = k_cache.shape[1]
    if hq % hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    group = hq // hkv
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    mass = np.zeros((b_n, r_n, hq, 3))
    entropy = np.zeros((b_n, r_n, hq))
    for b in range(b_n):
        prefix = int(lens[b]) - r_n
        n_vis = int(n_visual[b])
        if prefix < 0 or not 0 <= n_vis <= prefix:
            raise ValueError("need 0 <= n_visual <= lens - R")
        for h in range(hq):
            k = k_cache[b, h // group]
            for i in range(r_n):
                visible = prefix + i + 1
                s = (k[:visible] @ q[b, i, h]) * scale
                w = np.exp(s - s.max())
                p = w / w.sum()
                mass[b, i, h] = [p[:n_vis].sum(), p[n_vis:prefix].sum(), p[prefix:visible].sum()]
                rest = p[n_vis:visible]
                n_rest = rest.size
                if n_rest > 1 and rest.sum() > 0:
                    pr = rest / rest.sum()
                    nz = pr[pr > 0]
                    entropy[b, i, h] = -(nz * np.log(nz)).sum() / np.log(n_rest)
    return mass, entropy
