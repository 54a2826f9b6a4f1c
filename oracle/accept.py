"""Acceptance rules of the verify step, float64 (test infrastructure, oracle only).

Greedy (Sec. 3.2, Eqs. verify, accept, commit; Sec. 4.3, Eq. accept-length):
  r*_j = argmax_v logits[j, v]                       (Eq. verify)
  l    = max{l <= K : r^_j = r*_j for all j <= l}    (Eq. accept)
  emit (r^_1 .. r^_l, r*_{l+1}), t <- t + l + 1      (Eq. commit)
With 0-based rows: row j (j = 0..K) is the target's prediction after the
committed prefix and drafts 0..j-1, so draft[j] is checked against argmax of
row j and the bonus is argmax of row l.

Sampling (Leviathan et al. / Chen et al., cited in Sec. 1 and 2; the paper
evaluates greedy only and does not print the rule):
  p_j = softmax(z_T[j] / T), q_j = softmax(z_D[j] / T)
  for j = 0..K-1, x = draft[j]: accept iff u_j * q_j(x) <= p_j(x)
  first rejection at j: sample r(v) = max(0, p_j(v) - q_j(v)) with u_K
  all K accepted:       sample p_K with u_K (the bonus)
  "sample w with u" = the smallest v with sum_{w <= v} w(v') > u * sum(w)
  (inverse CDF). One uniform per draft position plus one shared by the
  residual / bonus draw: K + 1 uniforms per scene.

Readings where the paper is silent: ties in the argmax go to the lowest index
and compare numerically (+0 == -0); NaN logits are outside the contract.
"<=" in the acceptance test, the inverse-CDF convention and the uniform count
are as above.

Parity: pinned (tests/test_oracle_accept.py): greedy by constructed cases
(identical drafts commit K + 1, exact-l matches, planted ties, K = 0) and a
brute-force scan; sampling by exact enumeration on a 5-token vocabulary
against the theorem that the emitted token is distributed as p, by p == q
always accepting, and by T -> 0 agreeing with greedy.
"""

import numpy as np


def argmax_lowest(row):
    """Index of the maximum of a 1-D array; among equal maxima the lowest index."""
    row = np.asarray(row, dtype=np.float64)
    best = row.max()
    return int(np.flatnonzero(row == best)[0])


def accept_greedy(logits, draft):
    """Greedy longest-prefix acceptance plus bonus token.

    logits: [B, K+1, V] (stored values widened exactly to float64)
    draft:  [B, K] ints
    returns (n_emit [B], tokens [B, K+1] with -1 after n_emit, argmax [B, K+1])
    """
    logits = np.asarray(logits, dtype=np.float64)
    draft = np.asarray(draft, dtype=np.int64).reshape(logits.shape[0], -1)
    b_n, r_n, _ = logits.shape
    k = r_n - 1
    if draft.shape[1] != k:
        raise ValueError("draft must have K = rows - 1 tokens")
    r_star = np.empty((b_n, r_n), dtype=np.int64)
    n_emit = np.empty(b_n, dtype=np.int64)
    tokens = np.full((b_n, r_n), -1, dtype=np.int64)
    for b in range(b_n):
        for j in range(r_n):
            r_star[b, j] = argmax_lowest(logits[b, j])
        ell = k
        for j in range(k):
            if draft[b, j] != r_star[b, j]:
                ell = j
                break
        n_emit[b] = ell + 1
        tokens[b, :ell] = draft[b, :ell]
        tokens[b, ell] = r_star[b, ell]
    return n_emit, tokens, r_star


def _softmax_t(z, temperature):
    """softmax(z / T) in float64."""
    s = np.asarray(z, dtype=np.float64) / np.float64(temperature)
    s = s - s.max()
    e = np.exp(s)
    return e / e.sum()


def _inverse_cdf(w, u):
    """Smallest v with sum_{v' <= v} w(v') > u * sum(w); also the distance of
    u * sum(w) to the nearest step of that cumulative sum, in the units of w
    (probability units: w is p - q clipped, or p)."""
    c = np.cumsum(w)
    total = c[-1]
    target = np.float64(u) * total
    v = int(np.searchsorted(c, target, side="right"))
    v = min(v, len(w) - 1)
    lo = c[v - 1] if v > 0 else 0.0
    margin = min(abs(c[v] - target), abs(target - lo))
    return v, float(margin)


def accept_sample(z_target, z_draft, draft, u, temperature):
    """Leviathan/Chen rejection sampling with caller-supplied uniforms.

    z_target: [B, K+1, V], z_draft: [B, K, V], draft: [B, K] ints,
    u: [B, K+1] uniforms in [0, 1), temperature T > 0.
    returns (n_emit [B], tokens [B, K+1] with -1 after n_emit, margins), where
    margins[b] lists the distance of every decision taken to its boundary:
    |u q - p| / max(p, u q) (relative) for each acceptance test, then the
    inverse-CDF distance of the final draw in probability units.
    """
    z_target = np.asarray(z_target, dtype=np.float64)
    z_draft = np.asarray(z_draft, dtype=np.float64)
    draft = np.asarray(draft, dtype=np.int64)
    u = np.asarray(u, dtype=np.float64)
    b_n, r_n, _ = z_target.shape
    k = r_n - 1
    n_emit = np.empty(b_n, dtype=np.int64)
    tokens = np.full((b_n, r_n), -1, dtype=np.int64)
    margins = []
    for b in range(b_n):
        marg = []
        ell = k
        for j in range(k):
            p = _softmax_t(z_target[b, j], temperature)
            q = _softmax_t(z_draft[b, j], temperature)
            x = draft[b, j]
            lhs, rhs = u[b, j] * q[x], p[x]
            top = max(lhs, rhs)
            marg.append(abs(lhs - rhs) / top if top > 0 else 0.0)
            if lhs <= rhs:
                continue
            ell = j
            break
        if ell < k:
            p = _softmax_t(z_target[b, ell], temperature)
            q = _softmax_t(z_draft[b, ell], temperature)
            w = np.maximum(p - q, 0.0)
            if w.sum() <= 0.0:
                w = p
        else:
            w = _softmax_t(z_target[b, k], temperature)
        tok, m = _inverse_cdf(w, u[b, k])
        marg.append(m)
        n_emit[b] = ell + 1
        tokens[b, :ell] = draft[b, :ell]
        tokens[b, ell] = tok
        margins.append(marg)
    return n_emit, tokens, margins
