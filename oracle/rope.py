"""Rotary position embeddings in float64 (test infrastructure, oracle only).

Sec. 3.3, Eq. rope-1d: 1D RoPE rotates each adjacent pair (2d, 2d+1) of a
head vector by the angle m * w_d, w_d = b^(-2d/h); the rotation is the
block-diagonal direct sum of 2x2 rotations.

Sec. 3.3, Eq. rope-3d, and Sec. 4.2, Eqs. axis-assign and mrope-phase: 3D
M-RoPE gives each token a (T, H, W) coordinate. Rotary pair d takes its angle
from the coordinate of axis a(d): phi_d = theta_d * p_{a(d)}, with a(d)
blocked over mrope_section = (s_T, s_H, s_W) or interleaved as d mod 3.

Sec. 4.2, Eq. flatrope-proj: FlatRoPE sets p_T = p_H = p_W = m, the sequence
index, so the phase is theta_d * m at every pair.

Readings taken where the paper is loose:
  * theta_d is one global schedule indexed by the global pair d (Eq.
    mrope-phase), not three per-axis vectors (Eq. rope-3d's w^T, w^H, w^W).
    Only this reading makes M-RoPE reduce to 1D RoPE when t = h = w, which the
    paper states in Sec. 3.3 and Sec. 4.2.
  * Pairs are adjacent dimensions (2d, 2d+1), the literal block-diagonal form
    of Eq. rope-1d.
  * The base is a parameter (the paper's example is 10000; the workloads use
    1e6).

Parity: pinned (tests/test_oracle_rope.py): hand-derived closed-form values,
the M-RoPE == 1D identity through the explicit matrix of Eq. rope-1d, norm
preservation, per-axis relative-position invariance, FlatRoPE independence of
the section layout, and the per-axis support of each rotation.
"""

import numpy as np

AXIS_T, AXIS_H, AXIS_W = 0, 1, 2


def rope_frequencies(head_dim, base):
    """theta_d = base^(-2d/h) for d = 0 .. h/2-1 (Eq. rope-1d, Eq. mrope-phase)."""
    if head_dim % 2:
        raise ValueError("head_dim must be even")
    d = np.arange(head_dim // 2, dtype=np.float64)
    return np.power(np.float64(base), -2.0 * d / head_dim)


def axis_assignment(head_dim, sections, interleaved):
    """a(d) in {T, H, W} for each rotary pair d (Eq. axis-assign).

    Blocked: T for d < s_T, H for s_T <= d < s_T + s_H, W after.
    Interleaved: (T, H, W)[d mod 3]; the section sizes play no part there,
    which is what the equation prints.
    """
    d_r = head_dim // 2
    s_t, s_h, s_w = (int(s) for s in sections)
    if s_t + s_h + s_w != d_r:
        raise ValueError("mrope_section must sum to head_dim / 2")
    a = np.empty(d_r, dtype=np.int64)
    for d in range(d_r):
        if interleaved:
            a[d] = (AXIS_T, AXIS_H, AXIS_W)[d % 3]
        elif d < s_t:
            a[d] = AXIS_T
        elif d < s_t + s_h:
            a[d] = AXIS_H
        else:
            a[d] = AXIS_W
    return a


def mrope_apply(x, pos3, sections, interleaved, base):
    """3D M-RoPE of x (Eqs. rope-3d, axis-assign, mrope-phase).

    x:    [..., h] float64 head vectors.
    pos3: [..., 3] integer (T, H, W) coordinates, broadcastable against x's
          leading dimensions (pass [B, R, 1, 3] for x of shape [B, R, H, h]).
    For pair d: phi_d = theta_d * pos3[a(d)], and
    (x_2d, x_2d+1) -> (x_2d cos phi - x_2d+1 sin phi, x_2d sin phi + x_2d+1 cos phi).
    """
    x = np.asarray(x, dtype=np.float64)
    h = x.shape[-1]
    theta = rope_frequencies(h, base)
    a = axis_assignment(h, sections, interleaved)
    pos = np.asarray(pos3, dtype=np.float64)
    phi = theta * pos[..., a]
    c, s = np.cos(phi), np.sin(phi)
    x0, x1 = x[..., 0::2], x[..., 1::2]
    out = np.empty(np.broadcast_shapes(x.shape), dtype=np.float64)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def rope_1d_matrix(m, head_dim, base):
    """R(m, w) of Eq. rope-1d written out as an explicit h x h matrix.

    Block d (rows/cols 2d, 2d+1) is [[cos(m w_d), -sin(m w_d)],
    [sin(m w_d), cos(m w_d)]]; every other entry is zero.
    """
    w = rope_frequencies(head_dim, base)
    rot = np.zeros((head_dim, head_dim), dtype=np.float64)
    for d in range(head_dim // 2):
        c, s = np.cos(m * w[d]), np.sin(m * w[d])
        rot[2 * d, 2 * d] = c
        rot[2 * d, 2 * d + 1] = -s
        rot[2 * d + 1, 2 * d] = s
        rot[2 * d + 1, 2 * d + 1] = c
    return rot


def rope_1d(x, m, base):
    """1D RoPE of Eq. rope-1d for vectors x[..., h] that all sit at position m,
    computed as the matrix-vector product R(m, w) x."""
    x = np.asarray(x, dtype=np.float64)
    rot = rope_1d_matrix(m, x.shape[-1], base)
    return x @ rot.T


def flatrope_positions(m):
    """FlatRoPE's (T, H, W) coordinates (Eq. flatrope-proj): every axis takes
    the sequence index m. Returns [..., 3] integers."""
    m = np.asarray(m, dtype=np.int64)
    return np.stack([m, m, m], axis=-1)
