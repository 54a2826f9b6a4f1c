"""KV-cache append and rollback (test infrastructure, oracle only).

Sec. 3.2, Eq. commit: an iteration commits l + 1 tokens and advances
t_{i+1} = t_i + l_i + 1. The verify pass appended the keys/values of all
R = K + 1 rows; of those, the rows that stay valid are the last committed
token and the l accepted drafts, i.e. n_emit = l + 1 rows. The rejected rows'
entries are dropped by moving the length back, never by erasing data.

Parity: pinned (tests/test_oracle_kv.py) by a row-by-row shadow copy, by
rollback to n_appended being a no-op and rollback to 0 restoring the
pre-append length.
"""

import numpy as np


def kv_append(k_cache, v_cache, lens, k_new, v_new):
    """Write R new rows of every scene at positions lens[b] .. lens[b]+R-1.

    k_cache, v_cache: [B, Hkv, cap, D]; k_new, v_new: [B, R, Hkv, D];
    lens: [B]. Returns (k_cache', v_cache', lens + R) as new arrays.
    Raises ValueError when a scene would pass the capacity.
    """
    k_out = np.array(k_cache, copy=True)
    v_out = np.array(v_cache, copy=True)
    lens = np.asarray(lens, dtype=np.int64)
    b_n, r_n, hkv, _ = np.shape(k_new)
    cap = k_out.shape[2]
    for b in range(b_n):
        if lens[b] + r_n > cap:
            raise ValueError("append beyond capacity")
        for i in range(r_n):
            for g in range(hkv):
                k_out[b, g, lens[b] + i] = k_new[b, i, g]
                v_out[b, g, lens[b] + i] = v_new[b, i, g]
    return k_out, v_out, lens + r_n


def kv_rollback(lens, committed, n_appended):
    """lens[b] <- lens[b] - n_appended + committed[b], committed in [0, n_appended]."""
    lens = np.asarray(lens, dtype=np.int64)
    committed = np.asarray(committed, dtype=np.int64)
    if np.any(committed < 0) or np.any(committed > n_appended):
        raise ValueError("committed length outside [0, n_appended]")
    return lens - n_appended + committed
