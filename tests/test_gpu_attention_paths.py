"""Both verify-attention kernels against the oracle: the tcgen05 kernel
(head_dim 128, G*R <= 128) and the mma.sync kernel (every other shape, and
every shape when SD_ATTENTION_KERNEL=mma). The override is read once per
process, so the mma.sync leg runs in a child process."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r'''
import sys, numpy as np, torch
sys.path.insert(0, %r)
import oracle
from paper_2606_31160_gb300 import sd, workloads, build
from tests.helpers import to64, attn_within
build.build()
worst = 0.0
for (B, R, Hq, Hkv, D, prefix) in [(1, 8, 32, 8, 128, [4096]), (2, 8, 32, 8, 128, [4095, 1000]),
                                   (1, 1, 16, 4, 128, [4096]), (3, 5, 4, 1, 128, [1, 17, 300])]:
    rng = np.random.default_rng(B * 100 + R)
    cap = max(prefix) + R + 9
    k = rng.standard_normal((B, Hkv, cap, D)).astype(np.float32)
    v = rng.standard_normal((B, Hkv, cap, D)).astype(np.float32)
    for b in range(B):
        k[b, :, prefix[b] + R:] = np.nan
        v[b, :, prefix[b] + R:] = np.nan
    q = workloads.to_bf16(rng.standard_normal((B, R, Hq, D))).cuda()
    cache = sd.KVCache(workloads.to_bf16(k).cuda(), workloads.to_bf16(v).cuda(),
                       torch.tensor([p + R for p in prefix], dtype=torch.int32).cuda())
    out = sd.verify_attention(q, cache)
    ref = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy())
    err = float(np.abs(to64(out) - ref).max())
    assert np.isfinite(to64(out)).all() and attn_within(to64(out), ref), (B, R, Hq, Hkv, err)
    worst = max(worst, err)
assert sd.get_device_error() == 0
print("OK", worst)
''' % ROOT


@pytest.mark.parametrize("kernel", ["mma", "auto"])
def test_attention_kernel_paths(kernel):
    env = dict(os.environ, SD_ATTENTION_KERNEL=kernel)
    res = subprocess.run([sys.executable, "-c", CHILD], env=env, cwd=ROOT, capture_output=True,
                         text=True, timeout=600)
    assert res.returncode == 0, res.stdout + res.stderr
    assert "OK" in res.stdout


def _planted(seed, plants, fused, R=8, new_plants=()):
    """B=1, 32 q / 8 KV heads x 128, L=4096 prefix, R=8: key n of KV head h // 4
    is set to alpha * (rotated) q[i][h], so that row i of head h scores it far
    above everything in the first tile of its split."""
    import numpy as np
    import torch
    import oracle
    from paper_2606_31160_gb300 import sd, workloads
    rng = np.random.default_rng(seed)
    B, Hq, Hkv, D, L = 1, 32, 8, 128, 4096
    cap = L + R + 8
    q = workloads.to_bf16(rng.standard_normal((B, R, Hq, D)))
    k = rng.standard_normal((B, Hkv, cap, D)).astype(np.float32)
    v = rng.standard_normal((B, Hkv, cap, D)).astype(np.float32)
    k_new = workloads.to_bf16(rng.standard_normal((B, R, Hkv, D)))
    v_new = workloads.to_bf16(rng.standard_normal((B, R, Hkv, D)))
    pos = np.repeat(np.arange(L + 1, L + 1 + R, dtype=np.int32)[None, :, None], 3, axis=2)
    sections = (16, 24, 24)
    q64 = q.float().numpy().astype(np.float64)
    q_rot = oracle.mrope_apply(q64, pos[:, :, None, :], sections, 0, 1e6) if fused else q64
    for (h, i, n, alpha) in plants:
        k[0, h // (Hq // Hkv), n] = alpha * q_rot[0, i, h] / np.linalg.norm(q_rot[0, i, h]) * 12.0
    if new_plants:
        # new key rows i and 0 of KV head h // 4 set (after their rotation) to
        # alpha * q[i][h]: raw rows are the inverse rotation of the target
        kn = k_new.float().numpy().astype(np.float64)
        for (h, i, alpha) in new_plants:
            target = alpha * q_rot[0, i, h] / np.linalg.norm(q_rot[0, i, h]) * 12.0
            for n in (i, 0):
                kn[0, n, h // (Hq // Hkv)] = oracle.mrope_apply(target, -pos[0, n], sections, 0, 1e6)
        k_new = workloads.to_bf16(kn)
    if fused:
        k[:, :, L:] = np.nan  # stale rows past the prefix
        v[:, :, L:] = np.nan
        cache = sd.KVCache(workloads.to_bf16(k).cuda(), workloads.to_bf16(v).cuda(),
                           torch.full((B,), L, dtype=torch.int32).cuda())
        qd, kd = q.cuda(), k_new.cuda()
        out = sd.verify_layer(qd, kd, v_new.cuda(), torch.from_numpy(pos).cuda(), sections, cache, 0, 1e6)
        q_ref = qd
    else:
        cache = sd.KVCache(workloads.to_bf16(k).cuda(), workloads.to_bf16(v).cuda(),
                           torch.full((B,), L + R, dtype=torch.int32).cuda())
        q_ref = q.cuda()
        out = sd.verify_attention(q_ref, cache)
    torch.cuda.synchronize()
    ref = oracle.verify_attention(q_ref.cpu().float().numpy().astype(np.float64),
                                  cache.k.cpu().float().numpy().astype(np.float64),
                                  cache.v.cpu().float().numpy().astype(np.float64), cache.len.cpu().numpy())
    return out.cpu().float().numpy().astype(np.float64), ref, sd.get_device_error()


@pytest.mark.parametrize("R", [8, 12])
@pytest.mark.parametrize("fused", [False, True])
def test_fixed_reference_fallback_pass(fused, R):
    # a planted key scores ~17 * alpha in log2 units (|k| = 12 alpha along q,
    # |q| ~ 11.3, scale log2(e) / sqrt(128)): alpha 6 puts it ~100 above the
    # row's reference (the first tile's maximum, or in the fused layer the
    # row's score against its own new key and new key 0; beyond the 64 one pass
    # allows, so its split runs the fallback pass), alpha 2.5 ~40 above (kept by
    # the single pass), alpha -6 far below; keys in later tiles of splits 0, 3 and 7
    import numpy as np
    from tests.helpers import ATTN_ATOL
    plants = [(0, 0, 300, 6.0), (5, 3, 2000, 6.0), (31, 7, 4000, 6.0), (12, 2, 1700, 2.5),
              (13, 2, 130, -6.0)]
    out, ref, err = _planted(7, plants, fused, R)
    assert err == 0
    assert np.isfinite(out).all()
    e = np.abs(out - ref).max()
    assert e <= ATTN_ATOL, e
    # the planted rows are dominated by their key (the output is its value row)
    assert np.abs(ref[0, 0, 0]).max() > 0.5


@pytest.mark.parametrize("alpha", [-9.0, -2.5])
def test_fused_reference_below_the_prefix(alpha):
    # the fused layer's reference of a row is its larger score against its own
    # new key and new key 0; both planted at ~17 * alpha in log2 units leave
    # every prefix key of that row ~150 (alpha -9: beyond the 64 one pass
    # allows, so its head's splits run the fallback pass; a single pass would
    # overflow fp32 there) or ~40 (alpha -2.5) above the reference
    import numpy as np
    from tests.helpers import ATTN_ATOL
    out, ref, err = _planted(11, [], True, 8, new_plants=[(9, 5, alpha), (22, 3, alpha), (30, 0, alpha)])
    assert err == 0
    assert np.isfinite(out).all()
    e = np.abs(out - ref).max()
    assert e <= ATTN_ATOL, e


def _fused_case(R, prefix, layer):
    import numpy as np
    from paper_2606_31160_gb300 import workloads
    B = len(prefix)
    qpos = np.stack([workloads.text_positions(int(p) + 1, R) for p in prefix])
    return workloads.verify_case(workloads.TARGET_LAYER, B=B, Hq=32, Hkv=8, D=128, prefix=prefix, K=R - 1,
                                 sections=(16, 24, 24), base=1e6, query_pos=qpos, cap=max(prefix) + R + 40,
                                 layer=layer, tail_fill=float("nan"))


# R = 8: 32 packed rows (32-row tile); R = 9 and 16: 36 and 64 rows (64-row
# tile); R = 17: 68 rows, two 64-row m-blocks (the fused layer caps the
# cluster size at 32 - R, so a forced 16 falls back to the automatic choice)
@pytest.mark.parametrize("cluster", [1, 2, 4, 6, 8, 16])
@pytest.mark.parametrize("R", [8, 9, 16, 17])
def test_every_cluster_size(cluster, R):
    # the split of each head's keys over `cluster` CTAs and the merge of their
    # partial states (uneven rows per rank for 6); ragged short prefixes leave
    # some ranks without keys
    import numpy as np
    import torch
    import oracle
    from paper_2606_31160_gb300 import sd, workloads
    from tests.helpers import attn_within, gpu_case, to64
    sd.set_cluster_size(cluster)
    try:
        if R <= 31:
            case = _fused_case(R, [4096, 777], layer=500 + R)
            q, k_new, v_new, pos, cache = gpu_case(case)
            out = sd.verify_layer(q, k_new, v_new, pos, case.sections, cache, 0, 1e6)
            ref = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy())
            assert np.isfinite(to64(out)).all()
            assert attn_within(to64(out), ref)
            assert cache.len.cpu().tolist() == [4096 + R, 777 + R]
        prefix = [0, 31, 130, 4095]
        B = len(prefix)
        rng = np.random.default_rng(cluster * 100 + R)
        cap = max(prefix) + R + 5
        k = rng.standard_normal((B, 8, cap, 128)).astype(np.float32)
        v = rng.standard_normal((B, 8, cap, 128)).astype(np.float32)
        for b in range(B):
            k[b, :, prefix[b] + R:] = np.nan
            v[b, :, prefix[b] + R:] = np.nan
        q2 = workloads.to_bf16(rng.standard_normal((B, R, 32, 128))).cuda()
        cache2 = sd.KVCache(workloads.to_bf16(k).cuda(), workloads.to_bf16(v).cuda(),
                            torch.tensor([p + R for p in prefix], dtype=torch.int32).cuda())
        out2 = sd.verify_attention(q2, cache2)
        ref2 = oracle.verify_attention(to64(q2), to64(cache2.k), to64(cache2.v), cache2.len.cpu().numpy())
        assert np.isfinite(to64(out2)).all()
        assert attn_within(to64(out2), ref2)
        assert sd.get_device_error() == 0
    finally:
        sd.set_cluster_size(0)
