"""Both verify-attention kernels against the oracle: the tcgen05 kernel
(head_dim 128, G*R <= 32) and the mma.sync kernel (every other shape, and
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
from tests.helpers import to64, ATTN_ATOL
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
    assert np.isfinite(to64(out)).all() and err <= ATTN_ATOL, (B, R, Hq, Hkv, err)
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
