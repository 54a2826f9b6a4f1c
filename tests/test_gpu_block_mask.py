"""The block mask (every new row sees all R new rows: the block-diffusion
draft's pattern, Sec. 5) on both attention kernels and the fused layer,
against the float64 oracle."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import oracle
from paper_2606_31160_gb300 import sd, workloads
from tests.helpers import ATTN_ATOL, attn_within, ensure_lib, gpu_case, to64

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _lib():
    ensure_lib()


def _case(seed, B, R, Hq, Hkv, D, prefix):
    rng = np.random.default_rng(seed)
    cap = max(prefix) + R + 5
    k = rng.standard_normal((B, Hkv, cap, D)).astype(np.float32)
    v = rng.standard_normal((B, Hkv, cap, D)).astype(np.float32)
    for b in range(B):
        k[b, :, prefix[b] + R:] = np.nan
        v[b, :, prefix[b] + R:] = np.nan
    q = workloads.to_bf16(rng.standard_normal((B, R, Hq, D))).cuda()
    cache = sd.KVCache(workloads.to_bf16(k).cuda(), workloads.to_bf16(v).cuda(),
                       torch.tensor([p + R for p in prefix], dtype=torch.int32).cuda())
    return q, cache


# tcgen05 32-row tile, 64-row tile, two m-blocks (K = 16); mma.sync (D = 64)
@pytest.mark.parametrize("B,R,Hq,Hkv,D,prefix", [
    (2, 8, 32, 8, 128, [4095, 30]),
    (1, 12, 32, 8, 128, [700]),
    (2, 17, 32, 8, 128, [2000, 0]),
    (2, 8, 16, 4, 64, [300, 1]),
])
def test_block_mask_attention(B, R, Hq, Hkv, D, prefix):
    q, cache = _case(B * 100 + R + D, B, R, Hq, Hkv, D, prefix)
    out = sd.verify_attention(q, cache, block=True)
    ref = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy(), block=True)
    assert np.isfinite(to64(out)).all() and attn_within(to64(out), ref)
    causal = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy())
    assert np.abs(ref - causal).max() > 10 * ATTN_ATOL   # the mask matters for these rows
    assert sd.get_device_error() == 0


@pytest.mark.parametrize("K", [7, 16])
def test_block_mask_fused_layer(K):
    R = K + 1
    prefix = [4096, 1500]
    qpos = np.stack([workloads.text_positions(int(p) + 1, R) for p in prefix])
    case = workloads.verify_case(workloads.TARGET_LAYER, B=2, Hq=32, Hkv=8, D=128, prefix=prefix, K=K,
                                 sections=(16, 24, 24), base=1e6, query_pos=qpos, cap=max(prefix) + R + 8,
                                 layer=700 + K, tail_fill=float("nan"))
    q, k_new, v_new, pos, cache = gpu_case(case)
    out = sd.verify_layer(q, k_new, v_new, pos, case.sections, cache, 0, 1e6, block=True)
    ref = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy(), block=True)
    assert np.isfinite(to64(out)).all() and attn_within(to64(out), ref)
    assert sd.get_device_error() == 0


def test_block_mask_on_the_mma_kernel_for_tcgen05_shapes():
    # the shapes the tcgen05 kernel serves, forced onto the mma.sync kernel
    child = r'''
import sys, numpy as np, torch
sys.path.insert(0, %r)
import oracle
from paper_2606_31160_gb300 import sd, workloads, build
from tests.helpers import to64, attn_within
build.build()
rng = np.random.default_rng(5)
B, R, Hq, Hkv, D, prefix = 2, 8, 32, 8, 128, [4095, 30]
cap = max(prefix) + R + 5
k = workloads.to_bf16(rng.standard_normal((B, Hkv, cap, D)))
v = workloads.to_bf16(rng.standard_normal((B, Hkv, cap, D)))
q = workloads.to_bf16(rng.standard_normal((B, R, Hq, D))).cuda()
cache = sd.KVCache(k.cuda(), v.cuda(), torch.tensor([p + R for p in prefix], dtype=torch.int32).cuda())
out = sd.verify_attention(q, cache, block=True)
ref = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy(), block=True)
assert attn_within(to64(out), ref)
assert sd.get_device_error() == 0
print("OK")
''' % ROOT
    env = dict(os.environ, SD_ATTENTION_KERNEL="mma")
    res = subprocess.run([sys.executable, "-c", child], env=env, cwd=ROOT, capture_output=True, text=True,
                         timeout=600)
    assert res.returncode == 0 and "OK" in res.stdout, res.stdout + res.stderr
