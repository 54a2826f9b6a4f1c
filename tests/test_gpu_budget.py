"""GPU parity of sd_attention_budget against the float64 oracle
(Sec. 4.2, Table tab:attn-budget): masses and normalised entropies within
1e-4 (fp32 scores and sums against float64)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_31160_gb300 import sd, workloads
from tests.helpers import ensure_lib, gpu_case, to64

pytestmark = pytest.mark.gpu
TOL = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _lib():
    ensure_lib()


def _check(q, cache, n_visual):
    mass, ent = sd.attention_budget(q, cache, n_visual)
    rm, re_ = oracle.attention_budget(to64(q), to64(cache.k), cache.len.cpu().numpy(), n_visual.cpu().numpy())
    assert np.abs(mass.cpu().numpy() - rm).max() <= TOL
    assert np.abs(ent.cpu().numpy() - re_).max() <= TOL
    assert sd.get_device_error() == 0
    return mass, ent


def test_target_layer_budget():
    # 8B target layer: 3584 visual patches of 4096 prefix keys, 8 rows
    case = workloads.target_layer()
    q, k_new, v_new, pos, cache = gpu_case(case)
    sd.rope_apply(q, k_new, pos, case.sections, case.interleaved, case.base)
    sd.kv_append(cache, k_new, v_new)
    mass, _ = _check(q, cache, torch.tensor([3584], dtype=torch.int32, device="cuda"))
    assert torch.allclose(mass.sum(-1), torch.ones_like(mass[..., 0]), atol=1e-5)


@pytest.mark.parametrize("B,R,Hq,Hkv,D,prefix,nvis", [
    (3, 5, 4, 1, 64, [1, 17, 300], [0, 9, 300]),     # no visual keys / all visual
    (2, 17, 32, 8, 128, [2000, 513], [1750, 448]),   # K = 16: three row groups
    (1, 1, 16, 4, 128, [4096], [3584]),              # draft-shaped single row
    (1, 8, 32, 8, 128, [8000], [7000]),              # two staged chunks of keys a CTA
    (1, 17, 32, 8, 128, [6000], [5000]),             # two chunks, reloaded for each of three row groups
])
def test_random_shapes(B, R, Hq, Hkv, D, prefix, nvis):
    rng = np.random.default_rng(B * 10 + R)
    cap = max(prefix) + R + 3
    k = workloads.to_bf16(rng.standard_normal((B, Hkv, cap, D)))
    q = workloads.to_bf16(rng.standard_normal((B, R, Hq, D))).cuda()
    cache = sd.KVCache(k.cuda(), k.cuda().clone(), torch.tensor([p + R for p in prefix], dtype=torch.int32).cuda())
    _check(q, cache, torch.tensor(nvis, dtype=torch.int32, device="cuda"))


def test_visual_count_out_of_range_sets_error():
    rng = np.random.default_rng(3)
    k = workloads.to_bf16(rng.standard_normal((1, 1, 40, 64))).cuda()
    cache = sd.KVCache(k, k.clone(), torch.tensor([30], dtype=torch.int32, device="cuda"))
    q = workloads.to_bf16(rng.standard_normal((1, 2, 2, 64))).cuda()
    sd.get_device_error()
    sd.attention_budget(q, cache, torch.tensor([29], dtype=torch.int32, device="cuda"))
    assert sd.get_device_error() & sd.SD_DEVERR_LENGTH
