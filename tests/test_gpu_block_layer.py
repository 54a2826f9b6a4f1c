"""Short block-masked fused layers on the tcgen05 kernel's 64-row tile: verify
layers with the block mask of the block-diffusion drafts (Sec. 5: every new
row sees the prefix and all R new rows) and up to 32 packed query rows per KV
head, which the causal-only 32-row tile does not take, against the float64
oracle and against the separate rotation, append and attention calls: ragged
scenes, stale NaN rows, an empty prefix and prefixes shorter than one key
tile, every cluster size, interleaved M-RoPE, chained dependent launches,
sequential steps on one cache, and the overflow error."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_31160_gb300 import sd, workloads
from tests.helpers import ATTN_ATOL, attn_within, ensure_lib, gpu_case, pair_magnitude, rope_bound, to64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    ensure_lib()


def _case(B, Hq, Hkv, K, prefix, layer, cap_pad=8, tail=float("nan"), sections=(16, 24, 24), D=128):
    R = K + 1
    qpos = np.stack([workloads.text_positions(int(p) + 1, R) for p in prefix])
    return workloads.verify_case(workloads.SWEEP, B=B, Hq=Hq, Hkv=Hkv, D=D, prefix=prefix, K=K,
                                 sections=sections, base=1e6, query_pos=qpos, cap=max(prefix) + R + cap_pad,
                                 layer=layer, tail_fill=tail)


def _oracle_block(q, cache):
    return oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy(), block=True)


def _same(x, y):  # stale cache rows hold NaN on both sides
    return bool(((x == y) | (x.isnan() & y.isnan())).all())


# (B, Hq, Hkv, K, prefix): the draft's shape (G*R = 4), K = 1..3 and 7 of the
# 8B target (8..32 rows), one KV head per query head with 16 rows, ragged
# scenes with an empty prefix and prefixes shorter than one key tile
SHAPES = [
    (1, 16, 4, 0, [4096]),
    (2, 32, 8, 1, [4096, 3001]),
    (3, 32, 8, 3, [0, 31, 1000]),
    (1, 32, 8, 7, [2500]),
    (2, 8, 8, 15, [77, 2048]),
    (4, 4, 1, 2, [1, 33, 64, 500]),
]


def test_block_masked_short_layers_take_the_tcgen05_kernel():
    # block-masked layers of <= 32 packed rows run as one tcgen05 launch (on
    # the 64-row tile), as causal layers and attention calls of the same shapes
    for B, Hq, Hkv, K, prefix in SHAPES:
        cap = max(prefix) + K + 9
        assert sd.lib().sd_verify_kernel(B, K + 1, Hq, Hkv, 128, cap, 2) == b"tcgen05"
        assert sd.verify_kernel(B, K + 1, Hq, Hkv, 128, cap, True) == "tcgen05"
        assert sd.verify_kernel(B, K + 1, Hq, Hkv, 128, cap) == "tcgen05"
    assert sd.lib().sd_verify_kernel(1, 17, 32, 8, 128, 4113, 2) == b"tcgen05"        # 68 rows: two m-blocks
    assert sd.verify_kernel(1, 5, 4, 1, 64, 300, True) == "three kernels"              # head_dim 64


@pytest.mark.parametrize("B,Hq,Hkv,K,prefix,D", [s + (128,) for s in SHAPES] + [(2, 8, 2, 3, [300, 5], 64)])
def test_block_masked_layer_matches_oracle_and_separate_calls(B, Hq, Hkv, K, prefix, D):
    # head_dim 64 runs the layer as the three kernels
    sections = (16, 24, 24) if D == 128 else (8, 12, 12)
    case = _case(B, Hq, Hkv, K, prefix, layer=760 + K, sections=sections, D=D)
    assert sd.verify_kernel(B, K + 1, Hq, Hkv, D, case.cap, True) == ("tcgen05" if D == 128 else "three kernels")
    # separate calls: rotation kernel, append kernel, block-masked attention
    qa, ka, va, pa, ca = gpu_case(case)
    sd.rope_apply(qa, ka, pa, case.sections, 0, case.base)
    sd.kv_append(ca, ka, va)
    oa = sd.verify_attention(qa, ca, block=True)
    # the fused layer
    qb, kb, vb, pb, cb = gpu_case(case)
    ob = sd.verify_layer(qb, kb, vb, pb, case.sections, cb, 0, case.base, block=True)
    torch.cuda.synchronize()
    assert torch.equal(qa, qb) and torch.equal(ka, kb)          # the rotation kernel's bits
    assert _same(ca.k, cb.k) and _same(ca.v, cb.v) and torch.equal(ca.len, cb.len)
    assert cb.len.cpu().tolist() == [p + K + 1 for p in prefix]
    pos = case.pos.numpy()[:, :, None, :]
    ref_q = oracle.mrope_apply(to64(case.q), pos, case.sections, 0, case.base)
    assert np.all(np.abs(to64(qb) - ref_q) <= rope_bound(ref_q, pair_magnitude(to64(case.q))))
    ref_o = _oracle_block(qb, cb)
    assert np.isfinite(to64(ob)).all() and attn_within(to64(ob), ref_o), np.abs(to64(ob) - ref_o).max()
    assert (ob.float() - oa.float()).abs().max().item() <= 2 * ATTN_ATOL
    assert sd.get_device_error() == 0


@pytest.mark.parametrize("cluster", [0, 1, 2, 4, 6, 8, 16])
@pytest.mark.parametrize("B,Hkv,L", [(1, 4, 2048), (3, 8, 1000)])
def test_block_masked_layer_every_cluster_size(cluster, B, Hkv, L):
    # each cluster size (0: the launch's own choice) splits a head's keys and
    # merges the same states through distributed shared memory
    prefix = [L - 13 * b for b in range(B)]
    case = _case(B, 4 * Hkv, Hkv, 1, prefix, layer=740 + B + cluster, tail=0.0)
    assert sd.lib().sd_verify_kernel(B, 2, 4 * Hkv, Hkv, 128, case.cap, 2) == b"tcgen05"
    q, k, v, p, cache = gpu_case(case)
    sd.set_cluster_size(cluster)
    try:
        out = sd.verify_layer(q, k, v, p, case.sections, cache, 0, case.base, block=True)
        torch.cuda.synchronize()
    finally:
        sd.set_cluster_size(0)
    ref = _oracle_block(q, cache)
    assert attn_within(to64(out), ref), np.abs(to64(out) - ref).max()
    assert sd.get_device_error() == 0


def test_block_masked_layer_interleaved_mrope():
    case = _case(2, 32, 8, 2, [900, 4096], layer=780)
    case.interleaved = 1
    rng = np.random.default_rng(781)
    case.pos = torch.from_numpy(rng.integers(0, 5000, size=(2, 3, 3)).astype(np.int32))
    q, k, v, p, cache = gpu_case(case)
    out = sd.verify_layer(q, k, v, p, case.sections, cache, 1, case.base, block=True)
    pos = case.pos.numpy()[:, :, None, :]
    ref_q = oracle.mrope_apply(to64(case.q), pos, case.sections, 1, case.base)
    ref_k = oracle.mrope_apply(to64(case.k_new), pos, case.sections, 1, case.base)
    assert np.all(np.abs(to64(q) - ref_q) <= rope_bound(ref_q, pair_magnitude(to64(case.q))))
    assert np.all(np.abs(to64(k) - ref_k) <= rope_bound(ref_k, pair_magnitude(to64(case.k_new))))
    ref_o = _oracle_block(q, cache)
    assert attn_within(to64(out), ref_o), np.abs(to64(out) - ref_o).max()
    assert sd.get_device_error() == 0


def test_block_masked_layers_chained_early_prefix():
    # back-to-back block-masked layers: every layer after the first streams its
    # prefix before the previous layer ends; same bits as plain launches
    cases = [_case(3, 16, 4, 2, [4096, 2500, 17], layer=800 + l) for l in range(5)]
    runs = []
    for early in (False, True):
        state = [gpu_case(c) for c in cases]
        outs = [sd.verify_layer(q, k, v, p, c.sections, cache, 0, c.base, early=early and l > 0, block=True)
                for l, (c, (q, k, v, p, cache)) in enumerate(zip(cases, state))]
        torch.cuda.synchronize()
        runs.append((outs, state))
    (oa, sa), (ob, sb) = runs
    for l in range(len(cases)):
        assert torch.equal(oa[l], ob[l]) and torch.equal(sa[l][0], sb[l][0])
        assert torch.equal(sa[l][4].len, sb[l][4].len)
    q, _, _, _, cache = sb[3]
    assert attn_within(to64(ob[3]), _oracle_block(q, cache))
    assert sd.get_device_error() == 0


def test_block_masked_steps_on_one_cache():
    # sequential steps on one cache (plain launches: each step's append is
    # the next step's prefix), three-row blocks of a 16 q / 4 KV head layer
    w = workloads.draft_flat()
    L = w["L"]
    rng = np.random.default_rng(830)
    steps, R = 2, 3
    k0 = torch.zeros((1, 4, L + steps * R, 128), dtype=torch.bfloat16)
    v0 = torch.zeros_like(k0)
    k0[:, :, :L] = w["k_cache"][:, :, :L]
    v0[:, :, :L] = w["v_cache"][:, :, :L]
    cache = sd.KVCache(k0.cuda(), v0.cuda(), torch.tensor([L], dtype=torch.int32).cuda())
    qs = [workloads.to_bf16(rng.standard_normal((1, R, 16, 128))).cuda() for _ in range(steps)]
    ks = [workloads.to_bf16(rng.standard_normal((1, R, 4, 128))).cuda() for _ in range(steps)]
    vs = [workloads.to_bf16(rng.standard_normal((1, R, 4, 128))).cuda() for _ in range(steps)]
    outs = []
    for s in range(steps):
        pos = torch.from_numpy(workloads.text_positions(L + R * s, R)[None]).cuda()
        outs.append(sd.verify_layer(qs[s], ks[s], vs[s], pos, (16, 24, 24), cache, 0, w["base"], block=True))
    torch.cuda.synchronize()
    assert cache.len.item() == L + steps * R
    k64, v64 = to64(cache.k), to64(cache.v)
    for s in range(steps):
        ref = oracle.verify_attention(to64(qs[s]), k64, v64, np.array([L + R * (s + 1)]), block=True)
        assert attn_within(to64(outs[s]), ref)
    assert sd.get_device_error() == 0


def test_block_masked_layer_overflow_sets_error_and_leaves_scene():
    case = _case(1, 16, 4, 0, [300], layer=820)
    q, k, v, p, cache = gpu_case(case)
    cache.len.fill_(case.cap)            # one more row does not fit
    out = torch.full_like(q, 5.0)
    k0 = cache.k.clone()
    sd.get_device_error()
    sd.verify_layer(q, k, v, p, case.sections, cache, 0, 1e6, out=out, block=True)
    assert sd.get_device_error() & sd.SD_DEVERR_KV_OVERFLOW
    assert cache.len.item() == case.cap
    assert torch.all(out == 5.0)
    assert _same(cache.k, k0)
