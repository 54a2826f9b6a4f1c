"""The small-tile kernel (up to 16 packed query rows per KV head: the draft's
single-row decode steps and short verify blocks) against the float64 oracle:
verify attention and the fused verify layer, ragged scenes, stale NaN rows,
every cluster size the launch picks, the block mask, chained dependent
launches and the draft's decode loop on one cache."""
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


def _case(B, Hq, Hkv, K, prefix, layer, cap_pad=8, tail=float("nan"), sections=(16, 24, 24)):
    R = K + 1
    qpos = np.stack([workloads.text_positions(int(p) + 1, R) for p in prefix])
    return workloads.verify_case(workloads.SWEEP, B=B, Hq=Hq, Hkv=Hkv, D=128, prefix=prefix, K=K,
                                 sections=sections, base=1e6, query_pos=qpos, cap=max(prefix) + R + cap_pad,
                                 layer=layer, tail_fill=tail)


def _appended(case):
    """Cache with the raw new rows appended on the host (attention-only tests:
    rotation is not under test, so q and the new keys are used as drawn)."""
    k, v = case.k_cache.clone(), case.v_cache.clone()
    for b, p in enumerate(case.prefix):
        k[b, :, p:p + case.R] = case.k_new[b].transpose(0, 1)
        v[b, :, p:p + case.R] = case.v_new[b].transpose(0, 1)
    lens = torch.from_numpy((case.prefix + case.R).astype(np.int32)).cuda()
    return sd.KVCache(k.cuda(), v.cuda(), lens)


def _oracle_attention(q, cache, block=False):
    return oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy(), block=block)


# (B, Hq, Hkv, K, prefix): draft decode (G*R = 4), K = 1..3 of the 8B target
# (8..16 rows), one KV head per query head with 16 rows, ragged scenes with an
# empty prefix and prefixes shorter than one 32-key block
SHAPES = [
    (1, 16, 4, 0, [4096]),
    (2, 32, 8, 1, [4096, 3001]),
    (3, 32, 8, 3, [0, 31, 1000]),
    (2, 8, 8, 15, [77, 2048]),
    (4, 4, 1, 2, [1, 33, 64, 500]),
]


@pytest.mark.parametrize("B,Hq,Hkv,K,prefix", SHAPES)
def test_attention_small_tiles_match_oracle(B, Hq, Hkv, K, prefix):
    case = _case(B, Hq, Hkv, K, prefix, layer=700 + K)
    cache = _appended(case)
    q = case.q.cuda()
    out = sd.verify_attention(q, cache)
    ref = _oracle_attention(q, cache)
    assert np.isfinite(to64(out)).all() and attn_within(to64(out), ref), np.abs(to64(out) - ref).max()
    assert sd.get_device_error() == 0


@pytest.mark.parametrize("B,Hq,Hkv,K,prefix", SHAPES[1:4])
def test_attention_small_tiles_block_mask(B, Hq, Hkv, K, prefix):
    case = _case(B, Hq, Hkv, K, prefix, layer=720 + K)
    cache = _appended(case)
    q = case.q.cuda()
    out = sd.verify_attention(q, cache, block=True)
    ref = _oracle_attention(q, cache, block=True)
    assert attn_within(to64(out), ref), np.abs(to64(out) - ref).max()
    assert sd.get_device_error() == 0


@pytest.mark.parametrize("B,Hkv", [(1, 4), (2, 8), (8, 4), (40, 8)])
def test_attention_every_cluster_size(B, Hkv):
    # the launch sizes its clusters from B * Hkv (16, 8, 4 ... 1 CTAs per head):
    # each size merges the same states through distributed shared memory
    prefix = [2048 - 13 * b for b in range(B)]
    case = _case(B, 4 * Hkv, Hkv, 1, prefix, layer=740 + B, tail=0.0)
    cache = _appended(case)
    q = case.q.cuda()
    out = sd.verify_attention(q, cache)
    ref = _oracle_attention(q, cache)
    assert attn_within(to64(out), ref), np.abs(to64(out) - ref).max()
    assert sd.get_device_error() == 0


@pytest.mark.parametrize("B,Hq,Hkv,K,prefix", SHAPES)
def test_layer_small_tiles_match_oracle_and_separate_calls(B, Hq, Hkv, K, prefix):
    case = _case(B, Hq, Hkv, K, prefix, layer=760 + K)
    # separate calls: rotation kernel, append kernel, attention
    qa, ka, va, pa, ca = gpu_case(case)
    sd.rope_apply(qa, ka, pa, case.sections, 0, case.base)
    sd.kv_append(ca, ka, va)
    oa = sd.verify_attention(qa, ca)
    # the fused layer
    qb, kb, vb, pb, cb = gpu_case(case)
    ob = sd.verify_layer(qb, kb, vb, pb, case.sections, cb, 0, case.base)
    torch.cuda.synchronize()

    def same(x, y):  # stale cache rows hold NaN on both sides
        return bool(((x == y) | (x.isnan() & y.isnan())).all())

    assert torch.equal(qa, qb) and torch.equal(ka, kb)          # the rotation kernel's bits
    assert same(ca.k, cb.k) and same(ca.v, cb.v) and torch.equal(ca.len, cb.len)
    assert cb.len.cpu().tolist() == [p + K + 1 for p in prefix]
    pos = case.pos.numpy()[:, :, None, :]
    ref_q = oracle.mrope_apply(to64(case.q), pos, case.sections, 0, case.base)
    assert np.all(np.abs(to64(qb) - ref_q) <= rope_bound(ref_q, pair_magnitude(to64(case.q))))
    ref_o = _oracle_attention(qb, cb)
    assert np.isfinite(to64(ob)).all() and attn_within(to64(ob), ref_o), np.abs(to64(ob) - ref_o).max()
    assert (ob.float() - oa.float()).abs().max().item() <= 2 * ATTN_ATOL
    assert sd.get_device_error() == 0


def test_layer_small_tiles_block_mask_and_interleaved():
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
    ref_o = _oracle_attention(q, cache, block=True)
    assert attn_within(to64(out), ref_o), np.abs(to64(out) - ref_o).max()
    assert sd.get_device_error() == 0


def test_layer_small_tiles_chained_early_prefix():
    # back-to-back layers of a batched decode: every layer after the first
    # streams its prefix before the previous layer ends; same bits as plain
    cases = [_case(3, 16, 4, 0, [4096, 2500, 17], layer=800 + l) for l in range(5)]
    runs = []
    for early in (False, True):
        state = [gpu_case(c) for c in cases]
        outs = [sd.verify_layer(q, k, v, p, c.sections, cache, 0, c.base, early=early and l > 0)
                for l, (c, (q, k, v, p, cache)) in enumerate(zip(cases, state))]
        torch.cuda.synchronize()
        runs.append((outs, state))
    (oa, sa), (ob, sb) = runs
    for l in range(len(cases)):
        assert torch.equal(oa[l], ob[l]) and torch.equal(sa[l][0], sb[l][0])
        assert torch.equal(sa[l][4].len, sb[l][4].len)
    q, _, _, _, cache = sb[3]
    ref = _oracle_attention(q, cache)
    assert attn_within(to64(ob[3]), ref)
    assert sd.get_device_error() == 0


def test_draft_decode_loop_on_one_cache():
    # the draft's propose loop: single-row steps on one cache, each appending
    # the row the next step attends to (plain launches: each step waits for
    # the previous one), then the rollback
    w = workloads.draft_flat()
    L, steps = w["L"], w["steps"]
    cache = sd.KVCache(w["k_cache"].cuda(), w["v_cache"].cuda(), torch.tensor([L], dtype=torch.int32).cuda())
    qs = [w["q"][s].cuda() for s in range(steps)]
    outs = []
    for s in range(steps):
        pos = torch.full((1, 1, 3), L + s, dtype=torch.int32, device="cuda")
        outs.append(sd.verify_layer(qs[s], w["k_new"][s].cuda(), w["v_new"][s].cuda(), pos, (16, 24, 24), cache,
                                    0, w["base"]))
    torch.cuda.synchronize()
    assert cache.len.item() == L + steps
    k64, v64 = to64(cache.k), to64(cache.v)
    for s in range(steps):
        ref = oracle.verify_attention(to64(qs[s]), k64, v64, np.array([L + s + 1]))
        assert np.abs(to64(outs[s]) - ref).max() <= ATTN_ATOL
    assert sd.get_device_error() == 0


def test_layer_small_tiles_overflow_sets_error_and_leaves_scene():
    case = _case(1, 16, 4, 0, [300], layer=820)
    q, k, v, p, cache = gpu_case(case)
    cache.len.fill_(case.cap)            # one more row does not fit
    out = torch.full_like(q, 5.0)
    k0 = cache.k.clone()
    sd.get_device_error()
    sd.verify_layer(q, k, v, p, case.sections, cache, 0, 1e6, out=out)
    assert sd.get_device_error() & sd.SD_DEVERR_KV_OVERFLOW
    assert cache.len.item() == case.cap
    assert torch.all(out == 5.0)
    assert bool(((cache.k == k0) | (cache.k.isnan() & k0.isnan())).all())


def test_small_tiles_are_served_by_the_small_tile_kernel():
    # the shapes above must reach the small-tile kernel itself (a shape it
    # silently declined would still pass through the tcgen05 kernel)
    for B, Hq, Hkv, K, prefix in SHAPES:
        cap = max(prefix) + K + 9
        assert sd.verify_kernel(B, K + 1, Hq, Hkv, 128, cap) == "small-tile"
        assert sd.lib().sd_verify_kernel(B, K + 1, Hq, Hkv, 128, cap, 2) == b"small-tile"   # block mask
        # the fused layer: from 8 (scene, KV head) clusters on; one scene of
        # the draft's 4 KV heads stays on the tcgen05 layer kernel
        want = "small-tile" if B * Hkv >= 8 else "tcgen05"
        assert sd.verify_kernel(B, K + 1, Hq, Hkv, 128, cap, True) == want
    assert sd.verify_kernel(1, 8, 32, 8, 128, 4104) == "tcgen05"        # 32 rows
    assert sd.verify_kernel(1, 8, 32, 8, 128, 4104, True) == "tcgen05"
    assert sd.verify_kernel(1, 5, 4, 1, 64, 300) == "mma.sync"          # head_dim 64
    assert sd.verify_kernel(1, 5, 4, 1, 64, 300, True) == "three kernels"
