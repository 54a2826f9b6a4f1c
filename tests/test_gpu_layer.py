"""The fused verify layer (sd_verify_layer: M-RoPE + append + attention in one
call) against the three separate calls and against the float64 oracle,
including back-to-back layers issued as programmatic dependent launches."""
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


def _unfused(case):
    q, k_new, v_new, pos, cache = gpu_case(case)
    sd.rope_apply(q, k_new, pos, case.sections, case.interleaved, case.base)
    sd.kv_append(cache, k_new, v_new)
    out = sd.verify_attention(q, cache)
    torch.cuda.synchronize()
    return q, k_new, cache, out


def _fused(case, early=False):
    q, k_new, v_new, pos, cache = gpu_case(case)
    out = sd.verify_layer(q, k_new, v_new, pos, case.sections, cache, case.interleaved, case.base,
                          early=early)
    torch.cuda.synchronize()
    return q, k_new, cache, out


def _check_against_oracle(case, q, cache, out):
    pos = case.pos.numpy()[:, :, None, :]
    ref_q = oracle.mrope_apply(to64(case.q), pos, case.sections, case.interleaved, case.base)
    assert np.all(np.abs(to64(q) - ref_q) <= rope_bound(ref_q, pair_magnitude(to64(case.q))))
    ref_o = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy())
    err = np.abs(to64(out) - ref_o).max()
    assert np.isfinite(to64(out)).all() and attn_within(to64(out), ref_o), err


@pytest.mark.parametrize("make", [workloads.target_layer, workloads.tiny])
def test_fused_equals_separate_calls(make):
    case = make()
    qa, ka, ca, oa = _unfused(case)
    qb, kb, cb, ob = _fused(case)
    assert torch.equal(qa, qb) and torch.equal(ka, kb)            # identical rotations
    assert torch.equal(ca.k, cb.k) and torch.equal(ca.v, cb.v)    # identical appends
    assert torch.equal(ca.len, cb.len)
    _check_against_oracle(case, qb, cb, ob)
    assert (ob.float() - oa.float()).abs().max().item() <= 2 * ATTN_ATOL
    assert sd.get_device_error() == 0


@pytest.mark.parametrize("prefix", [[0, 31, 32], [33, 4095, 64], [5, 127, 128]])
def test_fused_ragged_batch(prefix):
    B = len(prefix)
    R = 8
    qpos = np.stack([workloads.text_positions(int(p) + 1, R) for p in prefix])
    case = workloads.verify_case(workloads.TARGET_LAYER, B=B, Hq=32, Hkv=8, D=128, prefix=prefix, K=R - 1,
                                 sections=(16, 24, 24), base=1e6, query_pos=qpos, cap=max(prefix) + R + 40,
                                 layer=77, tail_fill=float("nan"))
    q, _, cache, out = _fused(case)
    assert cache.len.cpu().tolist() == [p + R for p in prefix]
    _check_against_oracle(case, q, cache, out)
    assert sd.get_device_error() == 0


def test_back_to_back_layers_with_early_prefix():
    # a stack of layers issued back to back: every layer after the first may
    # start streaming its prefix while the previous one runs
    cases = [workloads.target_layer(layer=l) for l in range(6)]
    runs = []
    for early in (False, True):
        outs = []
        state = [gpu_case(c) for c in cases]
        for l, (q, k_new, v_new, pos, cache) in enumerate(state):
            outs.append(sd.verify_layer(q, k_new, v_new, pos, cases[l].sections, cache, 0, 1e6,
                                        early=early and l > 0))
        torch.cuda.synchronize()
        runs.append((outs, state))
    for (oa, sa), (ob, sb) in [(runs[0], runs[1])]:
        for l in range(len(cases)):
            assert torch.equal(oa[l], ob[l])
            assert torch.equal(sa[l][4].k, sb[l][4].k) and torch.equal(sa[l][4].len, sb[l][4].len)
    q, _, _, _, cache = runs[1][1][3]
    _check_against_oracle(cases[3], q, cache, runs[1][0][3])
    assert sd.get_device_error() == 0


@pytest.mark.parametrize("B,K", [(3, 7), (2, 8), (1, 16)])
def test_back_to_back_layers_several_scenes_and_tiles(B, K):
    # chained layers with ragged scenes (the cluster launched last is the last
    # KV head of the last scene) and with the 64-row tile (K = 8: one m-block,
    # K = 16: two): the early chain gives the same bits as the plain one
    R = K + 1
    prefix = [4096 - 37 * s for s in range(B)]
    qpos = np.stack([workloads.text_positions(int(p) + 1, R) for p in prefix])
    cases = [workloads.verify_case(workloads.TARGET_LAYER, B=B, Hq=32, Hkv=8, D=128, prefix=prefix, K=K,
                                   sections=(16, 24, 24), base=1e6, query_pos=qpos, cap=max(prefix) + R + 8,
                                   layer=300 + l) for l in range(4)]
    runs = []
    for early in (False, True):
        outs, state = [], [gpu_case(c) for c in cases]
        for l, (q, k_new, v_new, pos, cache) in enumerate(state):
            outs.append(sd.verify_layer(q, k_new, v_new, pos, cases[l].sections, cache, 0, 1e6,
                                        early=early and l > 0))
        torch.cuda.synchronize()
        runs.append((outs, state))
    (oa, sa), (ob, sb) = runs
    for l in range(len(cases)):
        assert torch.equal(oa[l], ob[l])
        assert torch.equal(sa[l][4].k, sb[l][4].k) and torch.equal(sa[l][4].len, sb[l][4].len)
        assert sb[l][4].len.cpu().tolist() == [p + R for p in prefix]
    q, _, _, _, cache = sb[2]
    _check_against_oracle(cases[2], q, cache, ob[2])
    assert sd.get_device_error() == 0


def test_fused_overflow_sets_error_and_leaves_scene():
    case = workloads.target_layer()
    q, k_new, v_new, pos, cache = gpu_case(case)
    cache.len.fill_(case.cap - 3)            # R = 8 rows do not fit
    out = torch.full_like(q, 5.0)
    sd.get_device_error()
    sd.verify_layer(q, k_new, v_new, pos, case.sections, cache, 0, 1e6, out=out)
    assert sd.get_device_error() & sd.SD_DEVERR_KV_OVERFLOW
    assert cache.len.item() == case.cap - 3
    assert torch.all(out == 5.0)


@pytest.mark.parametrize("K", [15, 16, 23])
def test_fused_layer_long_drafts(K):
    # block-diffusion drafts propose K = 16 tokens at once: R = K + 1 new rows
    # (68 packed rows for K = 16: two 64-row m-blocks) in one fused call
    R = K + 1
    prefix = [4096, 1500]
    qpos = np.stack([workloads.text_positions(int(p) + 1, R) for p in prefix])
    case = workloads.verify_case(workloads.TARGET_LAYER, B=2, Hq=32, Hkv=8, D=128, prefix=prefix, K=K,
                                 sections=(16, 24, 24), base=1e6, query_pos=qpos, cap=max(prefix) + R + 8,
                                 layer=300 + K, tail_fill=float("nan"))
    qa, ka, ca, oa = _unfused(case)
    qb, kb, cb, ob = _fused(case)

    def same(x, y):  # stale cache rows hold NaN on both sides
        return bool(((x == y) | (x.isnan() & y.isnan())).all())

    assert torch.equal(qa, qb) and torch.equal(ka, kb)
    assert same(ca.k, cb.k) and same(ca.v, cb.v) and torch.equal(ca.len, cb.len)
    _check_against_oracle(case, qb, cb, ob)
    assert (ob.float() - oa.float()).abs().max().item() <= 2 * ATTN_ATOL
    assert sd.get_device_error() == 0


@pytest.mark.parametrize("K", [7, 8, 16])
def test_fused_layer_interleaved_mrope(K):
    # interleaved axis assignment a(d) = (T, H, W)[d mod 3] (Sec. 4.2 Eq.
    # axis-assign) through the fused kernel's own rotation table, on the
    # 32-row tile (K = 7), the 64-row tile (K = 8) and two 64-row m-blocks
    # (K = 16); query rows at distinct (t, h, w) so that the layout matters
    R = K + 1
    prefix = [3000, 4096]
    rng = np.random.default_rng(900 + K)
    qpos = rng.integers(0, 5000, size=(2, R, 3)).astype(np.int32)
    case = workloads.verify_case(workloads.TARGET_LAYER, B=2, Hq=32, Hkv=8, D=128, prefix=prefix, K=K,
                                 sections=(16, 24, 24), base=1e6, query_pos=qpos, cap=max(prefix) + R + 8,
                                 interleaved=1, layer=500 + K, tail_fill=float("nan"))
    qa, ka, ca, oa = _unfused(case)
    qb, kb, cb, ob = _fused(case)

    def same(x, y):  # stale cache rows hold NaN on both sides
        return bool(((x == y) | (x.isnan() & y.isnan())).all())

    assert torch.equal(qa, qb) and torch.equal(ka, kb)
    assert same(ca.k, cb.k) and same(ca.v, cb.v) and torch.equal(ca.len, cb.len)
    pos = case.pos.numpy()[:, :, None, :]
    ref_k = oracle.mrope_apply(to64(case.k_new), pos, case.sections, 1, case.base)
    assert np.all(np.abs(to64(kb) - ref_k) <= rope_bound(ref_k, pair_magnitude(to64(case.k_new))))
    for b, p in enumerate(prefix):   # the appended rows are the rotated keys and the values
        assert torch.equal(cb.k[b, :, p:p + R].transpose(0, 1).cpu(), kb[b].cpu())
        assert torch.equal(cb.v[b, :, p:p + R].transpose(0, 1).cpu(), case.v_new[b])
    _check_against_oracle(case, qb, cb, ob)
    # the blocked layout rotates these rows differently: the test sees the layout
    ref_blocked = oracle.mrope_apply(to64(case.q), pos, case.sections, 0, case.base)
    assert np.abs(to64(qb) - ref_blocked).max() > 0.1
    assert sd.get_device_error() == 0
