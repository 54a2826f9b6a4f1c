"""GPU parity of sd_kv_append / sd_kv_rollback and of whole verify steps:
the target layer chain (M-RoPE -> append -> attention -> greedy accept ->
rollback) and the draft's FlatRoPE decode loop with append and rollback."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_31160_gb300 import sd, workloads
from tests.helpers import ATTN_ATOL, ensure_lib, rope_bound, pair_magnitude, run_verify_layer, to64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    ensure_lib()


def test_append_matches_shadow_copy():
    rng = np.random.default_rng(90)
    B, H, cap, D, R = 3, 4, 64, 128, 5
    cache = sd.KVCache.empty(B, H, cap, D)
    k0 = workloads.to_bf16(rng.standard_normal((B, H, cap, D)))
    cache.k.copy_(k0.cuda())
    cache.v.copy_(k0.cuda())
    lens = np.array([0, 17, 59])
    cache.len.copy_(torch.from_numpy(lens.astype(np.int32)))
    kn = workloads.to_bf16(rng.standard_normal((B, R, H, D)))
    vn = workloads.to_bf16(rng.standard_normal((B, R, H, D)))
    sd.kv_append(cache, kn.cuda(), vn.cuda())
    ek, ev, el = oracle.kv_append(to64(k0), to64(k0), lens, to64(kn), to64(vn))
    assert sd.get_device_error() == 0
    assert cache.len.cpu().numpy().tolist() == el.tolist()
    assert np.array_equal(to64(cache.k), ek) and np.array_equal(to64(cache.v), ev)


def test_append_overflow_sets_error_and_skips_scene():
    B, H, cap, D, R = 2, 1, 16, 64, 4
    cache = sd.KVCache.empty(B, H, cap, D)
    cache.len.copy_(torch.tensor([12, 13], dtype=torch.int32))
    ones = torch.ones((B, R, H, D), dtype=torch.bfloat16, device="cuda")
    sd.get_device_error()
    sd.kv_append(cache, ones, ones)
    assert sd.get_device_error() & sd.SD_DEVERR_KV_OVERFLOW
    assert cache.len.cpu().tolist() == [16, 13]
    assert float(cache.k[1].abs().sum()) == 0.0


def test_rollback_across_layers_and_errors():
    lens = torch.tensor([[20, 30, 40], [20, 30, 40]], dtype=torch.int32, device="cuda")
    committed = torch.tensor([1, 8, 0], dtype=torch.int32, device="cuda")
    sd.kv_rollback(lens, committed, 8)
    want = oracle.kv_rollback(np.array([20, 30, 40]), [1, 8, 0], 8).tolist()
    assert lens.cpu().tolist() == [want, want]
    sd.get_device_error()
    bad = torch.tensor([9, 0, -1], dtype=torch.int32, device="cuda")
    before = lens.clone()
    sd.kv_rollback(lens, bad, 8)
    assert sd.get_device_error() & sd.SD_DEVERR_ROLLBACK
    assert lens[:, 1].cpu().tolist() == [before[0, 1].item() - 8] * 2
    assert lens[:, 0].cpu().tolist() == before[:, 0].cpu().tolist()


def test_target_layer_step_chain():
    # rope -> append -> attention -> greedy accept -> rollback, each stage
    # checked against the oracle on the values the GPU actually read
    case = workloads.target_layer()
    q, k_rot, cache, out = run_verify_layer(case)
    pos = case.pos.numpy()[:, :, None, :]
    ref_q = oracle.mrope_apply(to64(case.q), pos, case.sections, 0, case.base)
    assert np.all(np.abs(to64(q) - ref_q) <= rope_bound(ref_q, pair_magnitude(to64(case.q))))
    L = int(case.prefix[0])
    ref_k = oracle.mrope_apply(to64(case.k_new), pos, case.sections, 0, case.base)
    got_k = to64(cache.k)[0, :, L:L + case.R].transpose(1, 0, 2)[None]
    assert np.all(np.abs(got_k - ref_k) <= rope_bound(ref_k, pair_magnitude(to64(case.k_new))))
    ref_o = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy())
    assert np.abs(to64(out) - ref_o).max() <= ATTN_ATOL
    n_emit, tokens, _ = sd.accept_greedy(case.extra["logits"].cuda(), case.extra["draft"].cuda())
    rn, rt, _ = oracle.accept_greedy(case.extra["logits"].float().numpy(), case.extra["draft"].numpy())
    assert n_emit.cpu().numpy().tolist() == rn.tolist() and tokens.cpu().numpy().tolist() == rt.tolist()
    sd.kv_rollback(cache.len, n_emit, case.R)
    assert cache.len.cpu().tolist() == oracle.kv_rollback([L + case.R], rn, case.R).tolist()
    assert sd.get_device_error() == 0


def test_draft_flatrope_decode_loop():
    # 7 sequential single-row FlatRoPE decode steps with append, then rollback
    w = workloads.draft_flat()
    L, steps, D = w["L"], w["steps"], w["D"]
    cache = sd.KVCache(w["k_cache"].cuda(), w["v_cache"].cuda(), torch.tensor([L], dtype=torch.int32).cuda())
    for s in range(steps):
        q = w["q"][s].cuda()
        k = w["k_new"][s].cuda()
        sd.rope_apply_1d(q, k, w["pos1d"][s:s + 1].reshape(1, 1).cuda(), w["base"])
        ref_q = oracle.rope_1d(to64(w["q"][s]), L + s, w["base"])
        assert np.all(np.abs(to64(q) - ref_q) <= rope_bound(ref_q, pair_magnitude(to64(w["q"][s]))))
        sd.kv_append(cache, k, w["v_new"][s].cuda())
        out = sd.verify_attention(q, cache)
        ref_o = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy())
        assert np.abs(to64(out) - ref_o).max() <= ATTN_ATOL
    assert cache.len.item() == L + steps
    committed = torch.tensor([w["committed"]], dtype=torch.int32, device="cuda")
    sd.kv_rollback(cache.len, committed, steps)
    assert cache.len.item() == L + w["committed"]
    assert sd.get_device_error() == 0


def test_k_zero_is_plain_decode():
    # K = 0: one row at position L over L + 1 keys equals unmasked attention
    rng = np.random.default_rng(91)
    L, H, D, Hq = 300, 2, 128, 8
    cache = sd.KVCache.empty(1, H, L + 1, D)
    cache.k.copy_(workloads.to_bf16(rng.standard_normal((1, H, L + 1, D))).cuda())
    cache.v.copy_(workloads.to_bf16(rng.standard_normal((1, H, L + 1, D))).cuda())
    cache.len.fill_(L + 1)
    q = workloads.to_bf16(rng.standard_normal((1, 1, Hq, D))).cuda()
    out = sd.verify_attention(q, cache)
    kk = torch.from_numpy(to64(cache.k)[0]).repeat_interleave(Hq // H, 0)
    vv = torch.from_numpy(to64(cache.v)[0]).repeat_interleave(Hq // H, 0)
    qq = torch.from_numpy(to64(q)[0]).permute(1, 0, 2)
    ref = torch.nn.functional.scaled_dot_product_attention(qq, kk, vv).permute(1, 0, 2).numpy()
    assert np.abs(to64(out)[0] - ref).max() <= ATTN_ATOL


def test_draft_step_as_one_fused_layer_call():
    # FlatRoPE is M-RoPE with (m, m, m): the draft's single-row decode step
    # (rotation at m = L + s, append, attention over L + s + 1 keys) as one
    # sd_verify_layer call per step, against the oracle's 1D rotation and attention
    w = workloads.draft_flat()
    L, steps = w["L"], w["steps"]
    cache = sd.KVCache(w["k_cache"].cuda(), w["v_cache"].cuda(), torch.tensor([L], dtype=torch.int32).cuda())
    for s in range(steps):
        q, k = w["q"][s].cuda(), w["k_new"][s].cuda()
        pos = torch.full((1, 1, 3), L + s, dtype=torch.int32, device="cuda")
        out = sd.verify_layer(q, k, w["v_new"][s].cuda(), pos, (16, 24, 24), cache, 0, w["base"])
        ref_q = oracle.rope_1d(to64(w["q"][s]), L + s, w["base"])
        ref_k = oracle.rope_1d(to64(w["k_new"][s]), L + s, w["base"])
        assert np.all(np.abs(to64(q) - ref_q) <= rope_bound(ref_q, pair_magnitude(to64(w["q"][s]))))
        assert np.all(np.abs(to64(k) - ref_k) <= rope_bound(ref_k, pair_magnitude(to64(w["k_new"][s]))))
        assert torch.equal(cache.k[0, :, L + s], k[0, 0]) and torch.equal(cache.v[0, :, L + s], w["v_new"][s][0, 0].cuda())
        ref_o = oracle.verify_attention(to64(q), to64(cache.k), to64(cache.v), cache.len.cpu().numpy())
        assert np.abs(to64(out) - ref_o).max() <= ATTN_ATOL
    assert cache.len.item() == L + steps
    sd.kv_rollback(cache.len, torch.tensor([w["committed"]], dtype=torch.int32, device="cuda"), steps)
    assert cache.len.item() == L + w["committed"]
    assert sd.get_device_error() == 0
