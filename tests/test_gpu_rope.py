"""GPU parity of sd_rope_apply / sd_rope_apply_1d against the float64 oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_31160_gb300 import sd, workloads
from tests.helpers import ensure_lib, to64, rope_bound, pair_magnitude

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    ensure_lib()


def _check(got, ref, x_in):
    err = np.abs(got - ref)
    bound = rope_bound(ref, pair_magnitude(x_in))
    assert np.all(err <= bound), float((err - bound).max())
    # nearly every element is the correctly rounded value itself
    exact = to64(torch.from_numpy(ref.astype(np.float32)).to(torch.bfloat16))
    assert np.mean(got == exact) > 0.995


@pytest.mark.parametrize("make", [workloads.tiny, workloads.target_layer])
def test_mrope_matches_oracle_on_workloads(make):
    case = make()
    q = case.q.cuda()
    k = case.k_new.cuda()
    sd.rope_apply(q, k, case.pos.cuda(), case.sections, 0, case.base)
    pos = case.pos.numpy()[:, :, None, :]
    _check(to64(q), oracle.mrope_apply(to64(case.q), pos, case.sections, 0, case.base), to64(case.q))
    _check(to64(k), oracle.mrope_apply(to64(case.k_new), pos, case.sections, 0, case.base), to64(case.k_new))


@pytest.mark.parametrize("D,sec", [(64, (8, 12, 12)), (128, (16, 24, 24)), (128, (64, 0, 0))])
@pytest.mark.parametrize("inter", [0, 1])
@pytest.mark.parametrize("base", [1e4, 1e6])
def test_mrope_vision_coordinates(D, sec, inter, base):
    rng = np.random.default_rng(60)
    B, R, Hq, Hkv = 3, 5, 8, 2
    x = workloads.to_bf16(rng.standard_normal((B, R, Hq, D)))
    y = workloads.to_bf16(rng.standard_normal((B, R, Hkv, D)))
    pos = torch.from_numpy(rng.integers(0, 40, size=(B, R, 3)).astype(np.int32))
    q, k = x.cuda(), y.cuda()
    sd.rope_apply(q, k, pos.cuda(), sec, inter, base)
    p = pos.numpy()[:, :, None, :]
    _check(to64(q), oracle.mrope_apply(to64(x), p, sec, inter, base), to64(x))
    _check(to64(k), oracle.mrope_apply(to64(y), p, sec, inter, base), to64(y))


@pytest.mark.parametrize("m0", [0, 4096, 16400, (1 << 20) - 8, (1 << 23) + 5])
def test_angle_precision_at_large_positions(m0):
    # positions up to 2^23: the angle stays accurate to ~1e-7 rad
    rng = np.random.default_rng(61)
    R, H, D = 8, 4, 128
    x = workloads.to_bf16(rng.standard_normal((1, R, H, D)))
    pos1d = torch.arange(m0, m0 + R, dtype=torch.int32).reshape(1, R)
    q = x.cuda()
    k = torch.zeros((1, R, 1, D), dtype=torch.bfloat16, device="cuda")
    sd.rope_apply_1d(q, k, pos1d.cuda(), 1e6)
    ref = np.stack([oracle.rope_1d(to64(x)[0, r], m0 + r, 1e6) for r in range(R)])[None]
    _check(to64(q), ref, to64(x))


def test_flatrope_equals_mrope_with_equal_coordinates_bitwise():
    # FlatRoPE (Eq. flatrope-proj) is M-RoPE at (m, m, m) under any section layout
    rng = np.random.default_rng(62)
    B, R, Hq, Hkv, D = 2, 7, 16, 4, 128
    x = workloads.to_bf16(rng.standard_normal((B, R, Hq, D)))
    y = workloads.to_bf16(rng.standard_normal((B, R, Hkv, D)))
    m = torch.from_numpy(rng.integers(0, 20000, size=(B, R)).astype(np.int32))
    flat_q, flat_k = x.cuda(), y.cuda()
    sd.rope_apply_1d(flat_q, flat_k, m.cuda(), 1e6)
    pos3 = m[..., None].expand(B, R, 3).contiguous().cuda()
    for sec, inter in [((16, 24, 24), 0), ((16, 24, 24), 1), ((64, 0, 0), 0), ((0, 32, 32), 1)]:
        q, k = x.cuda(), y.cuda()
        sd.rope_apply(q, k, pos3, sec, inter, 1e6)
        assert torch.equal(q, flat_q) and torch.equal(k, flat_k)
    ref = oracle.mrope_apply(to64(x), oracle.flatrope_positions(m.numpy())[:, :, None, :], (16, 24, 24), 0, 1e6)
    _check(to64(flat_q), ref, to64(x))


def test_position_zero_is_identity_and_k_may_be_empty():
    rng = np.random.default_rng(63)
    x = workloads.to_bf16(rng.standard_normal((2, 3, 4, 64)))
    q = x.cuda()
    k = torch.empty((2, 3, 0, 64), dtype=torch.bfloat16, device="cuda")
    sd.rope_apply(q, k, torch.zeros((2, 3, 3), dtype=torch.int32, device="cuda"), (8, 12, 12), 0, 1e6)
    assert torch.equal(q.cpu(), x)
