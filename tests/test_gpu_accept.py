"""GPU parity of sd_accept_greedy and sd_accept_sample against the float64 oracle.

Greedy: n_emit, tokens and argmax bit-exact. Sampling: bit-exact on every
decision that sits clear of its boundary in the oracle's float64 arithmetic
-- acceptance tests farther than ACCEPT_MARGIN (relative) and the final draw
farther than DRAW_MARGIN (probability units) from a step of the cumulative
sum; these bounds sit well above the fp32 error of the kernel's normalisers
(~1e-6 relative) and running sums (~1e-6 absolute). A near decision leaves
open only what depends on it: the accepted length and prefix before it are
still checked. Near decisions are counted per seed.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_31160_gb300 import sd, workloads
from tests.helpers import ensure_lib

pytestmark = pytest.mark.gpu

ACCEPT_MARGIN = 1e-5
DRAW_MARGIN = 2e-6


@pytest.fixture(scope="module", autouse=True)
def _lib():
    ensure_lib()


def _greedy_both(logits, draft):
    n, t, a = sd.accept_greedy(logits.cuda(), draft.cuda())
    rn, rt, ra = oracle.accept_greedy(logits.float().numpy(), draft.numpy())
    assert n.cpu().numpy().tolist() == rn.tolist()
    assert t.cpu().numpy().tolist() == rt.tolist()
    assert a.cpu().numpy().tolist() == ra.tolist()
    return rn


@pytest.mark.parametrize("make", [workloads.tiny, workloads.target_layer])
def test_greedy_workloads(make):
    case = make()
    rn = _greedy_both(case.extra["logits"], case.extra["draft"])
    assert rn.tolist() == (case.extra["ell"] + 1).tolist()


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
# V * element size a multiple of 16 bytes takes the cluster kernel (V = 151936
# fp32 with K = 16: 17 rows in four passes over 37,984-byte slices); other V
# the chunked kernel
@pytest.mark.parametrize("B,K,V", [(1, 0, 5), (3, 1, 4097), (8, 7, 151936), (2, 16, 32000), (5, 3, 123457),
                                   (2, 16, 151936)])
def test_greedy_random(dtype, B, K, V):
    rng = np.random.default_rng(B * 1000 + K + V)
    z = rng.standard_normal((B, K + 1, V)).astype(np.float32) * 2
    logits = torch.from_numpy(z).to(dtype)
    star = logits.float().argmax(-1).numpy()
    draft = np.where(rng.random((B, K)) < 0.7, star[:, :K], rng.integers(0, V, (B, K)))
    _greedy_both(logits, torch.from_numpy(draft.astype(np.int32)))


def test_greedy_all_match_and_planted_ties():
    B, K, V = 4, 7, 151936
    rng = np.random.default_rng(70)
    z = rng.standard_normal((B, K + 1, V)).astype(np.float32)
    # ties of the maximum in different chunks of the vocabulary, +0 / -0 ties,
    # and a row whose every entry is equal
    z[0, 0, [5, 70000, 151935]] = 9.0
    z[0, 1, [151935, 4096, 4095]] = 9.0
    z[1, 2, :] = -1.0
    z[1, 3, :] = 0.0
    z[1, 3, [100, 7]] = -0.0
    z[2, 0, [60000, 60001]] = np.float32(8.5)
    logits = torch.from_numpy(z).to(torch.bfloat16)
    star = oracle.accept_greedy(logits.float().numpy(), np.zeros((B, K), np.int64))[2]
    assert star[0, 0] == 5 and star[0, 1] == 4095 and star[1, 2] == 0 and star[1, 3] == 0
    draft = torch.from_numpy(star[:, :K].astype(np.int32))   # all drafts match
    rn = _greedy_both(logits, draft)
    assert rn.tolist() == [K + 1] * B


def test_greedy_workspace_reuse_and_counters_rearm():
    case = workloads.target_layer()
    logits, draft = case.extra["logits"].cuda(), case.extra["draft"].cuda()
    ws = sd.workspace(sd.greedy_workspace_bytes(1, 7, logits.shape[-1]))
    first = [x.clone() for x in sd.accept_greedy(logits, draft, ws=ws)]
    for _ in range(3):
        again = sd.accept_greedy(logits, draft, ws=ws)
        assert all(torch.equal(a, b) for a, b in zip(first, again))
    assert sd.get_device_error() == 0


def test_greedy_draft_out_of_range_sets_error():
    logits = torch.zeros((1, 3, 10), dtype=torch.float32, device="cuda")
    draft = torch.tensor([[0, 12]], dtype=torch.int32, device="cuda")
    sd.get_device_error()
    n, t, _ = sd.accept_greedy(logits, draft)
    assert sd.get_device_error() & sd.SD_DEVERR_TOKEN_RANGE
    assert n.item() == 2   # draft 0 matches argmax 0; draft 1 never can


# ------------------------------------------------------------------ sampling

def _sample_both(z_t, z_d, draft, u, T):
    """Kernel against oracle, every decision that the oracle's float64 margins
    decide. Acceptance tests are taken in order; when test j sits within
    ACCEPT_MARGIN of its boundary the tests before it were clear accepts, so
    the kernel must have accepted drafts 0..j-1 (n_emit > j, tokens[:j] equal)
    and only what follows test j is left open. When every acceptance test is
    clear, n_emit and the accepted prefix are exact, and the drawn token is too
    unless the draw sits within DRAW_MARGIN of a step of its cumulative sum.
    Returns (oracle n_emit, scenes with a near acceptance test, scenes whose
    only near decision is the final draw)."""
    n, t = sd.accept_sample(z_t.cuda(), z_d.cuda(), draft.cuda(), u.cuda(), T)
    rn, rt, margins = oracle.accept_sample(z_t.numpy(), z_d.numpy(), draft.numpy(), u.numpy(), T)
    n, t = n.cpu().numpy(), t.cpu().numpy()
    V = z_t.shape[-1]
    accept_near, draw_near = [], []
    for b in range(len(rn)):
        acc_m, draw_m = margins[b][:-1], margins[b][-1]
        assert 1 <= n[b] <= t.shape[1] and (t[b][n[b]:] == -1).all(), (b, n[b], t[b])
        j_near = next((j for j, m in enumerate(acc_m) if m < ACCEPT_MARGIN), None)
        if j_near is not None:
            accept_near.append(b)
            assert n[b] >= j_near + 1, (b, n[b], j_near)
            assert t[b][:j_near].tolist() == rt[b][:j_near].tolist(), (b, t[b], rt[b])
            continue
        assert n[b] == rn[b], (b, n[b], rn[b])
        assert t[b][:rn[b] - 1].tolist() == rt[b][:rn[b] - 1].tolist(), (b, t[b], rt[b])
        if draw_m < DRAW_MARGIN:
            draw_near.append(b)
            assert 0 <= t[b][rn[b] - 1] < V
        else:
            assert t[b][rn[b] - 1] == rt[b][rn[b] - 1], (b, t[b], rt[b])
    return rn, accept_near, draw_near


def test_sample_stochastic_workload():
    w = workloads.stochastic()
    rn, accept_near, draw_near = _sample_both(w["z_target"], w["z_draft"], w["draft"], w["u"], w["temperature"])
    assert accept_near == [] and draw_near == []
    assert rn.min() >= 1 and rn.max() <= w["K"] + 1


# scenes (of 16) whose final draw the oracle puts within DRAW_MARGIN of a step
# of its cumulative sum, per seed: only their drawn token goes unchecked
DRAW_NEAR_PER_SEED = (0, 0, 1, 2)


@pytest.mark.parametrize("seed", range(4))
def test_sample_more_seeds(seed):
    # flatter T = 0.8 rows over 50k tokens: smaller steps in the cumulative sums
    w = workloads.stochastic(B=16, K=5, V=50000, temperature=0.8, seed_layer=10 + seed)
    rn, accept_near, draw_near = _sample_both(w["z_target"], w["z_draft"], w["draft"], w["u"], w["temperature"])
    print("seed %d: near acceptance tests %s, near final draws %s" % (seed, accept_near, draw_near))
    assert accept_near == []
    assert len(draw_near) == DRAW_NEAR_PER_SEED[seed]


def test_sample_equal_distributions_always_accept():
    rng = np.random.default_rng(80)
    B, K, V = 8, 7, 20000
    z = torch.from_numpy(rng.standard_normal((B, K + 1, V)).astype(np.float32))
    draft = torch.from_numpy(rng.integers(0, V, (B, K)).astype(np.int32))
    u = torch.from_numpy(workloads.uniforms24(rng, (B, K + 1)))
    n, t = sd.accept_sample(z.cuda(), z[:, :K].contiguous().cuda(), draft.cuda(), u.cuda(), 0.7)
    assert n.cpu().tolist() == [K + 1] * B
    assert torch.equal(t[:, :K].cpu(), draft)


# V = 5 takes the scalar stats kernel, V = 8 (a multiple of 4) the streaming one
@pytest.mark.parametrize("V", [5, 8])
def test_sample_output_law_by_enumeration_on_gpu(V):
    # Leviathan/Chen on a small vocabulary through the kernel: every draft
    # token x (weight q(x)) times an N x N grid of uniforms, in one batch.
    rng = np.random.default_rng(81)
    T, N = 0.8, 64
    z_t = (rng.standard_normal((2, V)) * 1.5).astype(np.float32)
    z_d = (rng.standard_normal((1, V)) * 1.5).astype(np.float32)
    grid = (np.arange(N) + 0.5) / N
    u0, u1 = np.meshgrid(grid, grid, indexing="ij")
    u = np.stack([u0.ravel(), u1.ravel()], 1).astype(np.float32)
    n = u.shape[0]
    B = V * n
    zt = torch.from_numpy(np.ascontiguousarray(np.broadcast_to(z_t, (B, 2, V))))
    zd = torch.from_numpy(np.ascontiguousarray(np.broadcast_to(z_d, (B, 1, V))))
    draft = torch.from_numpy(np.repeat(np.arange(V), n).astype(np.int32).reshape(B, 1))
    uu = torch.from_numpy(np.tile(u, (V, 1)))
    nn, tt = sd.accept_sample(zt.cuda(), zd.cuda(), draft.cuda(), uu.cuda(), T)
    first = tt[:, 0].cpu().numpy().reshape(V, n)
    q = np.exp((z_d[0] - z_d[0].max()) / T)
    q /= q.sum()
    p = np.exp((z_t[0] - z_t[0].max()) / T)
    p /= p.sum()
    dist = sum(q[x] * np.bincount(first[x], minlength=V) / n for x in range(V))
    np.testing.assert_allclose(dist, p, atol=2.0 / N + 1e-6)
