"""Seeded synthetic inputs shaped like the paper's verify-step workloads.

Shared by the tests, bench.py and smoke(); both the CUDA path and the float64
oracle read the arrays made here, so this module holds none of the method's
arithmetic: no rotation, attention, softmax, argmax over model outputs, or
acceptance test. It only draws numbers and lays them out.

The paper's workloads are Alpamayo-R1 driving clips on an 8B Qwen3-VL
backbone (Sec. 5, "Targets and drafts", "Data"); neither the clips nor any
weights are available, so every tensor is synthetic with the shapes and
structure the paper states: a prompt that is ~96% multi-camera vision
patches (Sec. 4.2, "Empirical confirmation"), 15-20-token reasoning outputs
(Sec. 1) and verify blocks of K <= 16 (Sec. 5, "Metric").

Random streams: numpy Generator(Philox(key=(1000 + workload id, layer))).
Normals are drawn in float32 and rounded to bf16 (or kept fp32) before use,
so every consumer reads identical stored values.
"""

from dataclasses import dataclass, field

import numpy as np
import torch

# workload ids (Philox key = 1000 + id)
TINY, TARGET_LAYER, DRAFT_FLAT, SWEEP, STOCHASTIC = 1, 2, 3, 4, 5

# value planted at the intended argmax of each greedy-logit row: 8 standard
# deviations above the N(0, sigma) draws, so it is the unique maximum.
PLANT_SIGMAS = 8.0


def philox(workload, layer=0):
    return np.random.Generator(np.random.Philox(key=[1000 + int(workload), int(layer)]))


def to_bf16(x):
    """float array -> torch.bfloat16 (round to nearest even), contiguous, CPU."""
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)


def uniforms24(rng, shape):
    """u = (32-bit Philox word >> 8) * 2^-24 in [0, 1): exact in fp32 and fp64."""
    words = rng.integers(0, 2 ** 32, size=shape, dtype=np.uint64)
    return ((words >> np.uint64(8)).astype(np.float64) * 2.0 ** -24).astype(np.float32)


def grid_positions(n_vis, grid_h, grid_w):
    """(t, h, w) of n_vis vision patches filling grid_h x grid_w frames row-major,
    t = frame (camera) index. Returns int32 [n_vis, 3]."""
    k = np.arange(n_vis, dtype=np.int64)
    per = grid_h * grid_w
    return np.stack([k // per, (k % per) // grid_w, k % grid_w], axis=1).astype(np.int32)


def text_positions(start, n):
    """Text / trajectory tokens: t = h = w = start, start + 1, ... Returns [n, 3]."""
    m = np.arange(start, start + n, dtype=np.int64)
    return np.stack([m, m, m], axis=1).astype(np.int32)


@dataclass
class VerifyCase:
    """One batch of verify-step inputs for one attention layer (or a ring of layers)."""
    B: int
    R: int
    Hq: int
    Hkv: int
    D: int
    cap: int
    prefix: np.ndarray            # [B] L_b, keys cached before the step
    sections: tuple
    interleaved: int
    base: float
    k_cache: torch.Tensor         # [B, Hkv, cap, D] bf16, rows [0, L_b) filled
    v_cache: torch.Tensor
    q: torch.Tensor               # [B, R, Hq, D] bf16, before rotation
    k_new: torch.Tensor           # [B, R, Hkv, D] bf16, before rotation
    v_new: torch.Tensor           # [B, R, Hkv, D] bf16
    pos: torch.Tensor             # [B, R, 3] int32 (t, h, w) of the query rows
    extra: dict = field(default_factory=dict)

    @property
    def K(self):
        return self.R - 1


def _fill_cache(rng, B, Hkv, cap, D, prefix, tail_fill=0.0):
    """[B, Hkv, cap, D] bf16 with rows [0, L_b) ~ N(0, 1) and the rest tail_fill."""
    k = torch.empty((B, Hkv, cap, D), dtype=torch.bfloat16)
    v = torch.empty((B, Hkv, cap, D), dtype=torch.bfloat16)
    k.fill_(tail_fill)
    v.fill_(tail_fill)
    for b in range(B):
        n = int(prefix[b])
        for g in range(Hkv):
            k[b, g, :n] = to_bf16(rng.standard_normal((n, D), dtype=np.float32))
            v[b, g, :n] = to_bf16(rng.standard_normal((n, D), dtype=np.float32))
    return k, v


def verify_case(workload, *, B, Hq, Hkv, D, prefix, K, sections, base,
                query_pos, cap=None, interleaved=0, layer=0, tail_fill=0.0):
    """Generic verify-step inputs. query_pos: int32 [B, R, 3]."""
    rng = philox(workload, layer)
    R = K + 1
    prefix = np.asarray(prefix, dtype=np.int64).reshape(B)
    if cap is None:
        cap = int(prefix.max()) + R
    k_cache, v_cache = _fill_cache(rng, B, Hkv, cap, D, prefix, tail_fill)
    q = to_bf16(rng.standard_normal((B, R, Hq, D), dtype=np.float32))
    k_new = to_bf16(rng.standard_normal((B, R, Hkv, D), dtype=np.float32))
    v_new = to_bf16(rng.standard_normal((B, R, Hkv, D), dtype=np.float32))
    pos = torch.from_numpy(np.array(query_pos, dtype=np.int32, copy=True))
    return VerifyCase(B, R, Hq, Hkv, D, cap, prefix, tuple(sections), interleaved,
                      float(base), k_cache, v_cache, q, k_new, v_new, pos)


def planted_logits(rng, B, R, V, sigma, dtype, ell):
    """Greedy-acceptance logits [B, R, V] ~ N(0, sigma) with a known argmax.

    Row j of scene b gets the value PLANT_SIGMAS * sigma at a random index
    target[b, j], far above every other draw. The draft copies target[b, :ell_b]
    and differs at position ell_b (when ell_b < K), so exactly ell_b drafts
    match. Returns (logits tensor, draft int32 [B, K], target int32 [B, R]).
    """
    K = R - 1
    z = rng.standard_normal((B, R, V), dtype=np.float32) * np.float32(sigma)
    target = rng.integers(0, V, size=(B, R)).astype(np.int64)
    for b in range(B):
        for j in range(R):
            z[b, j, target[b, j]] = np.float32(PLANT_SIGMAS * sigma)
    draft = rng.integers(0, V, size=(B, K)).astype(np.int64)
    ell = np.asarray(ell, dtype=np.int64).reshape(B)
    for b in range(B):
        draft[b, :ell[b]] = target[b, :ell[b]]
        if ell[b] < K:
            draft[b, ell[b]] = (target[b, ell[b]] + 1) % V
    logits = to_bf16(z) if dtype == "bf16" else torch.from_numpy(z)
    return logits, torch.from_numpy(draft.astype(np.int32)), torch.from_numpy(target.astype(np.int32))


# --------------------------------------------------------------------------
# Named workloads
# --------------------------------------------------------------------------

def tiny(layer=0):
    """Tiny verify step: B=1, 4 q / 1 KV head, D=64, L=256 = 192 vision patches on
    an 8x24 grid at t=0 plus 64 text tokens at t=h=w=1..64; query rows at 65..69;
    M-RoPE sections [8,12,12], base 1e6; K=4; fp32 logits N(0,2) over V=4096 with
    exactly 2 drafts matching."""
    B, K, V = 1, 4, 4096
    R = K + 1
    qpos = text_positions(65, R)[None]
    case = verify_case(TINY, B=B, Hq=4, Hkv=1, D=64, prefix=[256], K=K,
                       sections=(8, 12, 12), base=1e6, query_pos=qpos, layer=layer)
    rng = philox(TINY, 100 + layer)
    logits, draft, target = planted_logits(rng, B, R, V, 2.0, "f32", [2])
    case.extra.update(logits=logits, draft=draft, target=target, ell=np.array([2]), V=V,
                      prefix_pos=np.concatenate([grid_positions(192, 8, 24), text_positions(1, 64)]))
    return case


def target_layer(B=1, layer=0, ell=None, scene=0):
    """8B-class target layer: 32 q / 8 KV heads x 128, sections [16,24,24], base 1e6.
    Prefix L=4096 = 4 cameras x 896 patches (28x32 grid, t = camera) + 512 text
    tokens at 32..543; K=7 query rows at 544..551. Greedy logits bf16 N(0,2) over
    V=151936 with the matching-prefix length uniform in 0..7. `scene` selects an
    independent draw (another driving clip): scene 0 is the default stream."""
    K, V, L = 7, 151936, 4096
    R = K + 1
    off = 10000 * int(scene)
    qpos = np.broadcast_to(text_positions(544, R)[None], (B, R, 3))
    case = verify_case(TARGET_LAYER, B=B, Hq=32, Hkv=8, D=128, prefix=[L] * B, K=K,
                       sections=(16, 24, 24), base=1e6, query_pos=qpos, layer=layer + off)
    rng = philox(TARGET_LAYER, 100 + layer + off)
    if ell is None:
        ell = rng.integers(0, K + 1, size=B)
    logits, draft, target = planted_logits(rng, B, R, V, 2.0, "bf16", ell)
    case.extra.update(logits=logits, draft=draft, target=target, ell=np.asarray(ell).reshape(B), V=V)
    return case


def target_prefix_positions():
    """(t, h, w) of the 4096-token target prefix: 4 x (28x32) patches then text 32..543."""
    return np.concatenate([grid_positions(4 * 896, 28, 32), text_positions(32, 512)])


def draft_flat(layer=0, steps=7):
    """Draft side, FlatRoPE: the same 4096-token prefix with positions flattened to
    0..L-1, 16 q / 4 KV heads x 128, base 1e6; `steps` sequential single-row decode
    steps at positions L .. L+steps-1, then a rollback to a committed count drawn
    from 0..steps."""
    L = 4096
    rng = philox(DRAFT_FLAT, layer)
    k_cache, v_cache = _fill_cache(rng, 1, 4, L + steps, 128, [L])
    q = to_bf16(rng.standard_normal((steps, 1, 1, 16, 128), dtype=np.float32))
    k_new = to_bf16(rng.standard_normal((steps, 1, 1, 4, 128), dtype=np.float32))
    v_new = to_bf16(rng.standard_normal((steps, 1, 1, 4, 128), dtype=np.float32))
    pos1d = torch.arange(L, L + steps, dtype=torch.int32)
    committed = int(rng.integers(0, steps + 1))
    return dict(L=L, steps=steps, Hq=16, Hkv=4, D=128, base=1e6, k_cache=k_cache,
                v_cache=v_cache, q=q, k_new=k_new, v_new=v_new, pos1d=pos1d,
                committed=committed)


def sweep_case(B, L, K, layer=0):
    """Batched verify sweep: B scenes with ragged prefixes L_b ~ U{ceil(0.75L)..L},
    87.5% vision patches (28x32 grids, t = grid index) then text; 32 q / 8 KV x 128,
    sections [16,24,24], base 1e6; capacity L + 17."""
    rng = philox(SWEEP, 7919 * layer + 31 * B + K)
    lo = -(-3 * L // 4)
    prefix = rng.integers(lo, L + 1, size=B)
    R = K + 1
    qpos = np.empty((B, R, 3), dtype=np.int32)
    for b in range(B):
        n_vis = (7 * int(prefix[b])) // 8
        vis = grid_positions(n_vis, 28, 32)
        start = int(vis.max()) + 1 if n_vis else 0
        n_text = int(prefix[b]) - n_vis
        qpos[b] = text_positions(start + n_text, R)
    return verify_case(SWEEP, B=B, Hq=32, Hkv=8, D=128, prefix=prefix, K=K,
                       sections=(16, 24, 24), base=1e6, query_pos=qpos,
                       cap=L + 17, layer=1000 * layer + 31 * B + K)


def sweep_case_device(B, L, K, device, layer=0):
    """The batched-sweep recipe at timing sizes, drawn on the device: the same
    ragged prefix lengths L_b and query positions as sweep_case (same Philox
    stream), K/V prefix rows, q, k_new and v_new ~ N(0, 1) bf16 from a seeded
    device generator (torch Philox), cache tails zero. Returns (prefix int64
    [B], q, k_new, v_new, pos, k_cache, v_cache, cap)."""
    rng = philox(SWEEP, 7919 * layer + 31 * B + K)
    lo = -(-3 * L // 4)
    prefix = rng.integers(lo, L + 1, size=B)
    R, Hq, Hkv, D, cap = K + 1, 32, 8, 128, L + 17
    qpos = np.empty((B, R, 3), dtype=np.int32)
    for b in range(B):
        n_vis = (7 * int(prefix[b])) // 8
        start = int(grid_positions(n_vis, 28, 32).max()) + 1 if n_vis else 0
        qpos[b] = text_positions(start + int(prefix[b]) - n_vis, R)
    gen = torch.Generator(device=device)
    gen.manual_seed(1000 * (1000 + SWEEP) + 7919 * layer + 31 * B + K)

    def normal(*shape):
        return torch.randn(shape, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)

    k_cache = torch.zeros((B, Hkv, cap, D), dtype=torch.bfloat16, device=device)
    v_cache = torch.zeros_like(k_cache)
    for b in range(B):
        n = int(prefix[b])
        k_cache[b, :, :n] = normal(Hkv, n, D)
        v_cache[b, :, :n] = normal(Hkv, n, D)
    q, k_new, v_new = normal(B, R, Hq, D), normal(B, R, Hkv, D), normal(B, R, Hkv, D)
    pos = torch.from_numpy(qpos).to(device)
    return prefix, q, k_new, v_new, pos, k_cache, v_cache, cap


def stochastic(B=8, K=7, V=151936, temperature=0.6, sigma_t=3.0, sigma_noise=0.5, seed_layer=0):
    """Stochastic acceptance inputs: fp32 target logits z_T ~ N(0, sigma_t) [B, K+1, V],
    draft logits z_D = z_T[:, :K] + N(0, sigma_noise) [B, K, V], draft tokens drawn
    from softmax(z_D / T) by the Gumbel-max trick on the same Philox stream, and
    uniforms u [B, K+1] (G12 form)."""
    rng = philox(STOCHASTIC, seed_layer)
    z_t = rng.standard_normal((B, K + 1, V), dtype=np.float32) * np.float32(sigma_t)
    z_d = z_t[:, :K] + rng.standard_normal((B, K, V), dtype=np.float32) * np.float32(sigma_noise)
    g = -np.log(-np.log(rng.random((B, K, V)) * (1 - 2 ** -53) + 2 ** -54))
    draft = np.argmax(z_d.astype(np.float64) / temperature + g, axis=-1).astype(np.int32)
    u = uniforms24(rng, (B, K + 1))
    return dict(z_target=torch.from_numpy(np.ascontiguousarray(z_t)),
                z_draft=torch.from_numpy(np.ascontiguousarray(z_d)),
                draft=torch.from_numpy(draft), u=torch.from_numpy(u),
                temperature=float(temperature), B=B, K=K, V=V)
