"""Helpers shared by the GPU parity tests: exact conversions and the GPU
chains that the tests compare against the float64 oracle."""
import numpy as np
import torch

from paper_2606_31160_gb300 import build, sd

# attention tolerance (bf16 I/O, fp32 accumulation): max-abs error vs float64
ATTN_ATOL = 1e-2


def attn_within(out, ref):
    """True when |out - ref| <= 1e-2 + 2^-8 |ref| everywhere: the 1e-2 bound
    plus the rounding of an exact result to bf16 (half an ulp is at most
    2^-8 |x|), which alone exceeds 1e-2 once |x| >= 4 -- rows that see only a
    few keys (short prefixes) average few values and reach that."""
    return bool(np.all(np.abs(out - ref) <= ATTN_ATOL + 2.0 ** -8 * np.abs(ref)))


def ensure_lib():
    build.build()
    return sd.lib()


def to64(t):
    """Exact float64 numpy copy of a bf16 / fp32 tensor (any device)."""
    return t.detach().float().cpu().numpy().astype(np.float64)


def bf16_ulp(x):
    """Spacing of bf16 numbers at |x| (8 significant bits)."""
    x = np.abs(np.asarray(x, dtype=np.float64))
    _, e = np.frexp(np.where(x > 0, x, 1.0))
    ulp = np.ldexp(1.0, e - 8)
    return np.where(x > 0, ulp, np.ldexp(1.0, -133))


def rope_bound(ref, x_in):
    """|gpu - oracle| bound for a rotated bf16 element: half a bf16 ulp of the
    exact value (the final rounding) plus fp32 evaluation error of the rotation."""
    return 0.5 * bf16_ulp(ref) + 2e-6 * (np.abs(x_in) + 1.0)


def pair_magnitude(x):
    """|x_2d| + |x_2d+1| broadcast to every element of the pair."""
    a = np.abs(x[..., 0::2]) + np.abs(x[..., 1::2])
    out = np.empty_like(x)
    out[..., 0::2] = a
    out[..., 1::2] = a
    return out


def gpu_case(case, device="cuda"):
    """Move a workloads.VerifyCase to the device: (q, k_new, v_new, pos, cache)."""
    q = case.q.to(device).contiguous()
    k_new = case.k_new.to(device).contiguous()
    v_new = case.v_new.to(device).contiguous()
    pos = case.pos.to(device).contiguous()
    lens = torch.from_numpy(case.prefix.astype(np.int32)).to(device)
    cache = sd.KVCache(case.k_cache.to(device).contiguous(), case.v_cache.to(device).contiguous(), lens)
    return q, k_new, v_new, pos, cache


def run_verify_layer(case, device="cuda"):
    """GPU chain rope -> append -> attention of one layer; returns
    (rotated q, cache after append, attention output) on the device."""
    q, k_new, v_new, pos, cache = gpu_case(case, device)
    sd.rope_apply(q, k_new, pos, case.sections, case.interleaved, case.base)
    sd.kv_append(cache, k_new, v_new)
    out = sd.verify_attention(q, cache)
    torch.cuda.synchronize()
    return q, k_new, cache, out
