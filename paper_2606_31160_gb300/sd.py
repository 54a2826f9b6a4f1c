"""ctypes binding of libsd.so: the C ABI of include/sd.h with torch tensors.

Argument marshalling only: every function checks shapes / dtypes / devices,
passes `tensor.data_ptr()` and torch's current CUDA stream to the C entry
point of the same name, and raises SDError on a non-zero status. All the
arithmetic of the verify step runs in the CUDA kernels of libsd.so; there is
no CPU fallback, and loading fails loudly when the library is missing.
"""

import ctypes
import os
import re

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libsd.so")
HEADER_PATH = os.path.join(os.path.dirname(_PKG), "include", "sd.h")

SD_BF16, SD_F32 = 0, 1
SD_DEVERR_KV_OVERFLOW = 0x1
SD_DEVERR_ROLLBACK = 0x2
SD_DEVERR_TOKEN_RANGE = 0x4
SD_DEVERR_LENGTH = 0x8
SD_DEVERR_TIMEOUT = 0x10


class SDError(RuntimeError):
    def __init__(self, what, status):
        super().__init__("%s failed: %s" % (what, status_str(status)))
        self.status = status


class KVCacheStruct(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("len", ctypes.c_void_p),
                ("batch", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("capacity", ctypes.c_int32), ("head_dim", ctypes.c_int32)]


_lib = None

_vp, _i, _f, _sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
_SIGNATURES = {
    "sd_status_str": ([_i], ctypes.c_char_p),
    "sd_version": ([], ctypes.c_char_p),
    "sd_rope_apply": ([_vp, _vp, _i, _i, _i, _i, _i, _vp, ctypes.POINTER(ctypes.c_int32), _i, _f, _vp], _i),
    "sd_rope_apply_1d": ([_vp, _vp, _i, _i, _i, _i, _i, _vp, _f, _vp], _i),
    "sd_kv_append": ([ctypes.POINTER(KVCacheStruct), _vp, _vp, _i, _vp], _i),
    "sd_kv_rollback": ([_vp, _i, _i, _vp, _i, _vp], _i),
    "sd_verify_attention_workspace": ([_i, _i, _i, _i, _i, _i], _sz),
    "sd_verify_attention": ([_vp, ctypes.POINTER(KVCacheStruct), _vp, _i, _i, _f, _vp, _sz, _vp], _i),
    "sd_verify_attention_ex": ([_vp, ctypes.POINTER(KVCacheStruct), _vp, _i, _i, _f, _i, _vp, _sz, _vp], _i),
    "sd_verify_layer_workspace": ([_i, _i, _i, _i, _i, _i], _sz),
    "sd_verify_layer": ([_vp, _vp, _vp, _vp, ctypes.POINTER(ctypes.c_int32), _i, _f,
                         ctypes.POINTER(KVCacheStruct), _vp, _i, _i, _f, _vp, _sz, _i, _vp], _i),
    "sd_accept_greedy_workspace": ([_i, _i, _i], _sz),
    "sd_accept_greedy": ([_vp, _i, _i, _i, _i, _vp, _vp, _vp, _vp, _vp, _sz, _vp], _i),
    "sd_accept_greedy_noalloc": ([_vp, _i, _i, _i, _i, _vp, _vp, _vp, _vp, _vp], _i),
    "sd_accept_greedy_noalloc_max_bytes": ([], _sz),
    "sd_accept_sample_workspace": ([_i, _i, _i], _sz),
    "sd_accept_sample": ([_vp, _vp, _i, _i, _i, _f, _vp, _vp, _vp, _vp, _vp, _sz, _vp], _i),
    "sd_get_device_error": ([_vp, ctypes.POINTER(ctypes.c_uint32)], _i),
    "sd_set_cluster_size": ([_i], _i),
    "sd_verify_kernel": ([_i, _i, _i, _i, _i, _i, _i], ctypes.c_char_p),
    "sd_attention_budget": ([_vp, ctypes.POINTER(KVCacheStruct), _i, _i, _f, _vp, _vp, _vp, _vp], _i),
}


def lib():
    """Load libsd.so (built in-tree by paper_2606_31160_gb300.build)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libsd.so not found at %s: run paper_2606_31160_gb300.build.build() "
                               "(there is no CPU fallback)" % LIB_PATH)
        handle = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGNATURES.items():
            fn = getattr(handle, name)
            fn.argtypes = args
            fn.restype = res
        _lib = handle
    return _lib


def header_symbols():
    """Names of every function include/sd.h declares."""
    with open(HEADER_PATH) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(sd_[a-z0-9_]+)\s*\(", text)))


def status_str(status):
    return lib().sd_status_str(int(status)).decode()


def version():
    return lib().sd_version().decode()


def _check(status, what):
    if status != 0:
        raise SDError(what, status)


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _dev(t, name, dtype=None, ndim=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError("%s must be a torch.Tensor" % name)
    if not t.is_cuda:
        raise ValueError("%s must be on a CUDA device (no CPU path exists)" % name)
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if dtype is not None and t.dtype != dtype:
        raise ValueError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if ndim is not None and t.dim() != ndim:
        raise ValueError("%s must have %d dims, got %s" % (name, ndim, tuple(t.shape)))
    return ctypes.c_void_p(t.data_ptr())


def workspace(nbytes, device=None):
    """A zero-filled device workspace of at least nbytes (16-byte aligned)."""
    return torch.zeros(max(int(nbytes), 16), dtype=torch.uint8,
                       device=device if device is not None else torch.cuda.current_device())


# ----------------------------------------------------------------------- RoPE

def rope_apply(q, k, pos, sections, interleaved=0, base=1e6):
    """In-place M-RoPE of q [B,R,Hq,D] and k [B,R,Hkv,D] (bf16) at pos [B,R,3] int32."""
    B, R, Hq, D = q.shape
    Hkv = k.shape[2]
    if tuple(k.shape) != (B, R, Hkv, D) or tuple(pos.shape) != (B, R, 3):
        raise ValueError("shape mismatch")
    sec = (ctypes.c_int32 * 3)(*[int(s) for s in sections])
    _check(lib().sd_rope_apply(_dev(q, "q", torch.bfloat16), _dev(k, "k", torch.bfloat16), B, R, Hq,
                               Hkv, D, _dev(pos, "pos", torch.int32), sec, int(interleaved),
                               float(base), _stream()), "sd_rope_apply")


def rope_apply_1d(q, k, pos1d, base=1e6):
    """In-place FlatRoPE / 1D RoPE at sequence positions pos1d [B,R] int32."""
    B, R, Hq, D = q.shape
    Hkv = k.shape[2]
    if tuple(k.shape) != (B, R, Hkv, D) or tuple(pos1d.shape) != (B, R):
        raise ValueError("shape mismatch")
    _check(lib().sd_rope_apply_1d(_dev(q, "q", torch.bfloat16), _dev(k, "k", torch.bfloat16), B, R,
                                  Hq, Hkv, D, _dev(pos1d, "pos1d", torch.int32), float(base),
                                  _stream()), "sd_rope_apply_1d")


# ------------------------------------------------------------------ KV cache

class KVCache:
    """One layer's bf16 KV cache [B, Hkv, cap, D] plus its device lengths [B]."""

    def __init__(self, k, v, lens):
        if k.shape != v.shape or k.dim() != 4:
            raise ValueError("k and v must both be [B, Hkv, cap, D]")
        _dev(k, "k", torch.bfloat16)
        _dev(v, "v", torch.bfloat16)
        _dev(lens, "len", torch.int32, 1)
        self.k, self.v, self.len = k, v, lens
        B, H, cap, D = k.shape
        self._struct = KVCacheStruct(k.data_ptr(), v.data_ptr(), lens.data_ptr(), B, H, cap, D)

    @classmethod
    def empty(cls, B, Hkv, cap, D, device="cuda"):
        k = torch.zeros((B, Hkv, cap, D), dtype=torch.bfloat16, device=device)
        return cls(k, torch.zeros_like(k), torch.zeros(B, dtype=torch.int32, device=device))

    @property
    def struct(self):
        return ctypes.byref(self._struct)

    @property
    def shape(self):
        return tuple(self.k.shape)


def kv_append(cache, k_new, v_new):
    """Write k_new / v_new [B,R,Hkv,D] at len[b] .. len[b]+R-1; len += R."""
    B, H, _, D = cache.shape
    R = k_new.shape[1]
    if tuple(k_new.shape) != (B, R, H, D) or k_new.shape != v_new.shape:
        raise ValueError("shape mismatch")
    _check(lib().sd_kv_append(cache.struct, _dev(k_new, "k_new", torch.bfloat16),
                              _dev(v_new, "v_new", torch.bfloat16), R, _stream()), "sd_kv_append")


def kv_rollback(lens, committed, n_appended):
    """lens [..., B] (one or more layers' length arrays, contiguous) -= n_appended - committed[b]."""
    B = committed.numel()
    _check(lib().sd_kv_rollback(_dev(lens, "len", torch.int32), lens.numel(), B,
                                _dev(committed, "committed", torch.int32), int(n_appended), _stream()),
           "sd_kv_rollback")


# ----------------------------------------------------------------- attention

def attention_workspace_bytes(B, R, Hq, Hkv, D, capacity):
    return int(lib().sd_verify_attention_workspace(B, R, Hq, Hkv, D, capacity))


_attn_ws = {}


SD_ATTN_BLOCK_MASK = 1
SD_ATTN_PREFIX_EARLY = 2
SD_LAYER_BLOCK_MASK = 2


def verify_attention(q, cache, out=None, scale=0.0, ws=None, block=False, early=False):
    """Causal GQA verify attention of q [B,R,Hq,D] (rotated) over the cache (appended).
    ws: the split-merge workspace (see sd_verify_attention_workspace); when None a
    zero-filled one is kept per (device, shape) and reused by later calls.
    block=True sets SD_ATTN_BLOCK_MASK; early=True sets SD_ATTN_PREFIX_EARLY (the
    previous kernel on the stream writes neither this cache nor its len)."""
    B, R, Hq, D = q.shape
    if cache.shape[0] != B or cache.shape[3] != D:
        raise ValueError("q and cache disagree")
    if out is None:
        out = torch.empty_like(q)
    if ws is None:
        need = attention_workspace_bytes(B, R, Hq, cache.shape[1], D, cache.shape[2])
        key = (q.device.index, need)
        if need and key not in _attn_ws:
            _attn_ws[key] = workspace(need, q.device)
        ws = _attn_ws.get(key)
    wp = _dev(ws, "ws") if ws is not None else ctypes.c_void_p(0)
    nbytes = ws.numel() * ws.element_size() if ws is not None else 0
    _check(lib().sd_verify_attention_ex(_dev(q, "q", torch.bfloat16), cache.struct,
                                        _dev(out, "out", torch.bfloat16), R, Hq, float(scale),
                                        (SD_ATTN_BLOCK_MASK if block else 0) | (SD_ATTN_PREFIX_EARLY if early else 0),
                                        wp, nbytes, _stream()),
           "sd_verify_attention")
    return out


def attention_budget(q, cache, n_visual, scale=0.0, mass=None, entropy=None):
    """Per (scene, row, head): attention mass on the visual, trajectory / text and
    generated keys, and the normalised entropy over the non-visual keys.
    q [B,R,Hq,D] (rotated), cache appended, n_visual int32 [B] -> (mass [B,R,Hq,3],
    entropy [B,R,Hq]) float32."""
    B, R, Hq, D = q.shape
    if mass is None:
        mass = torch.empty((B, R, Hq, 3), dtype=torch.float32, device=q.device)
    if entropy is None:
        entropy = torch.empty((B, R, Hq), dtype=torch.float32, device=q.device)
    _check(lib().sd_attention_budget(_dev(q, "q", torch.bfloat16), cache.struct, R, Hq, float(scale),
                                     _dev(n_visual, "n_visual", torch.int32), _dev(mass, "mass", torch.float32),
                                     _dev(entropy, "entropy", torch.float32), _stream()),
           "sd_attention_budget")
    return mass, entropy


SD_LAYER_PREFIX_EARLY = 1


def layer_workspace_bytes(B, R, Hq, Hkv, D, capacity):
    return int(lib().sd_verify_layer_workspace(B, R, Hq, Hkv, D, capacity))


def verify_layer(q, k_new, v_new, pos, sections, cache, interleaved=0, base=1e6, out=None, scale=0.0,
                 ws=None, early=False, block=False):
    """sd_verify_layer: M-RoPE of q / k_new (in place), append of k_new / v_new at
    len[b] (the prefix length on entry; len += R) and the verify attention; returns out.
    early=True sets SD_LAYER_PREFIX_EARLY (the previous kernel on the stream writes
    neither this layer's cache nor its len); block=True sets SD_LAYER_BLOCK_MASK."""
    B, R, Hq, D = q.shape
    Hkv = k_new.shape[2]
    if tuple(k_new.shape) != (B, R, Hkv, D) or k_new.shape != v_new.shape or tuple(pos.shape) != (B, R, 3):
        raise ValueError("shape mismatch")
    if cache.shape[0] != B or cache.shape[1] != Hkv or cache.shape[3] != D:
        raise ValueError("q and cache disagree")
    if out is None:
        out = torch.empty_like(q)
    if ws is None:
        # one workspace per layer cache: calls with early=True overlap the
        # previous layer's kernel, so layers must not share their tickets
        need = layer_workspace_bytes(B, R, Hq, Hkv, D, cache.shape[2])
        ws = getattr(cache, "_layer_ws", None)
        if ws is None or ws.numel() < need:
            ws = workspace(need, q.device)
            cache._layer_ws = ws
    sec = (ctypes.c_int32 * 3)(*[int(x) for x in sections])
    _check(lib().sd_verify_layer(_dev(q, "q", torch.bfloat16), _dev(k_new, "k_new", torch.bfloat16),
                                 _dev(v_new, "v_new", torch.bfloat16), _dev(pos, "pos", torch.int32), sec,
                                 int(interleaved), float(base), cache.struct, _dev(out, "out", torch.bfloat16),
                                 R, Hq, float(scale), _dev(ws, "ws"), ws.numel() * ws.element_size(),
                                 (SD_LAYER_PREFIX_EARLY if early else 0) | (SD_LAYER_BLOCK_MASK if block else 0),
                                 _stream()), "sd_verify_layer")
    return out


# -------------------------------------------------------------- acceptance

def greedy_workspace_bytes(B, K, V):
    return int(lib().sd_accept_greedy_workspace(B, K, V))


def sample_workspace_bytes(B, K, V):
    return int(lib().sd_accept_sample_workspace(B, K, V))


def accept_greedy(logits, draft, ws=None, n_emit=None, tokens=None, argmax=None):
    """Greedy acceptance over logits [B,K+1,V] (bf16 or fp32) and draft [B,K] int32.
    Returns (n_emit [B], tokens [B,K+1], argmax [B,K+1]) int32 device tensors."""
    B, R, V = logits.shape
    K = R - 1
    dt = {torch.bfloat16: SD_BF16, torch.float32: SD_F32}.get(logits.dtype)
    if dt is None:
        raise ValueError("logits must be bf16 or fp32")
    dev = logits.device
    if ws is None:
        ws = workspace(greedy_workspace_bytes(B, K, V), dev)
    n_emit = torch.empty(B, dtype=torch.int32, device=dev) if n_emit is None else n_emit
    tokens = torch.empty((B, R), dtype=torch.int32, device=dev) if tokens is None else tokens
    argmax = torch.empty((B, R), dtype=torch.int32, device=dev) if argmax is None else argmax
    draft_p = _dev(draft, "draft", torch.int32) if K > 0 else ctypes.c_void_p(0)
    _check(lib().sd_accept_greedy(_dev(logits, "logits"), dt, B, K, V, draft_p,
                                  _dev(n_emit, "n_emit", torch.int32), _dev(tokens, "tokens", torch.int32),
                                  _dev(argmax, "argmax", torch.int32), _dev(ws, "ws"), ws.numel() * ws.element_size(),
                                  _stream()), "sd_accept_greedy")
    return n_emit, tokens, argmax


def accept_greedy_noalloc(logits, draft, n_emit=None, tokens=None, argmax=None):
    """sd_accept_greedy_noalloc: greedy acceptance with the library's fixed
    scratch array instead of a caller workspace (no device allocation)."""
    B, R, V = logits.shape
    K = R - 1
    dt = {torch.bfloat16: SD_BF16, torch.float32: SD_F32}.get(logits.dtype)
    if dt is None:
        raise ValueError("logits must be bf16 or fp32")
    dev = logits.device
    n_emit = torch.empty(B, dtype=torch.int32, device=dev) if n_emit is None else n_emit
    tokens = torch.empty((B, R), dtype=torch.int32, device=dev) if tokens is None else tokens
    argmax = torch.empty((B, R), dtype=torch.int32, device=dev) if argmax is None else argmax
    draft_p = _dev(draft, "draft", torch.int32) if K > 0 else ctypes.c_void_p(0)
    _check(lib().sd_accept_greedy_noalloc(_dev(logits, "logits"), dt, B, K, V, draft_p,
                                          _dev(n_emit, "n_emit", torch.int32),
                                          _dev(tokens, "tokens", torch.int32),
                                          _dev(argmax, "argmax", torch.int32), _stream()),
           "sd_accept_greedy_noalloc")
    return n_emit, tokens, argmax


def accept_sample(z_target, z_draft, draft, u, temperature, ws=None, n_emit=None, tokens=None):
    """Rejection-sampling acceptance; returns (n_emit [B], tokens [B,K+1]) int32."""
    B, R, V = z_target.shape
    K = R - 1
    dev = z_target.device
    if ws is None:
        ws = workspace(sample_workspace_bytes(B, K, V), dev)
    n_emit = torch.empty(B, dtype=torch.int32, device=dev) if n_emit is None else n_emit
    tokens = torch.empty((B, R), dtype=torch.int32, device=dev) if tokens is None else tokens
    zd = _dev(z_draft, "z_draft", torch.float32) if K > 0 else ctypes.c_void_p(0)
    dr = _dev(draft, "draft", torch.int32) if K > 0 else ctypes.c_void_p(0)
    _check(lib().sd_accept_sample(_dev(z_target, "z_target", torch.float32), zd, B, K, V,
                                  float(temperature), dr, _dev(u, "u", torch.float32),
                                  _dev(n_emit, "n_emit", torch.int32), _dev(tokens, "tokens", torch.int32),
                                  _dev(ws, "ws"), ws.numel() * ws.element_size(), _stream()),
           "sd_accept_sample")
    return n_emit, tokens


def set_cluster_size(cluster_size=0):
    """Force the tcgen05 attention cluster size (1, 2, 4, 6, 8, 16); 0 = automatic."""
    _check(lib().sd_set_cluster_size(int(cluster_size)), "sd_set_cluster_size")


def verify_kernel(B, R, Hq, Hkv, D, capacity, layer=False):
    """Name of the kernel that serves this shape on the current device
    (sd_verify_kernel): "tcgen05", "mma.sync" or "three kernels"."""
    return lib().sd_verify_kernel(B, R, Hq, Hkv, D, capacity, 1 if layer else 0).decode()


def get_device_error():
    """Synchronise the current stream; return and clear the device error bits."""
    bits = ctypes.c_uint32(0)
    st = lib().sd_get_device_error(_stream(), ctypes.byref(bits))
    if st not in (0, 5, 6):
        raise SDError("sd_get_device_error", st)
    return int(bits.value)
