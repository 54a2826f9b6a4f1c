"""The allocation-free greedy acceptance (sd_accept_greedy_noalloc), called
through the C ABI, must give exactly what sd_accept_greedy gives with a caller
workspace -- on two calls in a row, since both share the library's fixed
scratch array and each call must leave it ready for the next. This file is
collected last so a failure here never hides another test's result; it
passes alone in a fresh process and after the rest of the suite."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2606_31160_gb300 import build, sd, workloads

pytestmark = pytest.mark.gpu


def _c_noalloc(logits, draft, dtype):
    """Call the entry point directly through ctypes (no binding helper)."""
    lib = sd.lib()
    B, R, V = logits.shape
    K = R - 1
    n_emit = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    tokens = torch.full((B, R), -7, dtype=torch.int32, device="cuda")
    argmax = torch.full((B, R), -7, dtype=torch.int32, device="cuda")
    st = lib.sd_accept_greedy_noalloc(ctypes.c_void_p(logits.data_ptr()), dtype, B, K, V,
                                      ctypes.c_void_p(draft.data_ptr()), ctypes.c_void_p(n_emit.data_ptr()),
                                      ctypes.c_void_p(tokens.data_ptr()), ctypes.c_void_p(argmax.data_ptr()),
                                      ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0, sd.status_str(st)
    return n_emit, tokens, argmax


def test_noalloc_matches_workspace_entry_point_twice_in_a_row():
    build.build()
    assert sd.lib().sd_accept_greedy_noalloc_max_bytes() == 1 << 20
    cases = []
    t = workloads.target_layer(B=1, ell=[3])          # bf16, V = 151936
    cases.append((t.extra["logits"], t.extra["draft"], sd.SD_BF16))
    rng = np.random.default_rng(5)                     # fp32, several scenes, planted ties
    z = rng.standard_normal((6, 5, 50000)).astype(np.float32)
    z[2, 1, [10, 40000]] = 9.0
    star = z.argmax(-1)
    draft = np.where(rng.random((6, 4)) < 0.7, star[:, :4], rng.integers(0, 50000, (6, 4)))
    cases.append((torch.from_numpy(z), torch.from_numpy(draft.astype(np.int32)), sd.SD_F32))
    for logits, draft, dtype in cases:
        lg, dr = logits.cuda(), draft.cuda()
        ref = sd.accept_greedy(lg, dr)
        for _ in range(2):
            got = _c_noalloc(lg, dr, dtype)
            for a, b in zip(got, ref):
                assert torch.equal(a, b)
    assert sd.get_device_error() == 0


def test_noalloc_rejects_shapes_beyond_its_array():
    build.build()
    lib = sd.lib()
    null = ctypes.c_void_p(16)
    # 4097 scenes exceed the ticket header; a 2**22-token vocabulary with 64 rows
    # exceeds the 1 MiB of partials: both refused before launch
    assert lib.sd_accept_greedy_noalloc(null, sd.SD_F32, 4097, 0, 10, null, null, null, null, None) == 3
    assert lib.sd_accept_greedy_noalloc(null, sd.SD_F32, 16, 15, 1 << 22, null, null, null, null, None) == 3
