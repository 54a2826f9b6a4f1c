"""C ABI checks that need no GPU: libsd.so builds for sm_103a, loads, exports
every function include/sd.h declares, and rejects bad host arguments before
launching anything."""
import ctypes
import subprocess

import pytest

from paper_2606_31160_gb300 import build, sd


@pytest.fixture(scope="module")
def lib():
    build.build()
    return sd.lib()


def test_every_header_symbol_is_exported(lib):
    names = sd.header_symbols()
    assert len(names) >= 13
    for name in names:
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", sd.LIB_PATH], capture_output=True, text=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    assert set(names) <= exported
    # nothing else leaks out under the sd_ prefix
    assert {n for n in exported if n.startswith("sd_")} == set(names)


def test_built_for_sm103a_only():
    out = subprocess.run(["cuobjdump", "--list-elf", sd.LIB_PATH], capture_output=True, text=True)
    if out.returncode != 0:
        pytest.skip("cuobjdump unavailable")
    assert "sm_103a" in out.stdout


def test_status_strings(lib):
    assert sd.status_str(0) == "SD_OK"
    assert sd.status_str(1) == "SD_ERR_INVALID_ARG"
    assert sd.status_str(3) == "SD_ERR_WORKSPACE"
    assert sd.status_str(6) == "SD_ERR_TIMEOUT"
    assert sd.status_str(99) == "SD_ERR_UNKNOWN"
    assert "sm_103a" in sd.version()


def test_workspace_queries_are_host_arithmetic(lib):
    g = sd.greedy_workspace_bytes(1, 7, 151936)
    assert g >= 8 * 38 * 8
    assert sd.greedy_workspace_bytes(32, 16, 151936) > g
    assert sd.greedy_workspace_bytes(0, 7, 10) == 0
    s = sd.sample_workspace_bytes(8, 7, 151936)
    assert s >= 8 * 15 * 38 * 8
    assert sd.sample_workspace_bytes(8, 7, 0) == 0


def test_bad_arguments_return_status_before_launch(lib):
    null = ctypes.c_void_p(0)
    # NULL cache / unsupported head dim / bad GQA ratio
    assert lib.sd_verify_attention(null, None, null, 8, 32, 0.0, null, 0, null) == 1
    cache = sd.KVCacheStruct(16, 16, 16, 1, 8, 64, 96)
    assert lib.sd_verify_attention(ctypes.c_void_p(16), ctypes.byref(cache), ctypes.c_void_p(16), 8, 32, 0.0, null, 0, null) == 2
    cache = sd.KVCacheStruct(16, 16, 16, 1, 3, 64, 128)
    assert lib.sd_verify_attention(ctypes.c_void_p(16), ctypes.byref(cache), ctypes.c_void_p(16), 8, 32, 0.0, null, 0, null) == 1
    # G * R beyond the packed-tile limit
    cache = sd.KVCacheStruct(16, 16, 16, 1, 1, 64, 128)
    assert lib.sd_verify_attention(ctypes.c_void_p(16), ctypes.byref(cache), ctypes.c_void_p(16), 17, 8, 0.0, null, 0, null) == 2
    # misaligned pointer
    cache = sd.KVCacheStruct(18, 16, 16, 1, 8, 64, 128)
    assert lib.sd_verify_attention(ctypes.c_void_p(16), ctypes.byref(cache), ctypes.c_void_p(16), 8, 32, 0.0, null, 0, null) == 1
    # rope: unsupported head dim, bad sections
    sec = (ctypes.c_int32 * 3)(16, 24, 24)
    assert lib.sd_rope_apply(ctypes.c_void_p(16), ctypes.c_void_p(16), 1, 8, 32, 8, 96, ctypes.c_void_p(16), sec, 0, 1e6, null) == 2
    bad = (ctypes.c_int32 * 3)(16, 24, 23)
    assert lib.sd_rope_apply(ctypes.c_void_p(16), ctypes.c_void_p(16), 1, 8, 32, 8, 128, ctypes.c_void_p(16), bad, 0, 1e6, null) == 1
    assert lib.sd_rope_apply(ctypes.c_void_p(16), ctypes.c_void_p(16), 1, 8, 32, 8, 128, ctypes.c_void_p(16), sec, 2, 1e6, null) == 1
    # kv: NULL cache, rollback with count not a multiple of B
    assert lib.sd_kv_append(None, null, null, 8, null) == 1
    assert lib.sd_kv_rollback(ctypes.c_void_p(16), 5, 2, ctypes.c_void_p(16), 8, null) == 1
    # acceptance: short workspace, bad dtype, bad temperature
    assert lib.sd_accept_greedy(ctypes.c_void_p(16), 0, 1, 7, 151936, ctypes.c_void_p(16), ctypes.c_void_p(16),
                                ctypes.c_void_p(16), null, ctypes.c_void_p(16), 8, null) == 3
    assert lib.sd_accept_greedy(ctypes.c_void_p(16), 7, 1, 7, 100, ctypes.c_void_p(16), ctypes.c_void_p(16),
                                ctypes.c_void_p(16), null, ctypes.c_void_p(16), 1 << 20, null) == 1
    assert lib.sd_accept_sample(ctypes.c_void_p(16), ctypes.c_void_p(16), 1, 7, 100, 0.0, ctypes.c_void_p(16),
                                ctypes.c_void_p(16), ctypes.c_void_p(16), ctypes.c_void_p(16),
                                ctypes.c_void_p(16), 1 << 20, null) == 1
    # empty batches are a no-op success
    cache = sd.KVCacheStruct(0, 0, 0, 0, 8, 64, 128)
    assert lib.sd_verify_attention(null, ctypes.byref(cache), null, 8, 32, 0.0, null, 0, null) == 0


def test_cluster_size_override_is_host_only(lib):
    # accepted sizes and 0 (automatic); no device work, so it runs without a GPU
    for cs in (1, 2, 4, 6, 8, 16, 0):
        assert lib.sd_set_cluster_size(cs) == 0
    for cs in (-1, 3, 5, 7, 12, 32):
        assert lib.sd_set_cluster_size(cs) == 1
    assert lib.sd_set_cluster_size(0) == 0


def test_unknown_mask_flags_are_rejected_before_launch(lib):
    null = ctypes.c_void_p(0)
    cache = sd.KVCacheStruct(16, 16, 16, 1, 8, 64, 128)
    assert lib.sd_verify_attention_ex(ctypes.c_void_p(16), ctypes.byref(cache), ctypes.c_void_p(16), 8, 32, 0.0,
                                      4, null, 0, null) == 1
    assert lib.sd_verify_layer(ctypes.c_void_p(16), ctypes.c_void_p(16), ctypes.c_void_p(16), ctypes.c_void_p(16),
                               (ctypes.c_int32 * 3)(16, 24, 24), 0, 1e6, ctypes.byref(cache), ctypes.c_void_p(16),
                               8, 32, 0.0, null, 0, 4, null) == 1


def test_kernel_query_rejects_unsupported_shapes(lib):
    # sd_verify_kernel is host arithmetic: shapes no entry point takes are
    # "unsupported" without touching a device
    from paper_2606_31160_gb300 import sd
    assert sd.verify_kernel(1, 8, 30, 8, 128, 4104) == "unsupported"     # Hq % Hkv
    assert sd.verify_kernel(1, 8, 32, 8, 96, 4104) == "unsupported"      # head_dim
    assert sd.verify_kernel(1, 40, 32, 8, 128, 4104) == "unsupported"    # G * R > 128
    assert sd.verify_kernel(0, 8, 32, 8, 128, 4104, True) == "unsupported"


def _layer(lib, cache, q=16, out=16, R=8, Hq=32, interleaved=0, base=1e6, scale=0.0, ws=16, ws_bytes=1 << 30,
           flags=0, sections=(16, 24, 24)):
    sec = (ctypes.c_int32 * 3)(*sections)
    return lib.sd_verify_layer(ctypes.c_void_p(q), ctypes.c_void_p(16), ctypes.c_void_p(16), ctypes.c_void_p(16),
                               sec, interleaved, base, cache, ctypes.c_void_p(out), R, Hq, scale,
                               ctypes.c_void_p(ws), ws_bytes, flags, ctypes.c_void_p(0))


def test_layer_host_checks_return_before_launch(lib):
    # sd_verify_layer validates everything it can on the host, in this order:
    # shape, head dim, flags, pointers and alignment, scale and base, the
    # workspace, then the rotation sections; nothing reaches a device
    ok = sd.KVCacheStruct(16, 16, 16, 1, 8, 4200, 128)
    assert _layer(lib, None) == 1                                               # no cache
    assert _layer(lib, ctypes.byref(ok), R=0) == 1                              # no new rows
    assert _layer(lib, ctypes.byref(ok), Hq=30) == 1                            # Hq % Hkv
    assert _layer(lib, ctypes.byref(sd.KVCacheStruct(16, 16, 16, 1, 8, 4200, 96))) == 2   # head dim
    assert _layer(lib, ctypes.byref(ok), interleaved=2) == 1
    assert _layer(lib, ctypes.byref(ok), flags=8) == 1                          # unknown flag bit
    assert _layer(lib, ctypes.byref(sd.KVCacheStruct(0, 0, 0, 0, 8, 4200, 128)), q=0, out=0) == 0  # no scenes
    assert _layer(lib, ctypes.byref(ok), q=0) == 1                              # NULL q
    assert _layer(lib, ctypes.byref(ok), out=24) == 1                           # misaligned out
    assert _layer(lib, ctypes.byref(sd.KVCacheStruct(40, 16, 16, 1, 8, 4200, 128))) == 1  # misaligned cache
    assert _layer(lib, ctypes.byref(ok), scale=-1.0) == 1
    assert _layer(lib, ctypes.byref(ok), scale=float("nan")) == 1
    assert _layer(lib, ctypes.byref(ok), base=1.0) == 1
    assert _layer(lib, ctypes.byref(ok), base=float("inf")) == 1
    need = lib.sd_verify_layer_workspace(1, 8, 32, 8, 128, 4200)
    assert need >= 256                                                          # the tickets at least
    assert _layer(lib, ctypes.byref(ok), ws=0) == 3
    assert _layer(lib, ctypes.byref(ok), ws_bytes=need - 1) == 3
    assert _layer(lib, ctypes.byref(ok), ws=24) == 3                            # misaligned workspace
    assert _layer(lib, ctypes.byref(ok), sections=(16, 24, 23)) == 1            # sections must sum to D / 2
    assert lib.sd_verify_layer_workspace(0, 8, 32, 8, 128, 4200) == 0


def test_budget_host_checks_return_before_launch(lib):
    def budget(cache, R=8, Hq=32, scale=0.0, q=16, mass=16):
        return lib.sd_attention_budget(ctypes.c_void_p(q), cache, R, Hq, scale, ctypes.c_void_p(16),
                                       ctypes.c_void_p(mass), ctypes.c_void_p(16), ctypes.c_void_p(0))
    ok = sd.KVCacheStruct(16, 16, 16, 1, 8, 4200, 128)
    assert budget(None) == 1
    assert budget(ctypes.byref(ok), R=0) == 1
    assert budget(ctypes.byref(ok), Hq=12) == 1                                 # Hq % Hkv
    assert budget(ctypes.byref(sd.KVCacheStruct(16, 16, 16, 1, 8, 4200, 80))) == 2
    assert budget(ctypes.byref(sd.KVCacheStruct(16, 16, 16, 70000, 8, 4200, 128))) == 2   # grid z limit
    assert budget(ctypes.byref(sd.KVCacheStruct(0, 0, 0, 0, 8, 4200, 128)), q=0, mass=0) == 0
    assert budget(ctypes.byref(ok), mass=0) == 1
    assert budget(ctypes.byref(sd.KVCacheStruct(8, 16, 16, 1, 8, 4200, 128))) == 1        # misaligned keys
    assert budget(ctypes.byref(ok), scale=-0.5) == 1
    assert budget(ctypes.byref(ok), scale=float("inf")) == 1
