"""The C ABI library loads and exports every entry point include/vcs.h declares (CPU only)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LIB = os.path.join(ROOT, "paper_2607_11185_gb300", "libvcs.so")


def declared_functions():
    text = open(os.path.join(ROOT, "include", "vcs.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(vcs_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(LIB):
        from paper_2607_11185_gb300 import build
        build.build()
    return ctypes.CDLL(LIB)


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings_without_gpu(lib):
    lib.vcs_status_string.restype = ctypes.c_char_p
    for code in range(9):
        s = lib.vcs_status_string(code).decode()
        assert s.startswith("VCS_")
    assert lib.vcs_status_string(99).decode() == "VCS_ERR_UNKNOWN"


def test_host_side_argument_errors_without_gpu(lib):
    # rejected before any CUDA call: null pointers, bad window, unsupported head_dim
    f = lib.vcs_plan_segments
    f.restype = ctypes.c_int32
    f.argtypes = [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32,
                  ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
    assert f(None, 1, 4, None, None, 2, 0, None, None, 0, None) == 1          # INVALID_ARG
    assert f(8, 1, 4, 8, 8, 0, 0, 8, 256, 1 << 20, None) == 1                  # window 0
    assert f(256, 1, 4, 256, 256, 2, 0, 256, 256, 1, None) == 8               # workspace too small
    g = lib.vcs_attn_fwd
    g.restype = ctypes.c_int32
    g.argtypes = [ctypes.c_void_p] * 4 + [ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                          ctypes.c_int32, ctypes.c_int32, ctypes.c_float, ctypes.c_void_p,
                                          ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
    assert g(256, 256, 256, 256, 1, 10, 10, 2, 1, 96, 0.0, 256, 256, 256, 4096, None) == 2   # d=96 unsupported
    assert g(256, 256, 256, 256, 1, 10, 10, 3, 2, 64, 0.0, 256, 256, 256, 4096, None) == 2   # hq % hkv
    assert g(None, 256, 256, 256, 1, 10, 10, 2, 1, 64, 0.0, 256, 256, 256, 4096, None) == 1
    assert g(264, 256, 256, 256, 1, 10, 10, 2, 1, 64, 0.0, 256, 256, 256, 4096, None) == 1   # misaligned q
    lib.vcs_attn_fwd_workspace_size.restype = ctypes.c_size_t
    lib.vcs_attn_fwd_workspace_size.argtypes = [ctypes.c_int32, ctypes.c_int64] + [ctypes.c_int32] * 4
    assert g(256, 256, 256, 256, 1, 10, 10, 2, 1, 64, 0.0, 256, 256, 256, 0, None) == 8      # no workspace


def test_gathered_and_reuse_host_checks_without_gpu(lib):
    # size queries are host arithmetic; argument errors return before any CUDA call
    ws = lib.vcs_attn_bwd_workspace_size
    ws.restype = ctypes.c_size_t
    ws.argtypes = [ctypes.c_int32, ctypes.c_int64] + [ctypes.c_int32] * 4
    gws = lib.vcs_attn_bwd_gathered_workspace_size
    gws.restype = ctypes.c_size_t
    gws.argtypes = [ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, ctypes.c_int64] + [ctypes.c_int32] * 3
    r256 = lambda x: (x + 255) // 256 * 256  # noqa: E731
    for nt, tt, hq, hkv, d in ((1000, 700, 28, 4, 128), (17, 5, 2, 1, 64)):
        assert gws(3, nt, 500, tt, hq, hkv, d) == ws(3, nt, 500, hq, hkv, d) + r256(tt * hq * d * 4) + 2 * r256(
            tt * hkv * d * 4)
        assert gws(3, nt, 500, 0, hq, hkv, d) == ws(3, nt, 500, hq, hkv, d)
    f = lib.vcs_attn_fwd_gathered
    f.restype = ctypes.c_int32
    f.argtypes = [ctypes.c_void_p] * 3 + [ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32,
                                          ctypes.c_int64] + [ctypes.c_int32] * 4 + [ctypes.c_float] + \
        [ctypes.c_void_p] * 3 + [ctypes.c_size_t, ctypes.c_void_p]
    A = 256
    assert f(A, A, A, 100, None, A, 1, 10, 10, 2, 1, 64, 0.0, A, A, A, 4096, None) == 1        # no gather map
    assert f(A, A, A, 0, A, A, 1, 10, 10, 2, 1, 64, 0.0, A, A, A, 4096, None) == 1             # no trajectory rows
    assert f(A, A, A, 1 << 31, A, A, 1, 10, 10, 2, 1, 64, 0.0, A, A, A, 4096, None) == 4       # overflow
    assert f(A, A, A, 100, A, A, 1, 10, 10, 2, 1, 96, 0.0, A, A, A, 4096, None) == 2           # d = 96
    assert f(A, A, A, 100, A, A, 1, 10, 10, 2, 1, 64, 0.0, A, A, A, 0, None) == 8              # workspace
    sp = lib.vcs_shared_prefix
    sp.restype = ctypes.c_int32
    sp.argtypes = [ctypes.c_void_p] * 3 + [ctypes.c_int32, ctypes.c_int64] + [ctypes.c_void_p] * 3
    assert sp(A, A, A, -1, 10, A, None, None) == 1
    assert sp(None, A, A, 2, 10, A, None, None) == 1
    assert sp(A, A, A, 2, 1 << 31, A, None, None) == 4
    fr = lib.vcs_attn_fwd_reuse
    fr.restype = ctypes.c_int32
    fr.argtypes = [ctypes.c_void_p] * 5 + [ctypes.c_int32, ctypes.c_int64] + [ctypes.c_int32] * 4 + \
        [ctypes.c_float] + [ctypes.c_void_p] * 3 + [ctypes.c_size_t, ctypes.c_void_p]
    assert fr(A, A, A, A, None, 1, 10, 10, 2, 1, 64, 0.0, A, A, A, 4096, None) == 1           # no shared map
    assert fr(A, A, A, A, A, 1, 10, 10, 2, 1, 64, 0.0, A, A, A, 0, None) == 8                 # workspace


def test_selftest_bounded_wait_argument_errors_without_gpu(lib):
    # rejected before any launch: null or misaligned status word, limit outside 1 .. 4e9 cycles
    f = lib.vcs_selftest_bounded_wait
    f.restype = ctypes.c_int32
    f.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]
    assert f(None, 1000, None) == 1
    assert f(258, 1000, None) == 1
    assert f(256, 0, None) == 1
    assert f(256, -5, None) == 1
    assert f(256, 4_000_000_001, None) == 1


def test_forward_workspace_holds_the_unit_list(lib):
    # header, per-segment unit offsets, then 16 bytes per work unit: at most
    # hq * (num_tokens / 256 + num_segments + 1) units, which bounds hq * sum_s ceil(L_s / 256)
    import numpy as np
    f = lib.vcs_attn_fwd_workspace_size
    f.restype = ctypes.c_size_t
    f.argtypes = [ctypes.c_int32, ctypes.c_int64] + [ctypes.c_int32] * 4
    r256 = lambda x: (x + 255) // 256 * 256  # noqa: E731
    for s, t, hq in ((1, 10, 2), (56, 1_972_928, 40), (1040, 7_727_164, 40), (5, 0, 8)):
        assert f(s, t, 4096, hq, 1, 128) == 256 + r256((s + 1) * 4) + r256(hq * (t // 256 + s + 1) * 16)
    rng = np.random.default_rng(0)
    for _ in range(500):
        lens = rng.integers(0, 5000, size=int(rng.integers(1, 60)))
        t, s = int(lens.sum()), len(lens)
        assert int(((lens + 255) // 256).sum()) <= t // 256 + s + 1
