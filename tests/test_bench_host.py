"""The bench's host-side layout arithmetic (no GPU): the segment lengths behind the credited
flops agree with the oracle's segmentation, and the trajectory chunks cover the batch in order
within the per-chunk budget."""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from oracle import segments as oseg  # noqa: E402
from paper_2607_11185_gb300 import workloads  # noqa: E402
from tests.gpu_cases import random_steps  # noqa: E402


@pytest.mark.parametrize("seed", range(12))
@pytest.mark.parametrize("window,keep", [(1, 0), (2, 0), (3, 0), (5, 0), (1, 1), (3, 2), (5, 5), (5, 8)])
def test_layout_stats_match_oracle_segmentation(seed, window, keep):
    cu, img, txt = random_steps(seed)
    lens, traj = bench.layout_stats(cu, img, txt, window, keep)
    lay = oseg.build(cu, img, txt, window, keep)
    assert np.array_equal(lens, np.diff(lay["cu_seqlens"]).astype(np.int64))
    assert np.array_equal(traj, np.asarray(lay["seg_traj"], np.int64))


@pytest.mark.parametrize("name", ["tiny", "traj8_w3", "traj32_w3", "traj16x50_w8"])
def test_layout_stats_on_the_workloads(name):
    w = workloads.WORKLOADS[name]
    cu, img, txt = workloads.draw_steps(w)
    lens, traj = bench.layout_stats(cu, img, txt, w.window, w.keep)
    lay = oseg.build(cu, img, txt, w.window, w.keep, method="closed")
    assert np.array_equal(lens, np.diff(lay["cu_seqlens"]).astype(np.int64))
    total, fwd, bwd = bench.credited_flops(lens, w.hq, w.d)
    pairs = sum(int(L) * (int(L) + 1) // 2 for L in lens)
    assert total == 12.0 * w.d * w.hq * pairs and fwd + bwd == total and bwd == 2 * fwd


@pytest.mark.parametrize("name", ["traj8_w3", "traj32_w3", "traj16x50_w8"])
def test_chunks_cover_the_batch_within_budget(name):
    w = workloads.WORKLOADS[name]
    cu, img, txt = workloads.draw_steps(w)
    lens, traj = bench.layout_stats(cu, img, txt, w.window, w.keep)
    ntraj = len(cu) - 1
    chunks = bench.make_chunks(lens, traj, ntraj, w.hq, w.hkv, w.d)
    assert chunks[0][0] == 0 and chunks[-1][1] == ntraj
    assert all(a < b for a, b in chunks) and all(chunks[i][1] == chunks[i + 1][0] for i in range(len(chunks) - 1))
    per_tok = (2 * w.hq * w.d * 2 + 2 * w.hkv * w.d * 2) * 2 + w.hq * w.d * 4 + w.hq * 8 + 16
    tok = np.bincount(traj, weights=lens, minlength=ntraj)
    for a, b in chunks:
        if b - a > 1:                      # a single trajectory may exceed the budget on its own
            assert tok[a:b].sum() * per_tok <= bench.CHUNK_BYTES


def test_code_hash_ignores_comments_only():
    base = b"int a = 1;  // one\n/* block\n comment */ int b = a;\n"
    assert bench.code_hash(base) == bench.code_hash(b"int a = 1;  // uno\n\n/* other */ int b = a;   \n")
    assert bench.code_hash(base) != bench.code_hash(b"int a = 2;  // one\n/* block\n comment */ int b = a;\n")
    assert bench.code_hash(base) != bench.code_hash(b"int a = 1;\nint b = a + 1;\n")


def test_code_hash_keeps_string_literals():
    # a '//' or '/*' inside a string literal is code, not a comment
    a = b'const char* s = "a // b"; int x = 1;\n'
    b = b'const char* s = "a // c"; int x = 1;\n'
    assert bench.code_hash(a) != bench.code_hash(b)
    assert bench.strip_comments(b'f("/* x */"); /* y */ g();') == b'f("/* x */");  g();'
