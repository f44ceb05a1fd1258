"""Attention forward and backward on every comparison layout of the 32-trajectory draw, and on
the paper-exact K = delta = 8 layout of the long-horizon draw, against the fp64 oracle.

The same trajectories are laid out the ways the comparison runs them through the same
kernels: step-wise (one item per step, the history as text; the same as a window of one
screenshot), a window of five screenshots, and the paper's own retained-plus-new settings
K = delta = 1, K = delta = 5 and K = 8, delta = 5 (Sec. 3.4, Algorithm 1; App. C.2).  Each
layout runs in exactly the chunks the benchmark launches it in, and in every chunk O and
lse are checked on sampled rows (ends, tile edges, random rows of the shortest, longest,
first, last and random segments), dQ on sampled rows, dK and dV on the last keys of
sampled segments, and the per-segment gradient sums.

Tolerances as in the other attention tests: O max-abs 2e-2, lse max-abs 2e-3, gradients
relative L2 1e-2.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import segments as oseg
from paper_2607_11185_gb300 import workloads
from tests.gpu_cases import bench_chunks
from tests.test_gpu_attn_bwd import check_sampled_grads
from tests.test_gpu_attn_fwd import check_sampled

pytestmark = pytest.mark.gpu

LAYOUTS = ["stepwise", "w5", "paper_k1", "paper_k5", "paper_k8_d5"]
CASES = [("traj32_w3", lay) for lay in LAYOUTS] + [
    # the paper-exact reading of the long-horizon workload's window (K = delta = 8): the longest
    # segments of any layout here (67,800 tokens), 40/8 heads, 5% of key rows scaled by 8
    ("traj16x50_w8", "paper_k8"),
]


@pytest.mark.parametrize("name,layout", CASES)
def test_comparison_layout_every_chunk_sampled(name, layout):
    from paper_2607_11185_gb300 import vcs
    w = workloads.WORKLOADS[name]
    window, keep = workloads.COMPARISON_LAYOUTS[layout]
    cu_s, img, txt = workloads.draw_steps(w)
    lay = oseg.build(cu_s, img, txt, window, keep)
    qt, kt, vt = workloads.draw_traj_qkv(w, workloads.trajectory_tokens(img, txt), device="cuda")
    cu = lay["cu_seqlens"]
    chunks = bench_chunks(w, lay, len(cu_s) - 1)
    for i, (s0, s1) in enumerate(chunks):
        t0, t1 = int(cu[s0]), int(cu[s1])
        g = torch.from_numpy(lay["tok_gather"][t0:t1].astype(np.int64)).cuda()
        q, k, v = qt[g], kt[g], vt[g]
        del g
        ccu = (cu[s0:s1 + 1] - cu[s0]).astype(np.int32)
        do = workloads.draw_dout(dataclasses.replace(w, seed=w.seed + 700 + i), t1 - t0, device="cuda")
        dcu = torch.from_numpy(ccu).cuda()
        mx = int(np.diff(ccu).max())
        o, lse = vcs.attn_fwd(q, k, v, dcu, mx)
        dq, dk, dv = vcs.attn_bwd(q, k, v, o, lse, do, dcu, mx)
        torch.cuda.synchronize()
        rng = np.random.default_rng(1000 + 10 * CASES.index((name, layout)) + i)
        check_sampled(q, k, v, ccu, o, lse, rng, n_seg=2)
        check_sampled_grads(q, k, v, do, ccu, dq, dk, dv, rng, n_seg=2, n_rows=3, tail=16 if w.hq < 40 else 8)
        del q, k, v, do, o, lse, dq, dk, dv
        torch.cuda.empty_cache()
    assert len(chunks) >= 1
