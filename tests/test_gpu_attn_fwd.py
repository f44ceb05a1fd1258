"""GPU attention forward vs the fp64 oracle.

Tolerances: O max-abs 2e-2 (bf16 inputs, fp32 accumulation, bf16 output);
lse max-abs 2e-3 (fp32 score accumulation over d <= 128 bf16 products and
the hardware exp2/log2, whose relative error is ~1e-6 on values |lse| < 100).
"""
import math

import numpy as np
import pytest
import torch

from oracle import attention as oatt
from oracle import segments as oseg
from paper_2607_11185_gb300 import workloads
from tests.gpu_cases import bench_chunks, cu_from_lengths, sample_rows

pytestmark = pytest.mark.gpu

O_TOL = 2e-2
LSE_TOL = 2e-3


def run_fwd(q, k, v, cu):
    from paper_2607_11185_gb300 import vcs
    dcu = torch.from_numpy(np.asarray(cu, np.int32)).cuda()
    lens = np.diff(cu)
    return vcs.attn_fwd(q, k, v, dcu, int(lens.max()) if len(lens) else 0)


def compare_full(q, k, v, cu, o, lse):
    ro, rl = oatt.attn_fwd(q.cpu(), k.cpu(), v.cpu(), cu)
    err_o = np.abs(o.float().cpu().numpy() - ro).max()
    err_l = np.abs(lse.cpu().numpy() - rl).max()
    assert err_o <= O_TOL, err_o
    assert err_l <= LSE_TOL, err_l


CASES = [
    # (lengths, hq, hkv, d)
    ([1, 127, 128, 129, 255, 256, 257, 300], 2, 1, 64),
    ([1, 127, 128, 129, 255, 256, 257, 300], 2, 1, 128),
    ([600, 1, 383, 513], 7, 1, 128),           # GQA 7:1, odd number of tiles
    ([640, 129], 4, 4, 64),                    # MHA
    ([1000], 6, 2, 128),
]


@pytest.mark.parametrize("lengths,hq,hkv,d", CASES)
def test_small_shapes_full_oracle(lengths, hq, hkv, d):
    cu = cu_from_lengths(lengths)
    q, k, v, _ = workloads.draw_dense(11 + d + hq, int(cu[-1]), hq, hkv, d, device="cuda")
    o, lse = run_fwd(q, k, v, cu)
    compare_full(q, k, v, cu, o, lse)


def test_tiny_workload_full_oracle():
    w = workloads.WORKLOADS["tiny"]
    cu_s, img, txt = workloads.draw_steps(w)
    lay = oseg.build(cu_s, img, txt, w.window, w.keep)
    qt, kt, vt = workloads.draw_traj_qkv(w, workloads.trajectory_tokens(img, txt), device="cuda")
    g = torch.from_numpy(lay["tok_gather"].astype(np.int64)).cuda()
    q, k, v = qt[g], kt[g], vt[g]
    o, lse = run_fwd(q, k, v, lay["cu_seqlens"])
    compare_full(q, k, v, lay["cu_seqlens"], o, lse)


def test_single_token_segments_copy_v():
    cu = cu_from_lengths([1] * 40)
    q, k, v, _ = workloads.draw_dense(5, 40, 4, 2, 128, device="cuda")
    o, lse = run_fwd(q, k, v, cu)
    ref_v = v.repeat_interleave(2, dim=1)
    assert torch.equal(o, ref_v)     # softmax over one key is exactly 1
    s = (q.float() * k.float().repeat_interleave(2, 1)).sum(-1).T / math.sqrt(128)
    assert (lse - s).abs().max().item() < LSE_TOL


def test_large_logits_stress_rescaling():
    # scores of magnitude ~40 force mid-loop maximum raises in the online softmax
    cu = cu_from_lengths([700, 333])
    q, k, v, _ = workloads.draw_dense(21, int(cu[-1]), 2, 1, 128, device="cuda", scale=6.0)
    o, lse = run_fwd(q, k, v, cu)
    compare_full(q, k, v, cu, o, lse)


def check_sampled(q, k, v, cu, o, lse, rng, n_seg=6, heads=None):
    nseg = len(cu) - 1
    lens = np.diff(cu)
    segs = sorted({int(np.argmin(lens)), int(np.argmax(lens)), 0, nseg - 1,
                   *[int(x) for x in rng.integers(0, nseg, size=n_seg)]})
    hq = q.shape[1]
    heads = heads if heads is not None else sorted({0, hq - 1, int(rng.integers(0, hq))})
    worst = 0.0
    for s in segs:
        b, e = int(cu[s]), int(cu[s + 1])
        if e == b:
            continue
        rows = sample_rows(e - b, rng)
        ro, rl = oatt.rows_fwd(q, k, v, (b, e), heads, rows)
        idx = torch.tensor([b + r for r in rows], device=o.device)
        got_o = o[idx][:, heads].float().cpu().numpy()
        got_l = lse[heads][:, idx].cpu().numpy()
        eo = np.abs(got_o - ro).max()
        el = np.abs(got_l - rl).max()
        worst = max(worst, eo)
        assert eo <= O_TOL, (s, eo)
        assert el <= LSE_TOL, (s, el)
    return worst


def _chunks_sampled(name, seed, **kw):
    """Every chunk of the workload in the benchmark's launch configuration, on sampled rows."""
    w = workloads.WORKLOADS[name]
    cu_s, img, txt = workloads.draw_steps(w)
    lay = oseg.build(cu_s, img, txt, w.window, w.keep)
    qt, kt, vt = workloads.draw_traj_qkv(w, workloads.trajectory_tokens(img, txt), device="cuda")
    cu = lay["cu_seqlens"]
    chunks = bench_chunks(w, lay, len(cu_s) - 1)
    for i, (s0, s1) in enumerate(chunks):
        t0, t1 = int(cu[s0]), int(cu[s1])
        g = torch.from_numpy(lay["tok_gather"][t0:t1].astype(np.int64)).cuda()
        q, k, v = qt[g], kt[g], vt[g]
        ccu = cu[s0:s1 + 1] - cu[s0]
        o, lse = run_fwd(q, k, v, ccu)
        check_sampled(q, k, v, ccu, o, lse, np.random.default_rng(seed + i), **kw)
        del q, k, v, o, lse
    return chunks


@pytest.mark.parametrize("name", ["traj8_w3", "traj32_w3"])
def test_workload_full_size_sampled_rows(name):
    chunks = _chunks_sampled(name, 3)
    assert len(chunks) == (1 if name == "traj8_w3" else 2)


def test_long_horizon_outliers_sampled_rows():
    # 16 x 50 steps, W=8, 40/8 heads, 5% of K rows scaled by 8; both 8-trajectory chunks
    chunks = _chunks_sampled("traj16x50_w8", 5, n_seg=3, heads=[0, 17, 39])
    assert len(chunks) == 2


def test_inconsistent_cu_seqlens_reported():
    from paper_2607_11185_gb300 import vcs
    q, k, v, _ = workloads.draw_dense(1, 64, 2, 1, 64, device="cuda")
    bad = torch.tensor([0, 40, 30, 64], dtype=torch.int32, device="cuda")
    with pytest.raises(vcs.VcsError) as e:
        vcs.attn_fwd(q, k, v, bad, 64)
    assert e.value.status == 6


@pytest.mark.parametrize("bounds,expect_units", [
    # overlapping segments that fit the unit list: both run (over the same rows), the bad one
    # in between is reported
    ([0, 512, 0, 512], 2 * (2 + 2)),
    # five full-length segments over the same 16,384 rows: 640 units against room for 148, so
    # none runs (nothing is written past the list) and the call reports the check
    ([0, 16384, 0, 16384, 0, 16384, 0, 16384, 0, 16384], 0),
])
def test_overlapping_segments_reported_and_bounded(bounds, expect_units):
    from paper_2607_11185_gb300 import vcs
    nt = bounds[-1]
    hq, hkv, d = 2, 1, 64
    q, k, v, _ = workloads.draw_dense(2, nt, hq, hkv, d, device="cuda")
    cu = torch.tensor(bounds, dtype=torch.int32, device="cuda")
    ns = len(bounds) - 1
    nb = vcs.vcs_attn_fwd_workspace_size(ns, nt, nt, hq, hkv, d)
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    o = torch.zeros_like(q)
    lse = torch.zeros((hq, nt), dtype=torch.float32, device="cuda")
    assert vcs.vcs_attn_fwd(q, k, v, cu, ns, nt, nt, hq, hkv, d, 0.0, o, lse, ws, nb) == 0
    torch.cuda.synchronize()
    hdr = ws[:256].view(torch.int32).cpu().numpy()
    assert hdr[0] == 6
    assert hdr[128 // 4] == expect_units


def _units_of(cu, hq):
    """Work units the forward lists: hq per 256-row pair of query tiles of each segment."""
    lens = np.diff(np.asarray(cu, np.int64))
    return int(hq * ((lens + 255) // 256).sum())


def test_work_unit_list_with_empty_segments():
    # empty segments at the start, in the middle and at the end, and segments that end a
    # pair of query tiles early or exactly: the listed unit count (workspace header, int32 at
    # byte 128) is exact, and every row matches the oracle
    from paper_2607_11185_gb300 import vcs
    lengths = [0, 0, 300, 0, 256, 1, 0, 513, 257, 0]
    hq, hkv, d = 5, 1, 128
    cu = cu_from_lengths(lengths)
    nt = int(cu[-1])
    q, k, v, _ = workloads.draw_dense(71, nt, hq, hkv, d, device="cuda")
    dcu = torch.from_numpy(np.asarray(cu, np.int32)).cuda()
    ns = len(lengths)
    nb = vcs.vcs_attn_fwd_workspace_size(ns, nt, max(lengths), hq, hkv, d)
    assert nb >= 256 + 4 * (ns + 1) + 16 * _units_of(cu, hq)
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    o = torch.empty_like(q)
    lse = torch.empty((hq, nt), dtype=torch.float32, device="cuda")
    assert vcs.vcs_attn_fwd(q, k, v, dcu, ns, nt, max(lengths), hq, hkv, d, 0.0, o, lse, ws, nb) == 0
    torch.cuda.synchronize()
    hdr = ws[:256].view(torch.int32).cpu().numpy()
    assert hdr[0] == 0
    assert hdr[128 // 4] == _units_of(cu, hq)
    compare_full(q, k, v, cu, o, lse)


@pytest.mark.parametrize("window", [1, 3])
def test_work_unit_count_on_builder_layouts(window):
    # the 8-trajectory draw laid out step-wise (W = 1: many short segments, the case the list
    # is for) and with W = 3: the listed unit count is the closed form over the oracle's
    # segment lengths, and sampled rows match the oracle
    from paper_2607_11185_gb300 import vcs
    w = workloads.WORKLOADS["traj8_w3"]
    cu_s, img, txt = workloads.draw_steps(w)
    lay = oseg.build(cu_s, img, txt, window, 0)
    cu = np.asarray(lay["cu_seqlens"], np.int64)
    nt, ns = int(cu[-1]), len(cu) - 1
    mx = int(np.diff(cu).max())
    q, k, v, _ = workloads.draw_dense(5 + window, nt, w.hq, w.hkv, w.d, device="cuda")
    dcu = torch.from_numpy(cu.astype(np.int32)).cuda()
    nb = vcs.vcs_attn_fwd_workspace_size(ns, nt, mx, w.hq, w.hkv, w.d)
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    o = torch.empty_like(q)
    lse = torch.empty((w.hq, nt), dtype=torch.float32, device="cuda")
    assert vcs.vcs_attn_fwd(q, k, v, dcu, ns, nt, mx, w.hq, w.hkv, w.d, 0.0, o, lse, ws, nb) == 0
    torch.cuda.synchronize()
    hdr = ws[:256].view(torch.int32).cpu().numpy()
    assert hdr[0] == 0 and hdr[128 // 4] == _units_of(cu, w.hq)
    check_sampled(q, k, v, cu, o, lse, np.random.default_rng(40 + window), n_seg=4, heads=[0, w.hq - 1])
