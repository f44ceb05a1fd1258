"""GPU parity of the gathered attention (vcs_attn_fwd_gathered / vcs_attn_bwd_gathered):
Q, K, V read from trajectory-layout tensors through the builder's gather map, the
backward's dQ, dK, dV summed over each trajectory token's segment copies.

The forward must equal vcs_attn_fwd on vcs_gather's copies bit for bit (same tiles,
same arithmetic).  The backward is compared with the fp64 oracle: the segment-layout
gradients of the attention oracle scattered into trajectory layout by the oracle's
scatter-add, relative L2 error <= 1e-2 per tensor (bf16 inputs, fp32 accumulation);
at full size on sampled trajectory tokens.
"""
import numpy as np
import pytest
import torch

from oracle import attention as oatt
from oracle import gather as og
from oracle import segments as oseg
from paper_2607_11185_gb300 import workloads
from tests.gpu_cases import random_steps

pytestmark = pytest.mark.gpu

REL = 1e-2


def _vcs():
    from paper_2607_11185_gb300 import vcs
    return vcs


def rel_err(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    nr = np.linalg.norm(ref)
    if nr < 1e-6:
        return np.abs(got - ref).max() / 1e-1
    return np.linalg.norm(got - ref) / nr


def _inputs(cu, img, txt, window, keep, hq, hkv, d, seed):
    vcs = _vcs()
    lay = vcs.build_segments(*(torch.from_numpy(np.asarray(x, np.int32)).cuda() for x in (cu, img, txt)), window, keep)
    ntraj = workloads.trajectory_tokens(np.asarray(img), np.asarray(txt))
    qt, kt, vt, _ = workloads.draw_dense(seed, max(ntraj, 1), hq, hkv, d, device="cuda")
    do = workloads.draw_dense(seed + 1, max(lay["num_tokens"], 1), hq, hkv, d, device="cuda")[3][: lay["num_tokens"]]
    return lay, qt, kt, vt, do.contiguous()


def _fwd_both(lay, qt, kt, vt):
    vcs = _vcs()
    o_g, lse_g = vcs.attn_fwd_gathered(qt, kt, vt, lay["tok_gather"], lay["cu_seqlens"], lay["max_seqlen"])
    q, k, v = vcs.gather(qt, kt, vt, lay["tok_gather"])
    o, lse = vcs.attn_fwd(q, k, v, lay["cu_seqlens"], lay["max_seqlen"])
    return (o_g, lse_g), (o, lse), (q, k, v)


FWD_CASES = [("tiny", None), ("traj8_w3", None), ("traj8_w3", (3, 2)), ("traj8_w3", (1, 0))]


@pytest.mark.parametrize("name,layout", FWD_CASES)
def test_fwd_equals_materialised_gather(name, layout):
    w = workloads.WORKLOADS[name]
    cu, img, txt = workloads.draw_steps(w)
    window, keep = layout if layout else (w.window, w.keep)
    lay, qt, kt, vt, _ = _inputs(cu, img, txt, window, keep, w.hq, w.hkv, w.d, w.seed)
    (o_g, lse_g), (o, lse), _ = _fwd_both(lay, qt, kt, vt)
    assert torch.equal(o_g, o)
    assert torch.equal(lse_g, lse)


@pytest.mark.parametrize("name,layout", [("tiny", None), ("traj8_w3", (3, 1))])
def test_fwd_against_oracle(name, layout):
    """The gathered forward directly against the fp64 oracle (on the oracle's own gather of the
    trajectory rows): the tiny workload in full, the 8-trajectory workload with one retained
    screenshot on sampled rows (O max-abs 2e-2, lse max-abs 2e-3)."""
    from tests.test_gpu_attn_fwd import LSE_TOL, O_TOL, check_sampled
    w = workloads.WORKLOADS[name]
    cu, img, txt = workloads.draw_steps(w)
    window, keep = layout if layout else (w.window, w.keep)
    lay, qt, kt, vt, _ = _inputs(cu, img, txt, window, keep, w.hq, w.hkv, w.d, w.seed)
    vcs = _vcs()
    o, lse = vcs.attn_fwd_gathered(qt, kt, vt, lay["tok_gather"], lay["cu_seqlens"], lay["max_seqlen"])
    torch.cuda.synchronize()
    g = lay["tok_gather"].cpu().numpy()
    cus = lay["cu_seqlens"].cpu().numpy()
    q, k, v = og.gather_rows(qt, g), og.gather_rows(kt, g), og.gather_rows(vt, g)
    if name == "tiny":
        ro, rl = oatt.attn_fwd(q, k, v, cus)
        assert np.abs(o.float().cpu().numpy() - ro).max() <= O_TOL
        assert np.abs(lse.cpu().numpy() - rl).max() <= LSE_TOL
    else:
        check_sampled(q, k, v, cus, o, lse, np.random.default_rng(17), n_seg=4)


@pytest.mark.parametrize("seed", range(301, 305))
def test_fwd_random_layouts(seed):
    cu, img, txt = random_steps(seed, max_traj=5, max_T=20, max_img=300, max_txt=40)
    lay, qt, kt, vt, _ = _inputs(cu, img, txt, 3, seed % 3, 4, 2, 128 if seed % 2 == 0 else 64, seed)
    assert lay["num_tokens"] > 0
    (o_g, lse_g), (o, lse), _ = _fwd_both(lay, qt, kt, vt)
    assert torch.equal(o_g, o) and torch.equal(lse_g, lse)


SMALL = [  # (cu, img, txt, window, keep, hq, hkv, d)
    ([0, 7, 10], [300, 200, 260, 100, 220, 200, 140, 300, 100, 200], [30, 60, 10, 50, 20, 40, 30, 60, 20, 30],
     2, 1, 4, 2, 128),
    ([0, 9], [100] * 9, [40, 30, 20, 60, 10, 50, 20, 30, 40], 2, 0, 2, 1, 64),
    ([0, 5, 5, 12], [120, 90, 60, 130, 70, 50, 80, 100, 90, 60, 40, 110],
     [20, 30, 40, 10, 20, 30, 10, 20, 30, 40, 10, 20], 3, 2, 6, 2, 128),
]


@pytest.mark.parametrize("case", range(len(SMALL)))
def test_bwd_full_oracle(case):
    cu, img, txt, window, keep, hq, hkv, d = SMALL[case]
    lay, qt, kt, vt, do = _inputs(cu, img, txt, window, keep, hq, hkv, d, 40 + case)
    vcs = _vcs()
    o, lse = vcs.attn_fwd_gathered(qt, kt, vt, lay["tok_gather"], lay["cu_seqlens"], lay["max_seqlen"])
    dq, dk, dv = vcs.attn_bwd_gathered(qt, kt, vt, lay["tok_gather"], o, lse, do, lay["cu_seqlens"],
                                       lay["max_seqlen"])
    g = lay["tok_gather"].cpu().numpy()
    cus = lay["cu_seqlens"].cpu().numpy()
    assert np.bincount(g).max() >= 2  # some trajectory tokens have several copies
    ntraj = qt.shape[0]
    rq, rk, rv = oatt.attn_bwd(og.gather_rows(qt, g), og.gather_rows(kt, g), og.gather_rows(vt, g), do.cpu(), cus)
    for name, got, seg in (("dq", dq, rq), ("dk", dk, rk), ("dv", dv, rv)):
        ref = og.scatter_add_rows(seg, g, ntraj)
        e = rel_err(got.float().cpu().numpy(), ref)
        assert e <= REL, (name, e)


def test_bwd_full_size_sampled():
    # traj8_w3 with keep 1 (screenshots and text carried into later segments): dQ of
    # trajectory tokens with several copies (the copies sit early in their segments,
    # where the oracle's row evaluation is cheap), dK/dV of tokens of each trajectory's
    # last step (one copy, near its segment's end)
    w = workloads.WORKLOADS["traj8_w3"]
    cu, img, txt = workloads.draw_steps(w)
    lay, qt, kt, vt, do = _inputs(cu, img, txt, w.window, 1, w.hq, w.hkv, w.d, 8)
    vcs = _vcs()
    o, lse = vcs.attn_fwd_gathered(qt, kt, vt, lay["tok_gather"], lay["cu_seqlens"], lay["max_seqlen"])
    dq, dk, dv = vcs.attn_bwd_gathered(qt, kt, vt, lay["tok_gather"], o, lse, do, lay["cu_seqlens"],
                                       lay["max_seqlen"])
    g = lay["tok_gather"].cpu().numpy()
    cus = lay["cu_seqlens"].cpu().numpy()
    seg_of = np.searchsorted(cus, np.arange(len(g)), side="right") - 1
    q, k, v = vcs.gather(qt, kt, vt, lay["tok_gather"])
    qc, kc, vc, doc = q.cpu(), k.cpu(), v.cpu(), do.cpu()
    rng = np.random.default_rng(3)
    counts = np.bincount(g, minlength=qt.shape[0])
    multi = np.flatnonzero(counts >= 3)
    got_q, ref_q = [], []
    heads = [0, w.hq - 1]
    for t in rng.choice(multi, size=4, replace=False):
        acc = np.zeros((len(heads), w.d))
        for n in np.flatnonzero(g == t):
            s = int(seg_of[n])
            b, e = int(cus[s]), int(cus[s + 1])
            acc += oatt.rows_dq(qc, kc, vc, doc, (b, e), heads, [int(n) - b])[0]
        got_q.append(dq[int(t)][heads].float().cpu().numpy())
        ref_q.append(acc)
    assert rel_err(np.concatenate([x.ravel() for x in got_q]), np.concatenate([x.ravel() for x in ref_q])) <= REL
    # the last 24 tokens of two trajectories: each has one copy, at the end of the last segment
    got_k, ref_k, got_v, ref_v = [], [], [], []
    gh = 1
    for tr in (0, len(cu) - 2):
        s = int(np.flatnonzero(lay["seg_traj"].cpu().numpy() == tr).max())
        b, e = int(cus[s]), int(cus[s + 1])
        keys = list(range(e - b - 24, e - b))
        rk, rv = oatt.keys_dkdv(qc, kc, vc, doc, (b, e), gh, keys)
        ts = g[b + np.asarray(keys)]
        assert (counts[ts] == 1).all()
        got_k.append(dk[torch.from_numpy(ts).cuda(), gh].float().cpu().numpy())
        got_v.append(dv[torch.from_numpy(ts).cuda(), gh].float().cpu().numpy())
        ref_k.append(rk)
        ref_v.append(rv)
    for got, ref in ((got_k, ref_k), (got_v, ref_v)):
        assert rel_err(np.concatenate([x.ravel() for x in got]), np.concatenate([x.ravel() for x in ref])) <= REL


def test_bwd_matches_segment_backward_scattered():
    # property at full size: the gathered backward equals the segment-layout backward's
    # gradients summed over each token's copies, to bf16 rounding of the per-copy terms
    w = workloads.WORKLOADS["traj8_w3"]
    cu, img, txt = workloads.draw_steps(w)
    lay, qt, kt, vt, do = _inputs(cu, img, txt, w.window, 1, w.hq, w.hkv, w.d, 9)
    vcs = _vcs()
    o, lse = vcs.attn_fwd_gathered(qt, kt, vt, lay["tok_gather"], lay["cu_seqlens"], lay["max_seqlen"])
    dq, dk, dv = vcs.attn_bwd_gathered(qt, kt, vt, lay["tok_gather"], o, lse, do, lay["cu_seqlens"],
                                       lay["max_seqlen"])
    q, k, v = vcs.gather(qt, kt, vt, lay["tok_gather"])
    sq, sk, sv = vcs.attn_bwd(q, k, v, o, lse, do, lay["cu_seqlens"], lay["max_seqlen"])
    g = lay["tok_gather"].long()
    for got, seg in ((dq, sq), (dk, sk), (dv, sv)):
        ref = torch.zeros(got.shape, dtype=torch.float32, device="cuda").index_add_(0, g, seg.float())
        assert ((got.float() - ref).norm() / ref.norm()).item() <= 5e-3


def test_edge_cases():
    vcs = _vcs()
    # no segment tokens: zero trajectory gradients
    qt, kt, vt, _ = workloads.draw_dense(5, 10, 2, 1, 64, device="cuda")
    z = torch.zeros(0, dtype=torch.int32, device="cuda")
    cu = torch.zeros(1, dtype=torch.int32, device="cuda")
    o = torch.zeros((0, 2, 64), dtype=torch.bfloat16, device="cuda")
    lse = torch.zeros((2, 0), dtype=torch.float32, device="cuda")
    o0, lse0 = vcs.attn_fwd_gathered(qt, kt, vt, z, cu, 0)
    assert o0.shape == (0, 2, 64) and lse0.shape == (2, 0)
    dq, dk, dv = vcs.attn_bwd_gathered(qt, kt, vt, z, o, lse, o, cu, 0)
    assert not dq.any() and not dk.any() and not dv.any()
    # one-token segments that all copy trajectory token 3: dV[3] = sum of dO over the group
    gi = torch.full((5,), 3, dtype=torch.int32, device="cuda")
    cu1 = torch.arange(6, dtype=torch.int32, device="cuda")
    o1, lse1 = vcs.attn_fwd_gathered(qt, kt, vt, gi, cu1, 1)
    assert (o1.float() - vt[3].float().expand(5, 2, 64)).abs().max().item() <= 1e-2
    do1 = workloads.draw_dense(6, 5, 2, 1, 64, device="cuda")[3]
    dq1, dk1, dv1 = vcs.attn_bwd_gathered(qt, kt, vt, gi, o1, lse1, do1, cu1, 1)
    ref = do1.float().sum((0, 1))
    assert rel_err(dv1[3, 0].float().cpu().numpy(), ref.cpu().numpy()) <= REL
    assert dv1[torch.arange(10, device="cuda") != 3].abs().max().item() == 0.0
    assert dq1.abs().max().item() <= 1e-3 and dk1.abs().max().item() <= 1e-3


def test_device_check_bad_gather_index():
    vcs = _vcs()
    qt, kt, vt, _ = workloads.draw_dense(7, 300, 2, 1, 128, device="cuda")
    gi = torch.arange(260, dtype=torch.int32, device="cuda")
    gi[200] = 300                                    # outside [0, 300)
    cu = torch.tensor([0, 260], dtype=torch.int32, device="cuda")
    with pytest.raises(vcs.VcsError) as e:
        vcs.attn_fwd_gathered(qt, kt, vt, gi, cu, 260)
    assert e.value.status == 6


def test_host_argument_errors():
    vcs = _vcs()
    qt, kt, vt, _ = workloads.draw_dense(8, 16, 2, 1, 64, device="cuda")
    gi = torch.arange(16, dtype=torch.int32, device="cuda")
    cu = torch.tensor([0, 16], dtype=torch.int32, device="cuda")
    o = torch.empty((16, 2, 64), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((2, 16), dtype=torch.float32, device="cuda")
    nb = vcs.vcs_attn_fwd_workspace_size(1, 16, 16, 2, 1, 64)
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    ok = vcs.vcs_attn_fwd_gathered(qt, kt, vt, 16, gi, cu, 1, 16, 16, 2, 1, 64, 0.0, o, lse, ws, nb)
    assert ok == 0
    assert vcs.vcs_attn_fwd_gathered(qt, kt, vt, 16, None, cu, 1, 16, 16, 2, 1, 64, 0.0, o, lse, ws, nb) == 1
    assert vcs.vcs_attn_fwd_gathered(qt, kt, vt, 0, gi, cu, 1, 16, 16, 2, 1, 64, 0.0, o, lse, ws, nb) == 1
    assert vcs.vcs_attn_fwd_gathered(qt, kt, vt, 1 << 31, gi, cu, 1, 16, 16, 2, 1, 64, 0.0, o, lse, ws, nb) == 4
    assert vcs.vcs_attn_fwd_gathered(qt, kt, vt, 16, gi, cu, 1, 16, 16, 2, 1, 32, 0.0, o, lse, ws, nb) == 2
    nbb = vcs.vcs_attn_bwd_gathered_workspace_size(1, 16, 16, 16, 2, 1, 64)
    assert nbb == vcs.vcs_attn_bwd_workspace_size(1, 16, 16, 2, 1, 64) + 16 * (2 + 2 * 1) * 64 * 4
    wsb = torch.zeros(nbb, dtype=torch.uint8, device="cuda")
    dq, dk, dv = torch.empty_like(qt), torch.empty_like(kt), torch.empty_like(vt)
    assert vcs.vcs_attn_bwd_gathered(qt, kt, vt, 16, gi, o, lse, o, cu, 1, 16, 16, 2, 1, 64, 0.0, dq, dk, dv, wsb,
                                     nbb - 256) == 8
