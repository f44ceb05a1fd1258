"""GPU attention backward vs the fp64 oracle.

Tolerance (from the method's precision: bf16 inputs, fp32 accumulation):
relative L2 error <= 1e-2 per gradient tensor over all checked rows; where
the reference norm is below 1e-6 (exact zeros of one-token segments) the
absolute error must be <= 1e-3.
"""
import numpy as np
import pytest
import torch

from oracle import attention as oatt
from oracle import segments as oseg
from paper_2607_11185_gb300 import workloads
from tests.gpu_cases import bench_chunks, cu_from_lengths

pytestmark = pytest.mark.gpu

REL = 1e-2


def rel_err(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    nr = np.linalg.norm(ref)
    if nr < 1e-6:
        return np.abs(got - ref).max() / 1e-1      # abs <= 1e-3 maps to <= 1e-2
    return np.linalg.norm(got - ref) / nr


def run(q, k, v, do, cu):
    from paper_2607_11185_gb300 import vcs
    dcu = torch.from_numpy(np.asarray(cu, np.int32)).cuda()
    mx = int(np.diff(cu).max())
    o, lse = vcs.attn_fwd(q, k, v, dcu, mx)
    dq, dk, dv = vcs.attn_bwd(q, k, v, o, lse, do, dcu, mx)
    return o, lse, dq, dk, dv


CASES = [
    ([1, 127, 128, 129, 255, 256, 257, 300], 2, 1, 64),
    ([1, 127, 128, 129, 255, 256, 257, 300], 2, 1, 128),
    ([600, 1, 383, 513], 7, 1, 128),
    ([640, 129], 4, 4, 64),
    ([1000], 6, 2, 128),
]


@pytest.mark.parametrize("lengths,hq,hkv,d", CASES)
def test_small_shapes_full_oracle(lengths, hq, hkv, d):
    cu = cu_from_lengths(lengths)
    q, k, v, do = workloads.draw_dense(31 + d + hq, int(cu[-1]), hq, hkv, d, device="cuda")
    _, _, dq, dk, dv = run(q, k, v, do, cu)
    rq, rk, rv = oatt.attn_bwd(q.cpu(), k.cpu(), v.cpu(), do.cpu(), cu)
    for name, got, ref in (("dq", dq, rq), ("dk", dk, rk), ("dv", dv, rv)):
        e = rel_err(got.float().cpu().numpy(), ref)
        assert e <= REL, (name, e)


def test_tiny_workload_full_oracle():
    w = workloads.WORKLOADS["tiny"]
    cu_s, img, txt = workloads.draw_steps(w)
    lay = oseg.build(cu_s, img, txt, w.window, w.keep)
    qt, kt, vt = workloads.draw_traj_qkv(w, workloads.trajectory_tokens(img, txt), device="cuda")
    g = torch.from_numpy(lay["tok_gather"].astype(np.int64)).cuda()
    q, k, v = qt[g], kt[g], vt[g]
    do = workloads.draw_dout(w, q.shape[0], device="cuda")
    _, _, dq, dk, dv = run(q, k, v, do, lay["cu_seqlens"])
    rq, rk, rv = oatt.attn_bwd(q.cpu(), k.cpu(), v.cpu(), do.cpu(), lay["cu_seqlens"])
    for got, ref in ((dq, rq), (dk, rk), (dv, rv)):
        assert rel_err(got.float().cpu().numpy(), ref) <= REL


def test_single_token_segments():
    cu = cu_from_lengths([1] * 24)
    q, k, v, do = workloads.draw_dense(9, 24, 4, 2, 64, device="cuda")
    _, _, dq, dk, dv = run(q, k, v, do, cu)
    assert dq.abs().max().item() <= 1e-3 and dk.abs().max().item() <= 1e-3
    ref_dv = do.float().view(24, 2, 2, 64).sum(2)
    assert rel_err(dv.float().cpu().numpy(), ref_dv.cpu().numpy()) <= REL


def test_large_logits_stress():
    cu = cu_from_lengths([700, 333])
    q, k, v, do = workloads.draw_dense(22, int(cu[-1]), 2, 1, 128, device="cuda", scale=6.0)
    _, _, dq, dk, dv = run(q, k, v, do, cu)
    rq, rk, rv = oatt.attn_bwd(q.cpu(), k.cpu(), v.cpu(), do.cpu(), cu)
    for got, ref in ((dq, rq), (dk, rk), (dv, rv)):
        assert rel_err(got.float().cpu().numpy(), ref) <= REL


def check_sampled_grads(q, k, v, do, cu, dq, dk, dv, rng, n_seg=4, n_rows=6, tail=48):
    """dQ on sampled rows; dK/dV on the last `tail` keys of sampled segments; gradient sums."""
    nseg = len(cu) - 1
    lens = np.diff(cu)
    hq, hkv = q.shape[1], k.shape[1]
    G = hq // hkv
    segs = sorted({int(np.argmin(lens)), int(np.argmax(lens)), 0, nseg - 1,
                   *[int(x) for x in rng.integers(0, nseg, size=n_seg)]})
    got_q, ref_q, got_k, ref_k, got_v, ref_v = [], [], [], [], [], []
    for s in segs:
        b, e = int(cu[s]), int(cu[s + 1])
        L = e - b
        heads = sorted({0, hq - 1, int(rng.integers(0, hq))})
        rows = sorted({0, L - 1, *[int(x) for x in rng.integers(0, L, size=n_rows)]})
        ref = oatt.rows_dq(q, k, v, do, (b, e), heads, rows)
        idx = torch.tensor([b + r for r in rows], device=dq.device)
        got_q.append(dq[idx][:, heads].float().cpu().numpy())
        ref_q.append(ref)
        g = int(rng.integers(0, hkv))
        keys = list(range(max(0, L - tail), L))
        rk, rv = oatt.keys_dkdv(q, k, v, do, (b, e), g, keys)
        kidx = torch.tensor([b + j for j in keys], device=dk.device)
        got_k.append(dk[kidx, g].float().cpu().numpy())
        ref_k.append(rk)
        got_v.append(dv[kidx, g].float().cpu().numpy())
        ref_v.append(rv)
        # sum_j dK_j = 0 and sum_j dV_j = sum_i dO_i over the group, per segment (any size)
        sdk = dk[b:e].float().sum(0)
        assert (sdk.abs().max() / dk[b:e].float().abs().sum(0).max().clamp_min(1e-6)).item() < 1e-2
        sdv = dv[b:e].float().sum(0)
        sdo = do[b:e].float().view(L, hkv, G, -1).sum((0, 2))
        assert ((sdv - sdo).norm() / sdo.norm()).item() < 1e-2
    for name, got, ref in (("dq", got_q, ref_q), ("dk", got_k, ref_k), ("dv", got_v, ref_v)):
        e = rel_err(np.concatenate([x.ravel() for x in got]), np.concatenate([x.ravel() for x in ref]))
        assert e <= REL, (name, e)


def _layout_inputs(name, first_chunk=False):
    """The workload's inputs in segment layout; with first_chunk, only the segments of the
    benchmark's first launch (its first trajectory chunk)."""
    w = workloads.WORKLOADS[name]
    cu_s, img, txt = workloads.draw_steps(w)
    lay = oseg.build(cu_s, img, txt, w.window, w.keep)
    qt, kt, vt = workloads.draw_traj_qkv(w, workloads.trajectory_tokens(img, txt), device="cuda")
    cu = lay["cu_seqlens"]
    if first_chunk:
        cu = cu[: bench_chunks(w, lay, len(cu_s) - 1)[0][1] + 1]
    nt = int(cu[-1])
    g = torch.from_numpy(lay["tok_gather"][:nt].astype(np.int64)).cuda()
    q, k, v = qt[g], kt[g], vt[g]
    do = workloads.draw_dout(w, len(lay["tok_gather"]), device="cuda")[:nt].contiguous()
    return q, k, v, do, cu


def test_traj8_full_size_sampled():
    q, k, v, do, cu = _layout_inputs("traj8_w3")
    _, _, dq, dk, dv = run(q, k, v, do, cu)
    check_sampled_grads(q, k, v, do, cu, dq, dk, dv, np.random.default_rng(8))


def test_traj32_first_chunk_sampled():
    q, k, v, do, cu = _layout_inputs("traj32_w3", first_chunk=True)
    _, _, dq, dk, dv = run(q, k, v, do, cu)
    check_sampled_grads(q, k, v, do, cu, dq, dk, dv, np.random.default_rng(32), n_seg=2, n_rows=4, tail=16)


def test_long_horizon_first_chunk_sampled():
    q, k, v, do, cu = _layout_inputs("traj16x50_w8", first_chunk=True)
    _, _, dq, dk, dv = run(q, k, v, do, cu)
    check_sampled_grads(q, k, v, do, cu, dq, dk, dv, np.random.default_rng(50), n_seg=1, n_rows=3, tail=8)


def test_long_horizon_early_and_middle_key_tiles():
    """dK, dV at full size where the backward does the most work: one kv head of the shortest
    segment of the benchmark's first long-horizon chunk (L = 25,696), on the first key tile
    (keys 0-127: every query tile of the segment and all five heads of the group reach it), a
    tile in the middle of the segment and the ragged last tile, against the oracle evaluated
    for those keys over all their query rows."""
    q, k, v, do, cu = _layout_inputs("traj16x50_w8", first_chunk=True)
    _, _, dq, dk, dv = run(q, k, v, do, cu)
    lens = np.diff(cu)
    s = int(np.argmin(lens))
    b, e = int(cu[s]), int(cu[s + 1])
    L = e - b
    mid = (L // 2) // 128 * 128
    last = (L - 1) // 128 * 128
    keys = list(range(0, 128)) + list(range(mid, mid + 128)) + list(range(last, L))
    g = 3
    rk, rv = oatt.keys_dkdv_blocked(q, k, v, do, (b, e), g, keys, row_block=1024)
    kidx = torch.tensor([b + j for j in keys], device=dk.device)
    for name, got, ref in (("dk", dk[kidx, g], rk), ("dv", dv[kidx, g], rv)):
        got = got.float().cpu().numpy()
        for lo, hi in ((0, 128), (128, 256), (256, len(keys))):   # each tile on its own
            err = rel_err(got[lo:hi], ref[lo:hi])
            assert err <= REL, (name, lo, err)


def test_traj8_longest_segment_every_key_and_row():
    """The 8-trajectory workload's longest segment (5,671 tokens) for one kv head in full: dK,
    dV of every key and dQ of every row of the group's seven query heads, against the full
    oracle on that group."""
    q, k, v, do, cu = _layout_inputs("traj8_w3")
    _, _, dq, dk, dv = run(q, k, v, do, cu)
    lens = np.diff(cu)
    s = int(np.argmax(lens))
    b, e = int(cu[s]), int(cu[s + 1])
    hq, hkv = q.shape[1], k.shape[1]
    G = hq // hkv
    g = 2
    heads = slice(g * G, (g + 1) * G)
    rq, rk, rv = oatt.attn_bwd(q[b:e, heads].cpu(), k[b:e, g:g + 1].cpu(), v[b:e, g:g + 1].cpu(),
                               do[b:e, heads].cpu(), [0, e - b])
    for name, got, ref in (("dq", dq[b:e, heads], rq), ("dk", dk[b:e, g:g + 1], rk), ("dv", dv[b:e, g:g + 1], rv)):
        err = rel_err(got.float().cpu().numpy(), ref)
        assert err <= REL, (name, err)
