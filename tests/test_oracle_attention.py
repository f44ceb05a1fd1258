"""Pins for the attention oracle (CPU only, fp64).

The paper does not spell attention out; the oracle computes the definition of
causal softmax attention within a segment.  These tests tie it to things
other than itself: a library routine (torch's scaled_dot_product_attention
on one segment), central finite differences of the analytic gradients,
closed forms on single-token segments, and invariants of softmax.
"""
import math

import numpy as np
import pytest
import torch

from oracle import attention as att


def rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def test_single_segment_matches_sdpa():
    L, hq, hkv, d = 37, 6, 2, 16
    q, k, v = rand((L, hq, d), 1), rand((L, hkv, d), 2), rand((L, hkv, d), 3)
    o, lse = att.attn_fwd(q, k, v, [0, L], row_block=8)
    G = hq // hkv
    tq = torch.from_numpy(q).permute(1, 0, 2)[None]
    tk = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(G, 0)[None]
    tv = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(G, 0)[None]
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=True)[0].permute(1, 0, 2)
    np.testing.assert_allclose(o, ref.numpy(), rtol=1e-12, atol=1e-12)
    # lse against logsumexp of the explicit masked score matrix
    s = torch.einsum("hid,hjd->hij", tq[0], tk[0]) / math.sqrt(d)
    s = s.masked_fill(torch.triu(torch.ones(L, L, dtype=torch.bool), 1), float("-inf"))
    np.testing.assert_allclose(lse, torch.logsumexp(s, -1).numpy(), rtol=1e-12, atol=1e-12)


def test_segments_are_independent():
    cu = [0, 5, 5, 17, 30]                       # includes an empty segment
    hq, hkv, d = 4, 2, 8
    N = cu[-1]
    q, k, v, do = rand((N, hq, d), 4), rand((N, hkv, d), 5), rand((N, hkv, d), 6), rand((N, hq, d), 7)
    o, lse = att.attn_fwd(q, k, v, cu)
    dq, dk, dv = att.attn_bwd(q, k, v, do, cu)
    for b, e in zip(cu[:-1], cu[1:]):
        if e == b:
            continue
        o1, l1 = att.attn_fwd(q[b:e], k[b:e], v[b:e], [0, e - b])
        g1 = att.attn_bwd(q[b:e], k[b:e], v[b:e], do[b:e], [0, e - b])
        np.testing.assert_allclose(o[b:e], o1, atol=1e-13)
        np.testing.assert_allclose(lse[:, b:e], l1, atol=1e-13)
        for full, part in zip((dq, dk, dv), g1):
            np.testing.assert_allclose(full[b:e], part, atol=1e-12)


def test_single_token_segments_closed_form():
    # a one-token segment attends only to itself: O = V, lse = s_00, dQ = dK = 0, dV = sum of dO over the group
    cu = list(range(0, 6))
    hq, hkv, d = 4, 2, 8
    q, k, v, do = rand((5, hq, d), 8), rand((5, hkv, d), 9), rand((5, hkv, d), 10), rand((5, hq, d), 11)
    o, lse = att.attn_fwd(q, k, v, cu)
    dq, dk, dv = att.attn_bwd(q, k, v, do, cu)
    G = hq // hkv
    for h in range(hq):
        g = h // G
        np.testing.assert_allclose(o[:, h], v[:, g], atol=1e-14)
        np.testing.assert_allclose(lse[h], (q[:, h] * k[:, g]).sum(-1) / math.sqrt(d), atol=1e-14)
    np.testing.assert_allclose(dq, 0, atol=1e-14)
    np.testing.assert_allclose(dk, 0, atol=1e-14)
    np.testing.assert_allclose(dv, do.reshape(5, hkv, G, d).sum(2), atol=1e-14)


def test_first_row_of_every_segment_copies_v():
    cu = [0, 9, 20]
    hq, hkv, d = 2, 1, 8
    q, k, v = rand((20, hq, d), 12), rand((20, hkv, d), 13), rand((20, hkv, d), 14)
    o, lse = att.attn_fwd(q, k, v, cu)
    for b in cu[:-1]:
        for h in range(hq):
            np.testing.assert_allclose(o[b, h], v[b, 0], atol=1e-14)


def test_lse_bounds():
    L, hq, hkv, d = 50, 2, 1, 16
    q, k, v = 3 * rand((L, hq, d), 15), rand((L, hkv, d), 16), rand((L, hkv, d), 17)
    _, lse = att.attn_fwd(q, k, v, [0, L])
    for h in range(hq):
        s = q[:, h] @ k[:, 0].T / math.sqrt(d)
        for i in range(L):
            m = s[i, : i + 1].max()
            assert m - 1e-12 <= lse[h, i] <= m + math.log(i + 1) + 1e-12


@pytest.mark.parametrize("hq,hkv", [(2, 1), (4, 2), (3, 3)])
def test_gradients_match_finite_differences(hq, hkv):
    cu = [0, 3, 8]
    N, d = 8, 4
    q, k, v, do = rand((N, hq, d), 20), rand((N, hkv, d), 21), rand((N, hkv, d), 22), rand((N, hq, d), 23)
    dq, dk, dv = att.attn_bwd(q, k, v, do, cu)

    def loss(qq, kk, vv):
        return float((att.attn_fwd(qq, kk, vv, cu)[0] * do).sum())

    h = 1e-6
    for name, x, g in (("q", q, dq), ("k", k, dk), ("v", v, dv)):
        num = np.zeros_like(x)
        for idx in np.ndindex(x.shape):
            xp = x.copy(); xp[idx] += h
            xm = x.copy(); xm[idx] -= h
            args = {"q": q, "k": k, "v": v}
            args[name] = xp
            fp = loss(args["q"], args["k"], args["v"])
            args[name] = xm
            fm = loss(args["q"], args["k"], args["v"])
            num[idx] = (fp - fm) / (2 * h)
        rel = np.linalg.norm(g - num) / np.linalg.norm(num)
        assert rel < 1e-6, (name, rel)


def test_gradient_sums():
    # sum_j dS_ij = 0 for every row => sum_j dK_j = 0 per segment; sum_j P_ij = 1 =>
    # sum_j dV_j = sum_i dO_i (over the group's heads) per segment
    cu = [0, 13, 40]
    hq, hkv, d = 4, 2, 8
    q, k, v, do = rand((40, hq, d), 30), rand((40, hkv, d), 31), rand((40, hkv, d), 32), rand((40, hq, d), 33)
    dq, dk, dv = att.attn_bwd(q, k, v, do, cu)
    for b, e in zip(cu[:-1], cu[1:]):
        np.testing.assert_allclose(dk[b:e].sum(0), 0, atol=1e-12)
        np.testing.assert_allclose(dv[b:e].sum(0), do[b:e].reshape(e - b, hkv, 2, d).sum((0, 2)), atol=1e-12)


def test_sampled_rows_match_full():
    cu = [0, 29, 70]
    hq, hkv, d = 4, 2, 8
    q, k, v, do = rand((70, hq, d), 40), rand((70, hkv, d), 41), rand((70, hkv, d), 42), rand((70, hq, d), 43)
    o, lse = att.attn_fwd(q, k, v, cu)
    dq, dk, dv = att.attn_bwd(q, k, v, do, cu)
    seg = (29, 70)
    rows = [0, 5, 40]
    heads = [1, 3]
    o_r, l_r = att.rows_fwd(q, k, v, seg, heads, rows)
    dq_r = att.rows_dq(q, k, v, do, seg, heads, rows)
    for c, i in enumerate(rows):
        for a, h in enumerate(heads):
            np.testing.assert_allclose(o_r[c, a], o[29 + i, h], atol=1e-13)
            np.testing.assert_allclose(l_r[a, c], lse[h, 29 + i], atol=1e-13)
            np.testing.assert_allclose(dq_r[c, a], dq[29 + i, h], atol=1e-12)
    keys = [3, 38, 40]
    dk_r, dv_r = att.keys_dkdv(q, k, v, do, seg, 1, keys)
    np.testing.assert_allclose(dk_r, dk[[29 + j for j in keys], 1], atol=1e-12)
    np.testing.assert_allclose(dv_r, dv[[29 + j for j in keys], 1], atol=1e-12)


@pytest.mark.parametrize("row_block", [1, 7, 512])
def test_blocked_key_gradients_match_full(row_block):
    # the blocked key-gradient function against the full backward and the row-by-row one,
    # on keys at the start, in the middle and at the end of a ragged segment, GQA 3:1
    cu = [0, 13, 61]
    hq, hkv, d = 6, 2, 8
    q, k, v, do = rand((61, hq, d), 50), rand((61, hkv, d), 51), rand((61, hkv, d), 52), rand((61, hq, d), 53)
    dq, dk, dv = att.attn_bwd(q, k, v, do, cu)
    seg = (13, 61)
    keys = [0, 1, 17, 30, 47]
    for g in range(hkv):
        dk_b, dv_b = att.keys_dkdv_blocked(q, k, v, do, seg, g, keys, row_block=row_block)
        np.testing.assert_allclose(dk_b, dk[[13 + j for j in keys], g], atol=1e-12)
        np.testing.assert_allclose(dv_b, dv[[13 + j for j in keys], g], atol=1e-12)
        dk_r, dv_r = att.keys_dkdv(q, k, v, do, seg, g, keys)
        np.testing.assert_allclose(dk_b, dk_r, atol=1e-12)
        np.testing.assert_allclose(dv_b, dv_r, atol=1e-12)
