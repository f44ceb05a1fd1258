"""Pins for the segment-builder oracle (CPU only).

The paper prints no worked example, so the fixtures under tests/golden/ are
segmentations traced by hand from Algorithm 1 (Sec. 3.4 / App. C.1).  The
closed forms and invariants below follow from the same algorithm and from
the item-count scaling stated in Sec. 3.4.
"""
import glob
import json
import os

import numpy as np
import pytest

from oracle import segments as seg
from paper_2607_11185_gb300 import workloads


def expected_from_fixture(fx):
    gather, src, mask, pos = [], [], [], []
    for s in fx["segments"]:
        g = np.concatenate([np.arange(a, b) for a, b in s["gather_ranges"]])
        st = np.concatenate([np.full(n, k) for k, n in s["src_steps"]])
        m = np.zeros(len(g), np.uint8)
        for a, b in s["mask_ranges"]:
            m[a:b] = 1
        assert len(st) == len(g)
        gather.append(g); src.append(st); mask.append(m); pos.append(np.arange(len(g)))
    return (np.concatenate(gather), np.concatenate(src), np.concatenate(mask), np.concatenate(pos))


FIXTURES = sorted(glob.glob(os.path.join(os.path.dirname(__file__), "golden", "seg_*.json")))


@pytest.mark.parametrize("path", FIXTURES, ids=[os.path.basename(p) for p in FIXTURES])
@pytest.mark.parametrize("method", ["replay", "closed"])
def test_hand_worked(path, method):
    fx = json.load(open(path))
    out = seg.build(fx["cu_steps"], fx["step_img"], fx["step_txt"], fx["window"], fx["keep"], method=method)
    g, st, m, p = expected_from_fixture(fx)
    np.testing.assert_array_equal(out["cu_seqlens"], fx["cu_seqlens"])
    np.testing.assert_array_equal(out["seg_traj"], fx["seg_traj"])
    np.testing.assert_array_equal(out["tok_gather"], g)
    np.testing.assert_array_equal(out["tok_src_step"], st)
    np.testing.assert_array_equal(out["tok_loss_mask"], m)
    np.testing.assert_array_equal(out["tok_pos"], p)


@pytest.mark.parametrize("keep,delta", [(0, 1), (0, 3), (0, 8), (1, 1), (5, 5), (8, 5), (2, 7)])
def test_segment_count_and_item_scaling(keep, delta):
    # S(T) closed form against the replay, and the O(nT/K) item count of Sec. 3.4
    for T in range(0, 120):
        n = len(seg.replay_episode(T, keep, delta))
        assert n == seg.segment_count(T, keep, delta)
        if T > keep + delta:
            assert n == 1 + int(np.ceil((T - keep - delta) / delta))
    # step-wise (K=0, delta=1) emits one item per turn (O(nT))
    assert seg.segment_count(50, 0, 1) == 50


def test_uniform_lengths_closed_form():
    # equal counts per step, K=0: L_j = j*delta*x + n_j*(i+x) with n_j new steps in segment j
    i, x, delta = 7, 3, 4
    for T in range(1, 40):
        L = seg.segment_lengths(np.full(T, i), np.full(T, x), 0, delta)
        for j, Lj in enumerate(L):
            n_j = min(delta, T - j * delta)
            assert Lj == j * delta * x + n_j * (i + x)


@pytest.mark.parametrize("seed", range(12))
def test_replay_matches_closed_form_random(seed):
    rng = np.random.default_rng(100 + seed)
    B = int(rng.integers(1, 6))
    Ts = rng.integers(0, 30, size=B)
    cu = np.concatenate([[0], np.cumsum(Ts)]).astype(np.int32)
    img = rng.integers(0, 40, size=cu[-1]).astype(np.int32)       # zero-token screenshots included
    txt = rng.integers(0, 9, size=cu[-1]).astype(np.int32)
    keep = int(rng.integers(0, 6))
    delta = int(rng.integers(1, 7))
    a = seg.build(cu, img, txt, delta, keep, method="replay")
    b = seg.build(cu, img, txt, delta, keep, method="closed")
    for key in a:
        np.testing.assert_array_equal(a[key], b[key], err_msg=key)


@pytest.mark.parametrize("seed", range(8))
def test_invariants(seed):
    rng = np.random.default_rng(200 + seed)
    B = int(rng.integers(1, 5))
    Ts = rng.integers(0, 25, size=B)
    cu = np.concatenate([[0], np.cumsum(Ts)]).astype(np.int32)
    img = rng.integers(0, 30, size=cu[-1]).astype(np.int32)
    txt = rng.integers(0, 7, size=cu[-1]).astype(np.int32)
    keep = int(rng.integers(0, 4))
    delta = int(rng.integers(1, 6))
    out = seg.build(cu, img, txt, delta, keep)
    cs = out["cu_seqlens"]
    step_off = np.concatenate([[0], np.cumsum(img.astype(np.int64) + txt)])
    traj_tok = np.concatenate([[0], step_off[cu[1:]]])
    trained = np.zeros(cu[-1], np.int64)
    for s in range(len(cs) - 1):
        b = out["seg_traj"][s]
        sl = slice(cs[s], cs[s + 1])
        g, st, p, m = out["tok_gather"][sl], out["tok_src_step"][sl], out["tok_pos"][sl], out["tok_loss_mask"][sl]
        # every token maps inside its own trajectory, at a token of its source step
        assert np.all((g >= traj_tok[b]) & (g < traj_tok[b + 1]))
        assert np.all((st >= cu[b]) & (st < cu[b + 1]))
        assert np.all((g >= step_off[st]) & (g < step_off[st + 1]))
        # source steps non-decreasing, positions 0..L-1, gather strictly increasing
        assert np.all(np.diff(st) >= 0) and np.all(np.diff(g) > 0)
        np.testing.assert_array_equal(p, np.arange(cs[s + 1] - cs[s]))
        # trainable tokens are response tokens
        resp = g >= step_off[st] + img[st]
        assert np.all(resp[m == 1])
        # screenshots appear for at most keep + delta steps
        img_steps = np.unique(st[~resp])
        assert len(img_steps) <= keep + delta
        np.add.at(trained, np.unique(st[m == 1]), 1)
    # each response is optimised exactly once (Sec. 3.4 / App. C.1); steps with
    # zero response tokens carry no trainable token
    has_txt = txt > 0
    assert np.all(trained[has_txt] == 1) and np.all(trained[~has_txt] == 0)


def test_window_covers_trajectory_is_identity():
    cu, img, txt = workloads.draw_steps(workloads.WORKLOADS["traj8_w3"])
    T_max = int(np.max(np.diff(cu)))
    out = seg.build(cu, img, txt, T_max, 0)
    assert len(out["cu_seqlens"]) - 1 == len(cu) - 1
    np.testing.assert_array_equal(out["tok_gather"], np.arange(int(img.sum()) + int(txt.sum())))
    # loss mask = response tokens of every step
    ref = np.concatenate([np.concatenate([np.zeros(i, np.uint8), np.ones(x, np.uint8)]) for i, x in zip(img, txt)])
    np.testing.assert_array_equal(out["tok_loss_mask"], ref)


def test_stepwise_is_window_one_and_keeps_only_last_screenshot():
    # K=0, delta=1: one item per turn, only that turn's screenshot (Sec. 1 step-wise training)
    cu, img, txt = workloads.draw_steps(workloads.WORKLOADS["traj8_w3"])
    out = seg.build(cu, img, txt, 1, 0)
    assert len(out["cu_seqlens"]) - 1 == len(img)
    step_off = np.concatenate([[0], np.cumsum(img.astype(np.int64) + txt)])
    for s in range(len(img)):
        sl = slice(out["cu_seqlens"][s], out["cu_seqlens"][s + 1])
        g, st = out["tok_gather"][sl], out["tok_src_step"][sl]
        is_img = g < step_off[st] + img[st]
        assert set(np.unique(st[is_img])) == {s}


def test_invalid_arguments():
    with pytest.raises(ValueError):
        seg.replay_episode(3, 0, 0)
    with pytest.raises(ValueError):
        seg.segment_count(3, -1, 2)
