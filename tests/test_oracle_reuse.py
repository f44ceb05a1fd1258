"""Pins for the prefix-reuse oracle (CPU only).

The shared prefix of consecutive segments is tied to the closed form of the segmentation
(segment j+1 of a trajectory repeats segment j's text history: the response tokens of the
steps before a_j, sum_{t < a_j} txt_t of them, where a screenshot of every step has at least
one token), and the reading that equal prefixes give equal attention rows is checked on the
attention oracle itself, segment by segment.
"""
import numpy as np
import pytest

from oracle import attention as att
from oracle import reuse
from oracle import segments as oseg


def _batch(seed, T=(1, 16), img=(1, 30), txt=(1, 9), ntraj=5):
    rng = np.random.default_rng(seed)
    Ts = rng.integers(T[0], T[1] + 1, size=ntraj)
    cu = np.concatenate([[0], np.cumsum(Ts)]).astype(np.int32)
    return (cu, rng.integers(img[0], img[1] + 1, size=int(cu[-1])).astype(np.int32),
            rng.integers(txt[0], txt[1] + 1, size=int(cu[-1])).astype(np.int32))


@pytest.mark.parametrize("window,keep", [(1, 0), (3, 0), (2, 1), (3, 2), (5, 5)])
def test_shared_prefix_closed_form(window, keep):
    cu, img, txt = _batch(window * 10 + keep)
    lay = oseg.build(cu, img, txt, window, keep)
    got = reuse.shared_prefix(lay["cu_seqlens"], lay["seg_traj"], lay["tok_gather"])
    want = []
    for b in range(len(cu) - 1):
        T = int(cu[b + 1] - cu[b])
        tx = txt[cu[b]:cu[b + 1]]
        for j, (a, s, e) in enumerate(oseg.episode_bounds(T, keep, window)):
            if j == 0:
                want.append(0)
            else:
                a_prev = oseg.episode_bounds(T, keep, window)[j - 1][0]
                want.append(int(tx[: a_prev - 1].sum()))
    np.testing.assert_array_equal(got, want)


def test_zero_token_screenshot_extends_the_prefix():
    # step 1's screenshot has no tokens: segment 0 then continues with step 1's text, which
    # is also where segment 1 continues, so the common prefix runs past the history
    cu = np.array([0, 4], np.int32)
    img = np.array([0, 5, 5, 5], np.int32)
    txt = np.array([2, 3, 1, 2], np.int32)
    lay = oseg.build(cu, img, txt, 1, 0)     # segments: steps {1}, {2}, {3}, {4}
    sp = reuse.shared_prefix(lay["cu_seqlens"], lay["seg_traj"], lay["tok_gather"])
    # segment 1 = txt1 | img2 txt2; segment 0 = img1 (empty) txt1: common prefix txt1 (2 tokens)
    assert list(sp) == [0, 2, 2, 5]


def test_rows_equal_over_the_shared_prefix():
    cu, img, txt = _batch(7, T=(6, 12), img=(20, 60), txt=(5, 20), ntraj=2)
    lay = oseg.build(cu, img, txt, 2, 1)
    sp = reuse.shared_prefix(lay["cu_seqlens"], lay["seg_traj"], lay["tok_gather"])
    ntraj = int(img.sum() + txt.sum())
    rng = np.random.default_rng(1)
    qt, kt, vt = rng.standard_normal((ntraj, 2, 8)), rng.standard_normal((ntraj, 1, 8)), rng.standard_normal((ntraj, 1, 8))
    g, cus = lay["tok_gather"], lay["cu_seqlens"]
    o, lse = att.attn_fwd(qt[g], kt[g], vt[g], cus)
    assert sp.max() > 0
    for s in range(1, len(cus) - 1):
        n = int(sp[s])
        b, pb = int(cus[s]), int(cus[s - 1])
        # equal up to fp64 rounding (the oracle evaluates rows in blocks through a library matmul)
        np.testing.assert_allclose(o[b:b + n], o[pb:pb + n], rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(lse[:, b:b + n], lse[:, pb:pb + n], rtol=1e-12, atol=1e-12)
        if n < min(cus[s + 1] - b, b - pb):   # the next row differs (different token)
            assert g[b + n] != g[pb + n]


def test_reuse_source_walks_back():
    skip = np.array([0, 256, 512, 0, 256])
    assert reuse.reuse_source(skip, 2, 100) == 0
    assert reuse.reuse_source(skip, 2, 300) == 1
    assert reuse.reuse_source(skip, 2, 600) == 2
    assert reuse.reuse_source(skip, 4, 10) == 3
