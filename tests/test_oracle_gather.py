"""Pins for the gather oracle and its adjoint, the scatter-add of segment-layout
gradients into trajectory layout (CPU only, fp64).

A segment token is a copy of a trajectory token (the history re-tokenised into
each fresh stream, Alg. 1 / App. C.1), so the gradient with respect to a
trajectory row is the sum over that row's copies.  These tests tie the
scatter-add to the gather's plain definition (the adjoint identity), to a hand-worked
map, to the copy counts, and to finite differences of attention composed with the
gather on a builder layout whose segments share tokens.
"""
import numpy as np

from oracle import attention as att
from oracle import gather as og
from oracle import segments as oseg


def test_hand_worked():
    x = np.arange(5 * 2, dtype=np.float64).reshape(5, 1, 2) + 1.0
    out = og.scatter_add_rows(x, [0, 2, 2, 1, 2], 4)
    np.testing.assert_array_equal(out[0], x[0])
    np.testing.assert_array_equal(out[1], x[3])
    np.testing.assert_array_equal(out[2], x[1] + x[2] + x[4])
    np.testing.assert_array_equal(out[3], np.zeros((1, 2)))


def _layout():
    # window 2, keep 1: text history and a kept screenshot are copied into later segments
    cu = np.array([0, 7, 10], np.int32)
    img = np.array([3, 2, 4, 1, 2, 2, 1, 3, 1, 2], np.int32)
    txt = np.array([1, 2, 1, 2, 1, 1, 1, 2, 2, 1], np.int32)
    lay = oseg.build(cu, img, txt, 2, 1)
    return lay, int(img.sum() + txt.sum())


def test_layout_has_copies():
    lay, ntraj = _layout()
    counts = np.bincount(lay["tok_gather"], minlength=ntraj)
    assert counts.min() >= 1 and counts.max() >= 3


def test_adjoint_identity():
    lay, ntraj = _layout()
    g = lay["tok_gather"]
    rng = np.random.default_rng(1)
    y = rng.standard_normal((ntraj, 3, 4))
    x = rng.standard_normal((len(g), 3, 4))
    lhs = np.sum(og.gather_rows(y, g) * x)
    rhs = np.sum(y * og.scatter_add_rows(x, g, ntraj))
    assert abs(lhs - rhs) <= 1e-12 * (abs(lhs) + 1.0)


def test_copy_counts():
    lay, ntraj = _layout()
    g = lay["tok_gather"]
    ones = np.ones((len(g), 1, 1))
    np.testing.assert_array_equal(og.scatter_add_rows(ones, g, ntraj)[:, 0, 0], np.bincount(g, minlength=ntraj))


def test_attention_through_the_gather_finite_differences():
    # f(q_t, k_t, v_t) = <dO, attn(gather(q_t), gather(k_t), gather(v_t))>: its gradient with
    # respect to the trajectory rows is the scatter-add of the segment-layout gradients
    lay, ntraj = _layout()
    g, cu = lay["tok_gather"], lay["cu_seqlens"]
    rng = np.random.default_rng(2)
    hq, hkv, d = 2, 1, 4
    qt, kt, vt = (rng.standard_normal((ntraj, h, d)) for h in (hq, hkv, hkv))
    do = rng.standard_normal((len(g), hq, d))

    def f(qt, kt, vt):
        o, _ = att.attn_fwd(og.gather_rows(qt, g), og.gather_rows(kt, g), og.gather_rows(vt, g), cu)
        return np.sum(o * do)

    dq, dk, dv = att.attn_bwd(og.gather_rows(qt, g), og.gather_rows(kt, g), og.gather_rows(vt, g), do, cu)
    grads = [og.scatter_add_rows(x, g, ntraj) for x in (dq, dk, dv)]
    eps = 1e-6
    for which, (base, grad) in enumerate(zip((qt, kt, vt), grads)):
        for t in (0, int(np.argmax(np.bincount(g))), ntraj - 1):
            for c in (0, d - 1):
                plus, minus = [x.copy() for x in (qt, kt, vt)], [x.copy() for x in (qt, kt, vt)]
                plus[which][t, 0, c] += eps
                minus[which][t, 0, c] -= eps
                fd = (f(*plus) - f(*minus)) / (2 * eps)
                assert abs(fd - grad[t, 0, c]) <= 1e-6 * (1.0 + abs(fd)), (which, t, c, fd, grad[t, 0, c])
