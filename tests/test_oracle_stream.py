"""Pins for oracle/stream.py: the gather-map form of Algorithm 1's (ids, mask, logp)
stream against a literal replay, and the compaction invariants.  CPU only."""
import numpy as np
import pytest

from oracle import segments as oseg
from oracle import stream as ostream


def _batch(seed, ntraj=5):
    rng = np.random.default_rng(seed)
    T = rng.integers(0, 14, size=ntraj)
    cu = np.concatenate([[0], np.cumsum(T)])
    img = rng.integers(0, 9, size=int(T.sum()))
    txt = rng.integers(0, 6, size=int(T.sum()))
    ntok = int((img + txt).sum())
    ids = rng.integers(0, 150000, size=ntok).astype(np.int32)
    logp = (-rng.random(ntok) * 5).astype(np.float32)
    return cu, img, txt, ids, logp


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("keep,delta", [(0, 1), (0, 3), (1, 1), (2, 3), (8, 5), (5, 5)])
def test_gather_form_equals_replay(seed, keep, delta):
    cu, img, txt, ids, logp = _batch(seed)
    lay = oseg.build(cu, img, txt, delta, keep, method="closed")
    f_ids, f_lp = ostream.stream_fields(ids, logp, lay["tok_gather"], lay["tok_loss_mask"])
    want_ids, want_mask, want_lp = [], [], []
    base = 0
    for b in range(len(cu) - 1):
        g0, g1 = cu[b], cu[b + 1]
        n = int((img[g0:g1] + txt[g0:g1]).sum())
        for s_ids, s_mask, s_lp in ostream.replay_stream(img[g0:g1], txt[g0:g1], ids[base:base + n],
                                                          logp[base:base + n], keep, delta):
            want_ids.append(s_ids)
            want_mask.append(s_mask)
            want_lp.append(s_lp)
        base += n
    cat = lambda xs, dt: np.concatenate(xs).astype(dt) if xs else np.zeros(0, dt)  # noqa: E731
    assert np.array_equal(f_ids, cat(want_ids, np.int32))
    assert np.array_equal(lay["tok_loss_mask"], cat(want_mask, np.uint8))
    assert np.array_equal(f_lp, cat(want_lp, np.float32))


@pytest.mark.parametrize("seed", range(4))
def test_each_response_token_trainable_once(seed):
    # "each assistant response is optimised exactly once": over the whole batch the
    # compacted trainable tokens map onto every response token exactly once, in order
    cu, img, txt, ids, logp = _batch(seed + 10, ntraj=7)
    lay = oseg.build(cu, img, txt, 3, 2, method="closed")
    idx = ostream.compact_trainable(lay["tok_loss_mask"])
    src = lay["tok_gather"][idx].astype(np.int64)
    off = np.concatenate([[0], np.cumsum(img + txt)])
    responses = np.concatenate([np.arange(off[t] + img[t], off[t + 1]) for t in range(len(img))]) \
        if len(img) else np.zeros(0, np.int64)
    assert np.array_equal(src, responses)
    # the compacted log-probabilities are exactly the trajectory's response log-probabilities
    _, f_lp = ostream.stream_fields(ids, logp, lay["tok_gather"], lay["tok_loss_mask"])
    assert np.array_equal(f_lp[idx], logp[responses])


def test_hand_worked():
    # one trajectory, 3 steps of 2 screenshot + 1 response tokens, keep 0, delta 2:
    # seg0 = steps 1, 2 (tokens 0..5), seg1 = response of steps 1, 2 as text + step 3 (tokens 2, 5, 6..8)
    ids = np.array([10, 11, 12, 20, 21, 22, 30, 31, 32], np.int32)
    lp = np.array([0, 0, -1.5, 0, 0, -2.5, 0, 0, -3.5], np.float32)
    lay = oseg.build([0, 3], [2, 2, 2], [1, 1, 1], 2, 0)
    f_ids, f_lp = ostream.stream_fields(ids, lp, lay["tok_gather"], lay["tok_loss_mask"])
    assert f_ids.tolist() == [10, 11, 12, 20, 21, 22, 12, 22, 30, 31, 32]
    assert f_lp.tolist() == [0, 0, -1.5, 0, 0, -2.5, 0, 0, 0, 0, -3.5]
    assert ostream.compact_trainable(lay["tok_loss_mask"]).tolist() == [2, 5, 10]
