"""Token-ID stream fields of Algorithm 1 (App. C.1), test infrastructure.

Every saved segment of Algorithm 1 is a triple (ids, mask, logp): response
tokens are appended with mask 1 and their rollout log-probabilities,
observation tokens and the re-tokenised history of a fresh stream with mask 0
and log-probability 0.  Over the segment layout (the builder's gather map and
loss mask) the fields are, for segment token n with trajectory token g(n):

  ids[n]  = traj_ids[g(n)]
  logp[n] = traj_logp[g(n)] if mask[n] = 1 else 0

and the trainable tokens, compacted in order, are the n with mask[n] = 1.
``replay_stream`` builds the same fields by replaying Algorithm 1 literally
(token diffs, prune, fresh stream) on one trajectory, as an independent check.
"""
from __future__ import annotations

import numpy as np

from . import segments as oseg


def stream_fields(traj_ids, traj_logp, tok_gather, tok_loss_mask):
    """(ids int32 [N], logp float32 [N]) from the gather map and loss mask."""
    g = np.asarray(tok_gather, dtype=np.int64)
    m = np.asarray(tok_loss_mask) != 0
    ids = np.asarray(traj_ids, dtype=np.int32)[g]
    lp = np.where(m, np.asarray(traj_logp, dtype=np.float32)[g], np.float32(0.0)).astype(np.float32)
    return ids, lp


def compact_trainable(tok_loss_mask):
    """Indices of the trainable tokens, in order (int32)."""
    return np.flatnonzero(np.asarray(tok_loss_mask) != 0).astype(np.int32)


def replay_stream(img, txt, ids, logp, keep: int, delta: int):
    """Algorithm 1 replayed on one trajectory's token IDs and log-probabilities.

    img, txt: per-step token counts; ids, logp: the trajectory's token buffer
    (step t = img_t screenshot tokens then txt_t response tokens).  Returns a
    list of (ids, mask, logp) per saved segment."""
    img = np.asarray(img, dtype=np.int64)
    txt = np.asarray(txt, dtype=np.int64)
    off = np.concatenate([[0], np.cumsum(img + txt)])
    out = []
    for runs in oseg.replay_episode(len(img), keep, delta):
        sid, smask, slp = [], [], []
        for t, kind, m in runs:
            lo = int(off[t - 1]) + (0 if kind == oseg.IMG else int(img[t - 1]))
            n = int(img[t - 1] if kind == oseg.IMG else txt[t - 1])
            for k in range(lo, lo + n):
                sid.append(int(ids[k]))
                smask.append(m)
                # trainable response tokens keep their rollout log-probability; every other
                # token of the stream (observations, re-tokenised history) carries 0
                slp.append(float(logp[k]) if m == 1 else 0.0)
        out.append((np.asarray(sid, np.int32), np.asarray(smask, np.uint8), np.asarray(slp, np.float32)))
    return out
