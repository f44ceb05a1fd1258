"""Segment-builder oracle (test infrastructure; see the package docstring).

Two independent builders of the same segmentation:

* ``replay_episode`` replays Algorithm 1 (Sec. 3.4; restated in App. C.1)
  turn by turn: a history of steps with an image flag, a screenshot counter
  ``n_img``, the prune trigger ``n_img > K + delta``, "drop the oldest delta
  screenshots", and a fresh zero-mask stream re-tokenised from the history.
* ``episode_bounds`` is the closed form of the same rule: the first segment
  takes K + delta new steps, every later one delta new steps, and retains the
  K most recent earlier steps with their screenshots.

Readings where the paper is silent:
  * the step model: step t contributes img[t] screenshot tokens followed by
    txt[t] response tokens; the screenshot of step 1 is the initial
    observation and every screenshot increments ``n_img`` (also zero-token
    ones);
  * a screenshot dropped from the window is carried by the step's own text
    tokens (no extra summary tokens);
  * the observation after the final action is not a step, so no trailing
    segment without trainable tokens is produced; an empty episode has no
    segment;
  * positions restart at 0 in every segment (a fresh stream).

Token-level outputs (``build``):
  cu_seqlens[S+1]   segment boundaries in the packed buffer
  seg_traj[S]       trajectory of each segment
  tok_gather[N]     index into the concatenated trajectory token buffer
  tok_src_step[N]   global (0-based) step index of the token
  tok_pos[N]        position within its segment
  tok_loss_mask[N]  1 on response tokens of the segment's new steps
"""
from __future__ import annotations

from typing import List, Tuple

import numpy as np

IMG, TXT = "img", "txt"
Run = Tuple[int, str, int]          # (step t 1-based, kind, trainable 0/1)


def _check(keep: int, delta: int):
    if delta < 1 or keep < 0:
        raise ValueError("need delta >= 1 and keep >= 0")


def replay_episode(num_steps: int, keep: int, delta: int) -> List[List[Run]]:
    """Algorithm 1 replayed literally on one episode of ``num_steps`` turns.

    Returns one list of runs per saved segment; a run names a step, which
    part of the step (screenshot or response) and its loss mask.
    """
    _check(keep, delta)
    saved: List[List[Run]] = []
    if num_steps == 0:
        return saved
    history: List[list] = []        # [step, screenshot still present]
    stream: List[Run] = []
    n_img = 0
    for t in range(1, num_steps + 1):
        # the screenshot this turn responds to arrives
        history.append([t, True])
        n_img += 1
        if n_img > keep + delta:
            # prune: save the stream, forget the oldest delta screenshots,
            # and re-tokenise the history into a fresh stream with mask 0
            saved.append(stream)
            removed = 0
            for entry in history:
                if removed == delta:
                    break
                if entry[1]:
                    entry[1] = False
                    removed += 1
            n_img -= delta
            stream = []
            for step, has_img in history:
                if has_img:
                    stream.append((step, IMG, 0))
                if step < t:                     # step t has not answered yet
                    stream.append((step, TXT, 0))
        else:
            # token-diff append of the new observation
            stream.append((t, IMG, 0))
        # the response of turn t is appended as trainable tokens
        stream.append((t, TXT, 1))
    saved.append(stream)
    return saved


def segment_count(num_steps: int, keep: int, delta: int) -> int:
    """S(T): 0 for an empty episode, 1 if T <= K + delta, else 1 + ceil((T-K-delta)/delta)."""
    _check(keep, delta)
    if num_steps == 0:
        return 0
    if num_steps <= keep + delta:
        return 1
    return 1 + -(-(num_steps - keep - delta) // delta)


def episode_bounds(num_steps: int, keep: int, delta: int) -> List[Tuple[int, int, int]]:
    """(a_j, s_j, e_j), 1-based: full steps a_j..e_j, new (trainable) steps s_j..e_j."""
    out = []
    for j in range(segment_count(num_steps, keep, delta)):
        if j == 0:
            s = 1
            e = min(keep + delta, num_steps)
        else:
            s = keep + delta + (j - 1) * delta + 1
            e = min(s + delta - 1, num_steps)
        out.append((max(1, s - keep), s, e))
    return out


def closed_form_episode(num_steps: int, keep: int, delta: int) -> List[List[Run]]:
    """Runs of every segment from the closed form ``episode_bounds``."""
    segs = []
    for a, s, e in episode_bounds(num_steps, keep, delta):
        runs: List[Run] = [(t, TXT, 0) for t in range(1, a)]
        for t in range(a, e + 1):
            runs.append((t, IMG, 0))
            runs.append((t, TXT, 1 if t >= s else 0))
        segs.append(runs)
    return segs


def segment_lengths(img: np.ndarray, txt: np.ndarray, keep: int, delta: int) -> List[int]:
    """L_j = sum_{t<a_j} txt_t + sum_{t=a_j}^{e_j} (img_t + txt_t), per segment."""
    out = []
    for a, s, e in episode_bounds(len(img), keep, delta):
        out.append(int(np.sum(txt[: a - 1], dtype=np.int64)
                       + np.sum(img[a - 1: e], dtype=np.int64) + np.sum(txt[a - 1: e], dtype=np.int64)))
    return out


def build(cu_steps, step_img, step_txt, window: int, keep: int = 0, method: str = "replay"):
    """Token-level segment layout for a batch of trajectories (see module docstring)."""
    cu_steps = np.asarray(cu_steps, dtype=np.int64)
    step_img = np.asarray(step_img, dtype=np.int64)
    step_txt = np.asarray(step_txt, dtype=np.int64)
    maker = replay_episode if method == "replay" else closed_form_episode
    cu = [0]
    seg_traj, gather, src, pos, mask = [], [], [], [], []
    traj_base = 0
    for b in range(len(cu_steps) - 1):
        g0, g1 = int(cu_steps[b]), int(cu_steps[b + 1])
        img, txt = step_img[g0:g1], step_txt[g0:g1]
        # token offset of step t's screenshot inside this trajectory
        step_off = np.concatenate([[0], np.cumsum(img + txt)])
        for runs in maker(g1 - g0, keep, window):
            length = 0
            for t, kind, m in runs:
                n = int(img[t - 1] if kind == IMG else txt[t - 1])
                first = traj_base + int(step_off[t - 1]) + (0 if kind == IMG else int(img[t - 1]))
                gather.append(np.arange(first, first + n, dtype=np.int64))
                src.append(np.full(n, g0 + t - 1, dtype=np.int64))
                pos.append(np.arange(length, length + n, dtype=np.int64))
                mask.append(np.full(n, m, dtype=np.int64))
                length += n
            cu.append(cu[-1] + length)
            seg_traj.append(b)
        traj_base += int(step_off[-1])

    def cat(parts, dtype):
        return np.concatenate(parts).astype(dtype) if parts else np.zeros(0, dtype)

    return dict(cu_seqlens=np.asarray(cu, dtype=np.int32),
                seg_traj=np.asarray(seg_traj, dtype=np.int32),
                tok_gather=cat(gather, np.int32),
                tok_src_step=cat(src, np.int32),
                tok_pos=cat(pos, np.int32),
                tok_loss_mask=cat(mask, np.uint8))
