"""Cross-segment prefix reuse (test infrastructure: only tests, smoke() and the bench's
CPU baseline may use this package).

A fresh stream re-tokenises the text of the steps before its window (Algorithm 1; Sec. 3.4,
App. C.1), and the steps that leave the window join that text, so the next segment of a
trajectory starts with the same tokens as the previous one.  Causal attention row r of a
segment depends only on the segment's tokens 0..r (positions restart at 0 in every
segment), so wherever two consecutive segments of a trajectory agree on tokens 0..r, their
attention rows 0..r are equal and need computing once.

shared_prefix: per segment, the length of the longest common prefix of its gather map with
the previous segment of the same trajectory (0 for a trajectory's first segment): the plain
definition, written as a loop.
reuse_source: the segment whose row r a segment's row r equals when rows below skip[s] of
every segment s are taken from the previous segment (walk back while r < skip[s]).
"""
import numpy as np


def shared_prefix(cu_seqlens, seg_traj, tok_gather):
    cu = np.asarray(cu_seqlens, np.int64)
    st = np.asarray(seg_traj, np.int64)
    g = np.asarray(tok_gather, np.int64)
    out = np.zeros(len(cu) - 1, np.int64)
    for s in range(1, len(cu) - 1):
        if st[s] != st[s - 1]:
            continue
        a, b = g[cu[s]:cu[s + 1]], g[cu[s - 1]:cu[s]]
        i = 0
        while i < min(len(a), len(b)) and a[i] == b[i]:
            i += 1
        out[s] = i
    return out


def reuse_source(skip, s: int, r: int) -> int:
    while r < skip[s]:
        s -= 1
    return s
