"""Gather oracle (test infrastructure): packed rows = trajectory rows at the gather map.

Each segment token n takes the Q/K/V rows of trajectory token tok_gather[n]
(the re-tokenised fresh stream of Algorithm 1 reuses the trajectory's tokens;
Sec. 3.4).  It is an exact copy, so the definition is plain indexing.
"""
import numpy as np


def gather_rows(x, tok_gather):
    """x[tok_gather] for a [Ntraj, H, d] array or tensor (returned as numpy)."""
    idx = np.asarray(tok_gather, dtype=np.int64)
    if hasattr(x, "detach"):
        import torch
        return x.detach().cpu()[torch.from_numpy(idx)]
    return np.asarray(x)[idx]


def scatter_add_rows(x_seg, tok_gather, traj_tokens: int):
    """Adjoint of gather_rows: out[t] = sum of x_seg[n] over the segment tokens n with
    tok_gather[n] = t (zero for a trajectory token no segment copies).  The gradient of a
    loss with respect to the trajectory rows is this sum over the token's copies (the
    chain rule through the copy); fp64."""
    x = np.asarray(x_seg, dtype=np.float64)
    out = np.zeros((int(traj_tokens),) + x.shape[1:], dtype=np.float64)
    np.add.at(out, np.asarray(tok_gather, dtype=np.int64), x)
    return out
