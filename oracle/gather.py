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
