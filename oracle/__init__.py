"""CPU oracle for the Visual Context Segmentation hot path (TEST INFRASTRUCTURE).

A plain, slow, obviously correct restatement of what the path computes,
written from the paper (Sec. 3.4, Algorithm 1, App. C.1 "Trajectory
Processing Algorithm", the RL objective of App. C.2) and from the definition
of causal softmax attention.
Floating point is fp64 throughout.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py`` (its CPU
baseline leg and its ``--impl reference`` arm) may import this package.  The
product path (``paper_2607_11185_gb300``) never imports, links or executes
anything here, and this package never imports the product path: the two share
no code.  Inputs arrive as plain numpy arrays / torch CPU tensors drawn by
``paper_2607_11185_gb300.workloads``, which holds none of the method's
arithmetic.

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
(hand-worked segmentations, closed forms, invariants, a library special case,
finite differences).  No function is "parity unpinned".
"""
from . import segments, attention, gather, loss, stream  # noqa: F401
