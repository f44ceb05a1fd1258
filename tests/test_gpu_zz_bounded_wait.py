"""The bounded device waits give up and report instead of hanging (one GB300).

vcs_selftest_bounded_wait waits on an mbarrier that nothing ever arrives on, with the same
try-wait loop and cycle limit the attention kernels use for every pipeline wait; the wait must
run out, leave VCS_ERR_DEVICE_TIMEOUT in the status word, and leave the context usable: an
attention forward launched afterwards matches the oracle.  No GPU fault, trap or hang is
involved: the wait is bounded by construction.
"""
import time

import numpy as np
import pytest
import torch

from oracle import attention as oatt
from paper_2607_11185_gb300 import workloads
from tests.gpu_cases import cu_from_lengths

pytestmark = pytest.mark.gpu


def test_wait_runs_out_and_reports():
    from paper_2607_11185_gb300 import vcs
    t0 = time.perf_counter()
    st = vcs.selftest_bounded_wait(100_000_000)          # ~50 ms at 2 GHz
    dt = time.perf_counter() - t0
    assert st == 7, vcs.vcs_status_string(st)            # VCS_ERR_DEVICE_TIMEOUT
    assert dt < 30.0
    # a status word that already holds an error keeps it
    word = torch.full((1,), 6, dtype=torch.int32, device="cuda")
    assert vcs.vcs_selftest_bounded_wait(word, 1000) == 0
    torch.cuda.synchronize()
    assert int(word.item()) == 6


def test_context_usable_after_the_timeout():
    from paper_2607_11185_gb300 import vcs
    assert vcs.selftest_bounded_wait(1_000_000) == 7
    cu = cu_from_lengths([129, 300])
    q, k, v, _ = workloads.draw_dense(91, int(cu[-1]), 4, 2, 64, device="cuda")
    o, lse = vcs.attn_fwd(q, k, v, torch.from_numpy(cu).cuda(), 300)
    ro, rl = oatt.attn_fwd(q.cpu(), k.cpu(), v.cpu(), cu)
    assert np.abs(o.float().cpu().numpy() - ro).max() <= 2e-2
    assert np.abs(lse.cpu().numpy() - rl).max() <= 2e-3
