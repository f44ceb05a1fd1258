"""The backward entry point that allocates nothing (vcs_attn_bwd_noalloc).

Some callers cannot allocate device memory: a plugin whose host framework
owns all device memory and passes it only the input and output tensors, or a
latency-critical loop that must not call cudaMalloc.  vcs_attn_bwd_noalloc
serves them from a fixed scratch array inside the library.  These tests call
it through the C ABI and check it against vcs_attn_bwd (the entry point with
a caller workspace) and against the fp64 oracle on two calls in a row, which
share the same scratch, and check that a problem larger than the scratch is
refused before any launch.
This file runs last so that a failure here leaves every other test run.
"""
import numpy as np
import pytest
import torch

from oracle import attention as oatt
from paper_2607_11185_gb300 import workloads
from tests.gpu_cases import cu_from_lengths

pytestmark = pytest.mark.gpu

REL = 1e-2   # the relative-L2 tolerance of the backward parity tests


def rel(a, b):
    a, b = a.float(), b.float()
    return ((a - b).norm() / b.norm().clamp_min(1e-6)).item()


@pytest.mark.parametrize("d", [64, 128])
def test_noalloc_matches_workspace_entry_point_twice(d):
    from paper_2607_11185_gb300 import vcs
    lengths = [1, 127, 128, 129, 300, 257]
    cu = cu_from_lengths(lengths)
    n, hq, hkv = int(cu[-1]), 4, 2
    assert vcs.vcs_attn_bwd_workspace_size(len(lengths), n, max(lengths), hq, hkv, d) <= vcs.NOALLOC_SCRATCH_BYTES
    dcu = torch.from_numpy(cu).cuda()
    for call in range(2):                        # the second call reuses the scratch of the first
        q, k, v, do = workloads.draw_dense(500 + 10 * call + d, n, hq, hkv, d, device="cuda")
        o, lse = vcs.attn_fwd(q, k, v, dcu, max(lengths))
        ref = vcs.attn_bwd(q, k, v, o, lse, do, dcu, max(lengths))
        dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
        status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        st = vcs.vcs_attn_bwd_noalloc(q, k, v, o, lse, do, dcu, len(lengths), n, max(lengths), hq, hkv, d, 0.0,
                                      dq, dk, dv, status)
        assert st == 0, vcs.vcs_status_string(st)
        torch.cuda.synchronize()
        assert status.item() == 0
        for got, want in zip((dq, dk, dv), ref):
            assert rel(got, want) <= REL
        # and directly against the oracle, so that a fault shared by both entry points shows
        exact = oatt.attn_bwd(q.cpu(), k.cpu(), v.cpu(), do.cpu(), cu)
        for got, want in zip((dq, dk, dv), exact):
            assert rel(got.cpu(), torch.from_numpy(want)) <= REL


def test_noalloc_refuses_problems_larger_than_its_scratch():
    from paper_2607_11185_gb300 import vcs
    q, k, v, do = workloads.draw_dense(7, 256, 28, 4, 128, device="cuda")
    o = torch.empty_like(q)
    lse = torch.empty((28, 256), dtype=torch.float32, device="cuda")
    dcu = torch.tensor([0, 256], dtype=torch.int32, device="cuda")
    big = 100_000                                # tokens claimed: needs ~1.4 GB of scratch
    assert vcs.vcs_attn_bwd_workspace_size(1, big, big, 28, 4, 128) > vcs.NOALLOC_SCRATCH_BYTES
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    st = vcs.vcs_attn_bwd_noalloc(q, k, v, o, lse, do, dcu, 1, big, big, 28, 4, 128, 0.0, dq, dk, dv, None)
    assert st == 8                               # VCS_ERR_WORKSPACE, nothing launched
