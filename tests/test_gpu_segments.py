"""GPU segment builder vs the oracle: bit-exact on every output (Sec. 3.4, Algorithm 1)."""
import glob
import json
import os

import numpy as np
import pytest
import torch

from oracle import segments as oseg
from paper_2607_11185_gb300 import workloads
from tests.gpu_cases import random_steps, steps_to_device

pytestmark = pytest.mark.gpu

KEYS = ["cu_seqlens", "seg_traj", "tok_gather", "tok_src_step", "tok_pos", "tok_loss_mask"]


def run_and_compare(cu, img, txt, window, keep):
    from paper_2607_11185_gb300 import vcs
    ref = oseg.build(cu, img, txt, window, keep, method="closed")
    dcu, dimg, dtxt = steps_to_device(cu, img, txt)
    out = vcs.build_segments(dcu, dimg, dtxt, window, keep)
    assert out["num_segments"] == len(ref["cu_seqlens"]) - 1
    assert out["num_tokens"] == len(ref["tok_gather"])
    lens = np.diff(ref["cu_seqlens"])
    assert out["max_seqlen"] == (int(lens.max()) if len(lens) else 0)
    for k in KEYS:
        got = out[k].cpu().numpy()
        assert got.dtype == ref[k].dtype, k
        assert np.array_equal(got, ref[k]), k
    return out


@pytest.mark.parametrize("path", sorted(glob.glob(os.path.join(os.path.dirname(__file__), "golden", "seg_*.json"))))
def test_hand_worked(path):
    fx = json.load(open(path))
    run_and_compare(fx["cu_steps"], fx["step_img"], fx["step_txt"], fx["window"], fx["keep"])


@pytest.mark.parametrize("name", ["tiny", "traj8_w3", "traj32_w3", "traj16x50_w8"])
def test_workloads(name):
    w = workloads.WORKLOADS[name]
    cu, img, txt = workloads.draw_steps(w)
    run_and_compare(cu, img, txt, w.window, w.keep)


@pytest.mark.parametrize("layout", list(workloads.COMPARISON_LAYOUTS))
def test_comparison_layouts(layout):
    window, keep = workloads.COMPARISON_LAYOUTS[layout]
    cu, img, txt = workloads.draw_steps(workloads.WORKLOADS["traj32_w3"])
    run_and_compare(cu, img, txt, window, keep)


def test_paper_exact_long_horizon():
    # the paper's K = delta = 8 reading on the long-horizon draw
    cu, img, txt = workloads.draw_steps(workloads.WORKLOADS["traj16x50_w8"])
    run_and_compare(cu, img, txt, 8, 8)


@pytest.mark.parametrize("seed", range(10))
def test_random_with_empty_and_zero_counts(seed):
    cu, img, txt = random_steps(1000 + seed)
    rng = np.random.default_rng(seed)
    run_and_compare(cu, img, txt, int(rng.integers(1, 6)), int(rng.integers(0, 5)))


def test_many_trajectories_multi_chunk_scan():
    # more steps and trajectories than one scan chunk (4096 steps / 1024 trajectories)
    rng = np.random.default_rng(7)
    Ts = rng.integers(0, 12, size=1500)
    cu = np.concatenate([[0], np.cumsum(Ts)]).astype(np.int32)
    img = rng.integers(0, 50, size=int(cu[-1])).astype(np.int32)
    txt = rng.integers(0, 20, size=int(cu[-1])).astype(np.int32)
    assert cu[-1] > 4096
    run_and_compare(cu, img, txt, 3, 1)


def test_no_trajectories():
    from paper_2607_11185_gb300 import vcs
    cu = torch.zeros(1, dtype=torch.int32, device="cuda")
    e = torch.zeros(0, dtype=torch.int32, device="cuda")
    out = vcs.build_segments(cu, e, e, 3, 0)
    assert out["num_segments"] == 0 and out["num_tokens"] == 0
    assert out["cu_seqlens"].cpu().tolist() == [0]


def _raw_build(cu, img, txt, window, keep, seg_cap, tok_cap):
    from paper_2607_11185_gb300 import vcs
    dcu, dimg, dtxt = steps_to_device(cu, img, txt)
    nb = vcs.vcs_segments_workspace_size(len(cu) - 1, len(img))
    ws = torch.empty(nb, dtype=torch.uint8, device="cuda")
    sizes = torch.zeros(3, dtype=torch.int64, device="cuda")
    cs = torch.full((seg_cap + 1,), -7, dtype=torch.int32, device="cuda")
    toks = [torch.full((tok_cap,), -7, dtype=torch.int32, device="cuda") for _ in range(3)]
    st = vcs.vcs_build_segments(dcu, len(cu) - 1, len(img), dimg, dtxt, window, keep, seg_cap, tok_cap, cs, None,
                                toks[0], toks[1], toks[2], None, sizes, ws, nb)
    torch.cuda.synchronize()
    dev_status = int((sizes[2].item() >> 32) & 0xFFFFFFFF)
    return st, dev_status, cs, toks


def test_capacity_error_writes_nothing():
    fx = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "seg_tiny_w2.json")))
    st, dst, cs, toks = _raw_build(fx["cu_steps"], fx["step_img"], fx["step_txt"], 2, 0, 2, 1000)
    assert st == 0 and dst == 3               # VCS_ERR_CAPACITY (1216 tokens > 1000)
    assert torch.all(cs == -7) and all(torch.all(t == -7) for t in toks)


def test_inconsistent_cu_steps_reported():
    st, dst, _, _ = _raw_build([0, 3, 2, 4], [1, 2, 3, 4], [1, 1, 1, 1], 2, 0, 8, 64)
    assert st == 0 and dst == 6               # VCS_ERR_DEVICE_CHECK


def test_negative_counts_reported():
    st, dst, _, _ = _raw_build([0, 3], [1, -2, 3], [1, 1, 1], 2, 0, 8, 64)
    assert st == 0 and dst == 6


def test_host_argument_errors():
    from paper_2607_11185_gb300 import vcs
    dcu, dimg, dtxt = steps_to_device([0, 2], [1, 1], [1, 1])
    nb = vcs.vcs_segments_workspace_size(1, 2)
    ws = torch.empty(nb, dtype=torch.uint8, device="cuda")
    sizes = torch.zeros(3, dtype=torch.int64, device="cuda")
    assert vcs.vcs_plan_segments(dcu, 1, 2, dimg, dtxt, 0, 0, sizes, ws, nb) == 1      # window 0
    assert vcs.vcs_plan_segments(dcu, 1, 2, dimg, dtxt, 2, -1, sizes, ws, nb) == 1     # keep < 0
    assert vcs.vcs_plan_segments(dcu, 1, 2, dimg, dtxt, 2, 0, sizes, ws, nb - 1) == 8  # workspace
