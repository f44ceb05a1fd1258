"""The bench's multi-rank host logic on CPU (gloo, world size 2, no GPU).

Segments of different trajectories are independent, so ranks shard the units with no
data-path exchange: each rank lays out its own batch of the workload, the job's time is the
slowest rank's, its flops and tokens the sum over ranks, and a decision that guards a
collective is reduced over ranks so that every rank takes the same branch.
"""
import contextlib
import io
import os
import socket
import sys
import types

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        from paper_2607_11185_gb300 import workloads
        dev = torch.device("cpu")
        res = {
            "max": bench.max_over_ranks(1.5 + rank, dev),
            "sum": bench.sum_over_ranks(10.0 * (rank + 1), dev),
            # a guard that only one rank would fail is seen as failed by both
            "guard": bench.sum_over_ranks(float(rank == 1), dev),
        }
        w = bench.rank_workload(workloads.WORKLOADS["traj8_w3"], rank)
        cu, img, txt = workloads.draw_steps(w)
        res["seed"] = w.seed
        res["steps"] = int(cu[-1])
        res["img_sum"] = int(img.sum())
        # the reference arm: only rank 0 runs and prints (the oracle is not run elsewhere)
        if rank == 1:
            buf = io.StringIO()
            args = types.SimpleNamespace(warmup=0, steps=1, gpus=world)
            with contextlib.redirect_stdout(buf):
                bench.run_reference(args, w, w.window, w.keep, rank, world)
            res["ref_out"] = buf.getvalue()
        torch.save(res, os.path.join(out, f"rank{rank}.pt"))
    finally:
        dist.destroy_process_group()


def test_two_ranks_gloo(tmp_path):
    port = _free_port()
    mp.spawn(_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True)
    r0 = torch.load(os.path.join(tmp_path, "rank0.pt"))
    r1 = torch.load(os.path.join(tmp_path, "rank1.pt"))
    for r in (r0, r1):
        assert r["max"] == 2.5
        assert r["sum"] == 30.0
        assert r["guard"] == 1.0
    assert r0["seed"] != r1["seed"]                       # each rank its own batch
    assert (r0["steps"], r0["img_sum"]) != (r1["steps"], r1["img_sum"])
    assert r1["ref_out"] == ""


def test_single_process_helpers_are_identity():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2607_11185_gb300 import workloads
    assert not dist.is_initialized()
    assert bench.max_over_ranks(3.25, torch.device("cpu")) == 3.25
    assert bench.sum_over_ranks(7.0, torch.device("cpu")) == 7.0
    w = workloads.WORKLOADS["traj8_w3"]
    assert bench.rank_workload(w, 0) is w
    w1 = bench.rank_workload(w, 1)
    assert w1.seed != w.seed and (w1.hq, w1.hkv, w1.d, w1.steps, w1.window) == (w.hq, w.hkv, w.d, w.steps, w.window)
    cu0, img0, txt0 = workloads.draw_steps(w)
    cu1, img1, txt1 = workloads.draw_steps(w1)
    assert len(cu0) == len(cu1)                          # same number of trajectories
    assert not (np.array_equal(cu0, cu1) and np.array_equal(txt0, txt1))
