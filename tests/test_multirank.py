"""The bench's multi-rank host logic on CPU (gloo, world size 2, no GPU).

Segments of different trajectories are independent, so ranks shard the units with no
data-path exchange: the job draws world x the workload's trajectories and each rank takes its
longest-processing-time share by attention cost, the job's time is the slowest rank's, its flops
and tokens the sum over ranks, and a decision that guards a collective is reduced over ranks so
that every rank takes the same branch.
"""
import contextlib
import dataclasses
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
        w = workloads.WORKLOADS["traj8_w3"]
        cu, img, txt, mine = bench.rank_batch(w, w.window, w.keep, rank, world)
        res["traj"] = mine
        res["steps"] = int(cu[-1])
        res["img_sum"] = int(img.sum())
        lens, _ = bench.layout_stats(cu, img, txt, w.window, w.keep)
        res["cost"] = float((lens * (lens + 1) // 2).sum())
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
    # the two shares are disjoint and together the job's 2 x 8 trajectories
    assert not set(r0["traj"]) & set(r1["traj"])
    assert sorted(r0["traj"] + r1["traj"]) == list(range(16))
    assert r0["steps"] > 0 and r1["steps"] > 0
    # longest processing time: the busier rank exceeds the mean by at most one trajectory's cost
    sys.path.insert(0, ROOT)
    import bench
    from paper_2607_11185_gb300 import workloads
    w = workloads.WORKLOADS["traj8_w3"]
    gcu, gimg, gtxt = workloads.draw_steps(dataclasses.replace(w, num_traj=16))
    lens, traj = bench.layout_stats(gcu, gimg, gtxt, w.window, w.keep)
    per = np.bincount(traj, weights=(lens * (lens + 1) // 2).astype(np.float64), minlength=16)
    assert r0["cost"] + r1["cost"] == pytest.approx(per.sum())
    assert max(r0["cost"], r1["cost"]) <= per.sum() / 2 + per.max()
    assert r1["ref_out"] == ""


def test_single_process_helpers_are_identity():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2607_11185_gb300 import workloads
    assert not dist.is_initialized()
    assert bench.max_over_ranks(3.25, torch.device("cpu")) == 3.25
    assert bench.sum_over_ranks(7.0, torch.device("cpu")) == 7.0
    # one rank runs exactly the workload's own draw
    w = workloads.WORKLOADS["traj8_w3"]
    cu, img, txt, mine = bench.rank_batch(w, w.window, w.keep, 0, 1)
    cu0, img0, txt0 = workloads.draw_steps(w)
    assert np.array_equal(cu, cu0) and np.array_equal(img, img0) and np.array_equal(txt, txt0)
    assert mine == list(range(w.num_traj))


def test_lpt_partition():
    sys.path.insert(0, ROOT)
    import bench
    # the textbook case: LPT puts 7 | 6 | 5 first, then 4 on the 5, 3 and 2 on the 6 and 7
    parts = bench.lpt_partition([7, 6, 5, 4, 3, 2], 3)
    loads = sorted(sum([7, 6, 5, 4, 3, 2][i] for i in p) for p in parts)
    assert loads == [9, 9, 9]
    assert sorted(i for p in parts for i in p) == list(range(6))
    # equal costs (the long-horizon workload): round robin, equal counts
    parts = bench.lpt_partition([1.0] * 16, 4)
    assert [len(p) for p in parts] == [4, 4, 4, 4]
    # more ranks than units: the extra ranks get nothing
    assert bench.lpt_partition([5, 1], 3) == [[0], [1], []]
    # random costs: disjoint cover, and the greedy bound max load <= mean + max cost
    rng = np.random.default_rng(3)
    for world in (2, 3, 5, 8):
        c = rng.integers(1, 1000, 40).astype(float).tolist()
        parts = bench.lpt_partition(c, world)
        assert sorted(i for p in parts for i in p) == list(range(40))
        loads = [sum(c[i] for i in p) for p in parts]
        assert max(loads) <= sum(c) / world + max(c)
