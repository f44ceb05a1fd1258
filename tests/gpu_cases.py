"""Shared seeded cases for the GPU parity tests (inputs only; no method arithmetic)."""
import numpy as np
import torch

from paper_2607_11185_gb300 import workloads


def steps_to_device(cu, img, txt, device="cuda"):
    return (torch.from_numpy(np.asarray(cu, np.int32)).to(device),
            torch.from_numpy(np.asarray(img, np.int32)).to(device),
            torch.from_numpy(np.asarray(txt, np.int32)).to(device))


def random_steps(seed, max_traj=6, max_T=30, max_img=40, max_txt=9):
    rng = np.random.default_rng(seed)
    B = int(rng.integers(0, max_traj + 1))
    Ts = rng.integers(0, max_T + 1, size=B)
    cu = np.concatenate([[0], np.cumsum(Ts)]).astype(np.int32)
    img = rng.integers(0, max_img + 1, size=int(cu[-1])).astype(np.int32)
    txt = rng.integers(0, max_txt + 1, size=int(cu[-1])).astype(np.int32)
    return cu, img, txt


def cu_from_lengths(lengths):
    return np.concatenate([[0], np.cumsum(lengths)]).astype(np.int32)


def sample_rows(L, rng, n_random=4):
    """Rows of a segment worth checking: ends, tile edges, a few random ones."""
    cand = {0, L - 1}
    for e in (127, 128, 129, 255, 256, 257):
        if e < L:
            cand.add(e)
    cand.update(int(x) for x in rng.integers(0, L, size=n_random))
    return sorted(cand)


def bench_chunks(w, lay, num_traj):
    """The chunks the benchmark launches a workload in, as (first segment, end segment) pairs of
    the oracle's layout: the full-size cases run exactly the launches the benchmark times."""
    import bench
    lens = np.diff(np.asarray(lay["cu_seqlens"], np.int64))
    traj = np.asarray(lay["seg_traj"], np.int64)
    chunks = bench.make_chunks(lens, traj, num_traj, w.hq, w.hkv, w.d)
    return [(int(np.searchsorted(traj, b0)), int(np.searchsorted(traj, b1))) for b0, b1 in chunks]


WORKLOADS = workloads.WORKLOADS
