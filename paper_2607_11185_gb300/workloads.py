"""Seeded synthetic workloads shaped like the paper's GUI trajectories.

This module holds NO arithmetic of the method: it only draws per-step token
counts and the dense bf16 tensors that both the CUDA path and the CPU oracle
consume.  It is the one module that the oracle side and the GPU side share.

Shapes follow the paper's rollouts (Sec. 4 training setup and App. D
hyperparameter table): at most 50 turns per episode, a 1280x800 screen per
step (a few thousand image tokens after patch merge), K=5 / K=8 windows.
The trajectories, screenshots and policy model of the paper are not
available; these draws stand in for them.

Draw order (fixed so that every consumer sees identical bytes):
  * step counts: ``numpy.random.default_rng(seed)``; per trajectory, in
    order: T, then img[1..T], then txt[1..T] (inclusive integer ranges);
  * Q_traj, K_traj, V_traj: one ``torch.Generator`` seeded with ``seed``,
    ``randn`` in fp32, rounded to bf16 (RNE), in that order, in row chunks;
  * dO (segment layout): a generator seeded with ``seed + 500``;
  * logit outliers (long-horizon stress workload only): a generator seeded
    with ``seed + 1000`` draws one uniform per (trajectory token, kv-head)
    row of K_traj; rows below the outlier fraction are multiplied by 8
    (exact in bf16).
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Tuple

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    num_traj: int
    steps: Tuple[int, int]      # inclusive range of T per trajectory
    img: Tuple[int, int]        # inclusive range of image tokens per screenshot
    txt: Tuple[int, int]        # inclusive range of text tokens per step
    window: int                 # delta (new screenshots per segment)
    keep: int                   # K (screenshots retained across a prune)
    hq: int
    hkv: int
    d: int
    seed: int
    outlier_frac: float = 0.0


WORKLOADS: Dict[str, Workload] = {
    # one trajectory, whole problem fits the oracle in seconds
    "tiny": Workload("tiny", 1, (4, 4), (256, 256), (32, 32), 2, 0, 2, 1, 64, 1),
    # 8 trajectories, 5-15 steps, fixed 1,024-token screenshots
    "traj8_w3": Workload("traj8_w3", 8, (5, 15), (1024, 1024), (64, 256), 3, 0, 28, 4, 128, 2),
    # 32 trajectories, 10-50 steps, 1080p-like 1,500-2,700-token screenshots
    "traj32_w3": Workload("traj32_w3", 32, (10, 50), (1500, 2700), (64, 512), 3, 0, 28, 4, 128, 3),
    # long-horizon stress: 16 x 50 steps, 2,700 + 512 tokens/step, W=8, outliers
    "traj16x50_w8": Workload("traj16x50_w8", 16, (50, 50), (2700, 2700), (512, 512), 8, 0, 40, 8, 128, 5,
                             outlier_frac=0.05),
}

# The same draw laid out several ways through the same kernels: (window,
# keep).  "stepwise" (one item per turn with the prior history as text)
# coincides with a window of one screenshot; the paper's own K = delta
# settings are added so that the layouts differ, its ScienceBoard setting
# K = 8, delta = 5 (App. C.2) as a K != delta case, and K = delta = 8 as the
# paper-exact reading of the long-horizon workload's window.
COMPARISON_LAYOUTS: Dict[str, Tuple[int, int]] = {
    "stepwise": (1, 0),
    "w5": (5, 0),
    "paper_k1": (1, 1),
    "paper_k5": (5, 5),
    "paper_k8_d5": (5, 8),
    "paper_k8": (8, 8),
}


def draw_steps(w: Workload):
    """Per-step token counts: (cu_steps[int32 B+1], step_img[int32 N], step_txt[int32 N])."""
    rng = np.random.default_rng(w.seed)
    imgs, txts, cu = [], [], [0]
    for _ in range(w.num_traj):
        t = int(rng.integers(w.steps[0], w.steps[1], endpoint=True))
        imgs.append(rng.integers(w.img[0], w.img[1], size=t, endpoint=True))
        txts.append(rng.integers(w.txt[0], w.txt[1], size=t, endpoint=True))
        cu.append(cu[-1] + t)
    step_img = np.concatenate(imgs).astype(np.int32) if imgs else np.zeros(0, np.int32)
    step_txt = np.concatenate(txts).astype(np.int32) if txts else np.zeros(0, np.int32)
    return np.asarray(cu, dtype=np.int32), step_img, step_txt


def trajectory_tokens(step_img: np.ndarray, step_txt: np.ndarray) -> int:
    """Length of the concatenated trajectory token buffer."""
    return int(step_img.astype(np.int64).sum() + step_txt.astype(np.int64).sum())


def _randn_bf16(gen: torch.Generator, shape, device, chunk_rows: int = 1 << 16) -> torch.Tensor:
    out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    rows = shape[0]
    flat = out.view(rows, -1)
    for r0 in range(0, rows, chunk_rows):
        r1 = min(rows, r0 + chunk_rows)
        flat[r0:r1].copy_(torch.randn((r1 - r0, flat.shape[1]), generator=gen, device=device,
                                      dtype=torch.float32))
    return out


def draw_traj_qkv(w: Workload, traj_tokens: int, device="cpu"):
    """Q_traj [Ntraj, Hq, d], K_traj / V_traj [Ntraj, Hkv, d], bf16 N(0,1)."""
    gen = torch.Generator(device=device)
    gen.manual_seed(w.seed)
    q = _randn_bf16(gen, (traj_tokens, w.hq, w.d), device)
    k = _randn_bf16(gen, (traj_tokens, w.hkv, w.d), device)
    v = _randn_bf16(gen, (traj_tokens, w.hkv, w.d), device)
    if w.outlier_frac > 0:
        g2 = torch.Generator(device=device)
        g2.manual_seed(w.seed + 1000)
        sel = torch.rand((traj_tokens, w.hkv), generator=g2, device=device) < w.outlier_frac
        k.mul_(torch.where(sel, 8.0, 1.0).to(torch.bfloat16).unsqueeze(-1))
    return q, k, v


def draw_dout(w: Workload, num_tokens: int, device="cpu") -> torch.Tensor:
    """dO [Ntok, Hq, d] bf16 N(0,1) in segment layout."""
    gen = torch.Generator(device=device)
    gen.manual_seed(w.seed + 500)
    return _randn_bf16(gen, (num_tokens, w.hq, w.d), device)


def draw_dense(seed: int, n: int, hq: int, hkv: int, d: int, device="cpu", scale: float = 1.0):
    """Q [n,hq,d], K/V [n,hkv,d], dO [n,hq,d] bf16 for direct attention cases."""
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    q = _randn_bf16(gen, (n, hq, d), device)
    k = _randn_bf16(gen, (n, hkv, d), device)
    v = _randn_bf16(gen, (n, hkv, d), device)
    do = _randn_bf16(gen, (n, hq, d), device)
    if scale != 1.0:
        q = (q.float() * scale).to(torch.bfloat16)
    return q, k, v, do
