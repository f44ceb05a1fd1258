"""Benchmark of the Visual Context Segmentation hot path on one GB300.

One step = the whole hot path over one batch of synthetic trajectories:
segment layout (vcs_build_segments), Q/K/V gather (vcs_gather), causal
segmented attention forward (vcs_attn_fwd) and backward (vcs_attn_bwd).
Trajectories are processed in chunks that fit HBM; every chunk's work is
inside the timed region.

Default workload: 16 trajectories x 50 steps, 2,700 screenshot + 512
response tokens per step, window W=8, 40 query / 8 key-value heads, head_dim
128, bf16, 5% of key rows scaled by 8 (the long-horizon stress workload).

The printed value is credited attention TFLOP/s: 12 * d * Hq * sum_s L_s(L_s+1)/2
(forward 4, backward 8; the backward's recomputation of S is not credited)
divided by the device time of the whole step.

--impl reference times the CPU oracle (fp64 numpy) on a bounded sample of the
same workload instead (the oracle is the only reference implementation of
this path).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2607_11185_gb300 import workloads  # noqa: E402

METRIC = "segmented attn fwd+bwd TFLOP/s & % BF16 peak; segment tokens/s; vs CPU oracle"
CHUNK_BYTES = 130 << 30   # per-chunk working set budget on the device (fewer, larger launches)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["bf16_tflops"]), float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), \
            float(p["hbm_gbs"]), "measured"
    except Exception:
        return 1900.0, 1700.0, 6800.0, "fallback"


BACKWARD_SOURCES = ("attn_bwd.cu", "sm100.cuh", "internal.h", "api.cu")


def backward_code_hash() -> str:
    """First 16 hex digits of the SHA-256 of the sources the backward's traffic depends on (its
    kernels, the PTX wrappers, the workspace layout and argument set-up of the C ABI) with
    comments, trailing blanks and blank lines removed: any change to the code changes it, a
    change to a comment does not."""
    return code_hash(b"".join(open(os.path.join(ROOT, "paper_2607_11185_gb300", "csrc", f), "rb").read()
                              for f in BACKWARD_SOURCES))


def strip_comments(src: bytes) -> bytes:
    """C/C++ source without its comments; string and character literals are kept whole (a
    '//' inside a string is not a comment)."""
    import re
    tok = re.compile(rb'"(?:\\.|[^"\\\n])*"|\'(?:\\.|[^\'\\\n])*\'|/\*.*?\*/|//[^\n]*', re.S)
    return tok.sub(lambda m: m.group(0) if m.group(0)[:1] in (b'"', b"'") else b"", src)


def code_hash(src: bytes) -> str:
    import hashlib
    lines = [ln.rstrip() for ln in strip_comments(src).split(b"\n")]
    return hashlib.sha256(b"\n".join(ln for ln in lines if ln)).hexdigest()[:16]


def measured_traffic(trajectories, profile="attn_traffic_traj16x50_w8_1traj.md"):
    """DRAM bytes per vcs_attn_bwd call of `trajectories` long-horizon trajectories, from the
    committed ncu capture of a one-trajectory small case (every trajectory of that workload has the
    same segments, so the bytes scale with the trajectory count), or None when the backward's code
    changed since those counters were taken."""
    try:
        text = open(os.path.join(ROOT, "profiles", profile)).read()
        vals = dict(line.split(": ", 1) for line in text.splitlines() if ": " in line and " " not in line.split(": ")[0])
        if backward_code_hash() != vals["code_sha256_16"].strip():
            return None
        return int(vals["traffic_bytes_per_trajectory"]) * int(trajectories)
    except Exception:
        return None


def layout_stats(cu_steps, img, txt, window, keep):
    """Host-side sizes of the layout from the closed form (input preparation only)."""
    seg_lens, seg_traj = [], []
    for b in range(len(cu_steps) - 1):
        g0, g1 = int(cu_steps[b]), int(cu_steps[b + 1])
        T = g1 - g0
        if T == 0:
            continue
        ti, tx = img[g0:g1].astype(np.int64), txt[g0:g1].astype(np.int64)
        s = 1
        j = 0
        while s <= T:
            e = min(keep + window, T) if j == 0 else min(s + window - 1, T)
            a = max(1, s - keep)
            seg_lens.append(int(tx[: a - 1].sum() + ti[a - 1: e].sum() + tx[a - 1: e].sum()))
            seg_traj.append(b)
            s = e + 1
            j += 1
    return np.asarray(seg_lens, np.int64), np.asarray(seg_traj, np.int64)


def credited_flops(seg_lens, hq, d):
    pairs = (seg_lens * (seg_lens + 1) // 2).sum()
    return 12.0 * d * hq * float(pairs), 4.0 * d * hq * float(pairs), 8.0 * d * hq * float(pairs)


class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self):
        self.rows = []
        self.proc = None

    def start(self):
        try:
            idx = os.environ.get("CUDA_VISIBLE_DEVICES", "0").split(",")[0] or "0"
            self.proc = subprocess.Popen(["nvidia-smi", "-i", idx, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.th = threading.Thread(target=self._read, daemon=True)
            self.th.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 8:
                self.rows.append(parts)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm = [float(r[0]) for r in self.rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in self.rows for i in range(4) if r[4 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.rows)}


def make_chunks(seg_lens, seg_traj, num_traj, hq, hkv, d):
    """Trajectory ranges whose per-chunk device buffers fit CHUNK_BYTES."""
    per_tok = (2 * hq * d * 2 + 2 * hkv * d * 2) * 2 + hq * d * 4 + hq * 8 + 16
    chunks, b0, acc = [], 0, 0
    tok_per_traj = np.bincount(seg_traj, weights=seg_lens, minlength=num_traj).astype(np.int64)
    for b in range(num_traj):
        t = int(tok_per_traj[b]) * per_tok
        if acc > 0 and acc + t > CHUNK_BYTES:
            chunks.append((b0, b))
            b0, acc = b, 0
        acc += t
    chunks.append((b0, num_traj))
    return chunks


class Path:
    """Device-resident inputs and per-chunk buffers for the hot path."""

    def __init__(self, w: workloads.Workload, window: int, keep: int, device, steps=None):
        from paper_2607_11185_gb300 import vcs
        self.vcs = vcs
        self.w, self.window, self.keep, self.dev = w, window, keep, device
        cu, img, txt = workloads.draw_steps(w) if steps is None else steps
        self.cu, self.img, self.txt = cu, img, txt
        self.seg_lens, self.seg_traj = layout_stats(cu, img, txt, window, keep)
        self.num_tokens = int(self.seg_lens.sum())
        self.ntraj_tok = workloads.trajectory_tokens(img, txt)
        step_off = np.concatenate([[0], np.cumsum(img.astype(np.int64) + txt)])
        self.traj_tok_off = step_off[cu]
        # resident inputs: step counts, trajectory Q/K/V, upstream gradient dO (segment layout)
        self.q_traj, self.k_traj, self.v_traj = workloads.draw_traj_qkv(w, self.ntraj_tok, device=device)
        self.dout = workloads.draw_dout(w, self.num_tokens, device=device)
        self.chunks = make_chunks(self.seg_lens, self.seg_traj, len(cu) - 1, w.hq, w.hkv, w.d)
        self.chunk_in = []
        seg_cum = np.concatenate([[0], np.cumsum(self.seg_lens)])
        max_tok = max_seg = max_steps = 0
        for b0, b1 in self.chunks:
            s0 = int(np.searchsorted(self.seg_traj, b0))
            s1 = int(np.searchsorted(self.seg_traj, b1))
            g0, g1 = int(cu[b0]), int(cu[b1])
            ci = dict(b0=b0, b1=b1, s0=s0, s1=s1, tok0=int(seg_cum[s0]), tok1=int(seg_cum[s1]),
                      cu=torch.from_numpy((cu[b0:b1 + 1] - cu[b0]).astype(np.int32)).to(device),
                      img=torch.from_numpy(img[g0:g1].copy()).to(device),
                      txt=torch.from_numpy(txt[g0:g1].copy()).to(device),
                      ttok0=int(self.traj_tok_off[b0]), ttok1=int(self.traj_tok_off[b1]),
                      nsteps=g1 - g0, max_seqlen=int(self.seg_lens[s0:s1].max()) if s1 > s0 else 0)
            self.chunk_in.append(ci)
            max_tok = max(max_tok, ci["tok1"] - ci["tok0"])
            max_seg = max(max_seg, s1 - s0)
            max_steps = max(max_steps, g1 - g0)
        hq, hkv, d = w.hq, w.hkv, w.d
        self.max_tok, self.max_seg = max_tok, max_seg
        T = lambda *s, dt=torch.bfloat16: torch.empty(s, dtype=dt, device=device)  # noqa: E731
        self.cu_seqlens = T(max_seg + 1, dt=torch.int32)
        self.tok_gather = T(max_tok, dt=torch.int32)
        self.tok_src = T(max_tok, dt=torch.int32)
        self.tok_pos = T(max_tok, dt=torch.int32)
        self.tok_mask = T(max_tok, dt=torch.uint8)
        self.sizes = torch.zeros(3, dtype=torch.int64, device=device)
        # each chunk's builder writes its layout sizes to a slot of its own, read back and checked
        # against the host's closed form once the timed steps are done (verify_sizes): the step
        # itself never waits for the device
        self.sizes_all = torch.zeros((len(self.chunks), 3), dtype=torch.int64, device=device)
        self.seg_ws_bytes = vcs.vcs_segments_workspace_size(max(b1 - b0 for b0, b1 in self.chunks), max_steps)
        self.seg_ws = T(self.seg_ws_bytes, dt=torch.uint8)
        self.q, self.k, self.v = T(max_tok, hq, d), T(max_tok, hkv, d), T(max_tok, hkv, d)
        self.o, self.lse = T(max_tok, hq, d), T(hq, max_tok, dt=torch.float32)
        self.dq, self.dk, self.dv = T(max_tok, hq, d), T(max_tok, hkv, d), T(max_tok, hkv, d)
        self.gstatus = torch.zeros(1, dtype=torch.int32, device=device)
        mxl = int(self.seg_lens.max())
        self.fwd_ws_bytes = vcs.vcs_attn_fwd_workspace_size(max_seg, max_tok, mxl, hq, hkv, d)
        self.bwd_ws_bytes = vcs.vcs_attn_bwd_workspace_size(max_seg, max_tok, mxl, hq, hkv, d)
        self.fwd_ws = T(self.fwd_ws_bytes, dt=torch.uint8)
        self.bwd_ws = T(self.bwd_ws_bytes, dt=torch.uint8)
        self.launches_per_step = 0

    def step(self, tstream, ev=None, before_chunk=None, after_chunk=None, before_bwd=None, grads=None):
        """One pass of the hot path over all chunks; optional per-chunk events appended to ev and
        hooks called before a chunk's first launch, before its backward and after its last one;
        grads(i) gives chunk i's (dq, dk, dv) output buffers (default: the path's own)."""
        vcs, w = self.vcs, self.w
        stream = tstream.cuda_stream
        hq, hkv, d = w.hq, w.hkv, w.d
        launches = 0
        for i, ci in enumerate(self.chunk_in):
            if before_chunk is not None:
                before_chunk(i)
            nseg, ntok = ci["s1"] - ci["s0"], ci["tok1"] - ci["tok0"]
            evs = [torch.cuda.Event(enable_timing=True) for _ in range(6)] if ev is not None else None
            if evs:
                evs[0].record(tstream)
            st = vcs.vcs_build_segments(ci["cu"], ci["b1"] - ci["b0"], ci["nsteps"], ci["img"], ci["txt"],
                                        self.window, self.keep, self.max_seg, self.max_tok, self.cu_seqlens, None,
                                        self.tok_gather, self.tok_src, self.tok_pos, self.tok_mask,
                                        self.sizes_all[i], self.seg_ws, self.seg_ws_bytes, stream)
            launches += 5
            assert st == 0, vcs.vcs_status_string(st)
            if evs:
                evs[1].record(tstream)
            # the attention launches take the layout sizes the host computed from the closed form
            # (the trajectories' step counts are the host's own input); the builder's sizes are
            # checked against them after the timed steps (verify_sizes)
            qt = self.q_traj[ci["ttok0"]:ci["ttok1"]]
            kt = self.k_traj[ci["ttok0"]:ci["ttok1"]]
            vt = self.v_traj[ci["ttok0"]:ci["ttok1"]]
            if evs:
                evs[2].record(tstream)
            st = vcs.vcs_gather(qt, kt, vt, ci["ttok1"] - ci["ttok0"], self.tok_gather, ntok, hq, hkv, d, self.q,
                                self.k, self.v, self.gstatus, stream)
            launches += 3
            assert st == 0
            if evs:
                evs[3].record(tstream)
            st = vcs.vcs_attn_fwd(self.q, self.k, self.v, self.cu_seqlens, nseg, ntok, ci["max_seqlen"], hq, hkv,
                                  d, 0.0, self.o, self.lse, self.fwd_ws, self.fwd_ws_bytes, stream)
            launches += 3  # the work-unit scan and fill, then the attention kernel
            assert st == 0
            if evs:
                evs[4].record(tstream)
            dout = self.dout[ci["tok0"]:ci["tok1"]]
            if before_bwd is not None:
                before_bwd(i)
            dq, dk, dv = (self.dq, self.dk, self.dv) if grads is None else grads(i)
            st = vcs.vcs_attn_bwd(self.q, self.k, self.v, self.o, self.lse, dout, self.cu_seqlens, nseg, ntok,
                                  ci["max_seqlen"], hq, hkv, d, 0.0, dq, dk, dv, self.bwd_ws, self.bwd_ws_bytes,
                                  stream)
            launches += 3
            assert st == 0
            if evs:
                evs[5].record(tstream)
                ev.append((evs, ci))
            if after_chunk is not None:
                after_chunk(i)
        self.launches_per_step = launches

    def verify_sizes(self):
        """The builder's layout sizes of every chunk (from the last step) equal the host's."""
        sz = self.sizes_all.cpu()
        for i, ci in enumerate(self.chunk_in):
            assert int(sz[i, 0]) == ci["s1"] - ci["s0"] and int(sz[i, 1]) == ci["tok1"] - ci["tok0"], (i, sz[i])
            assert int(sz[i, 2]) & 0xffffffff == ci["max_seqlen"] and (int(sz[i, 2]) >> 32) == 0, (i, sz[i])

    def device_status(self):
        return (int(self.gstatus.item()), int(self.fwd_ws[:4].view(torch.int32).item()),
                int(self.bwd_ws[:4].view(torch.int32).item()))


def oracle_sample(w, window, keep):
    """The CPU oracle on a bounded sample: the builder on the whole batch, plus attention
    forward + backward of one query head over the shortest segment, on all host cores.

    Returns the `cpu_baseline` fields: credited TFLOP/s of the sample, the causal
    (query, key) pairs per second of its attention part, the seconds the whole workload
    would take at that rate (extrapolated, not run), and a one-core figure."""
    from oracle import attention as oatt
    from oracle import segments as oseg
    cu, img, txt = workloads.draw_steps(w)
    t0 = time.perf_counter()
    lay = oseg.build(cu, img, txt, window, keep, method="closed")
    t_build = time.perf_counter() - t0
    lens = np.diff(lay["cu_seqlens"]).astype(np.int64)
    s = int(np.argmin(lens))
    L = int(lens[s])
    gen = torch.Generator().manual_seed(w.seed + 77)
    q = torch.randn((L, 1, w.d), generator=gen).to(torch.bfloat16)
    k = torch.randn((L, 1, w.d), generator=gen).to(torch.bfloat16)
    v = torch.randn((L, 1, w.d), generator=gen).to(torch.bfloat16)
    do = torch.randn((L, 1, w.d), generator=gen).to(torch.bfloat16)
    t0 = time.perf_counter()
    oatt.attn_bwd(q, k, v, do, [0, L])          # computes the forward too
    t_attn = time.perf_counter() - t0
    flops = 12.0 * w.d * 1 * L * (L + 1) / 2
    secs = t_build + t_attn
    tflops = flops / secs / 1e12
    job_flops = 12.0 * w.d * w.hq * float((lens * (lens + 1) // 2).sum())
    sample = (f"oracle builder over all {len(cu) - 1} trajectories ({t_build:.2f} s) + fp64 attention fwd+bwd of "
              f"1 query head over the shortest segment (L={L}, {t_attn:.2f} s)")
    return {"value": tflops, "unit": "TFLOP/s", "cores": os.cpu_count(), "kind": "oracle", "sample": sample,
            "seconds": secs, "pairs_per_s": L * (L + 1) / 2 / t_attn,
            "extrapolated_full_workload_s": job_flops / (tflops * 1e12),
            "one_core": oracle_one_core(w.d, min(L, 4096), w.seed + 78)}


def oracle_one_core(d: int, rows: int, seed: int):
    """The oracle's attention fwd+bwd of one query head over a `rows`-token segment with the
    BLAS held to one thread.  It runs in a fresh interpreter so that the thread limit is set
    before numpy loads its BLAS (and no state is shared with this process's CUDA context)."""
    code = (
        "import json, sys, time\n"
        "import numpy as np\n"
        f"sys.path.insert(0, {ROOT!r})\n"
        "from oracle import attention as oatt\n"
        f"rng = np.random.default_rng({seed})\n"
        f"x = [rng.standard_normal(({rows}, 1, {d})) for _ in range(4)]\n"
        "t0 = time.perf_counter()\n"
        f"oatt.attn_bwd(x[0], x[1], x[2], x[3], [0, {rows}])\n"
        "print(json.dumps({'s': time.perf_counter() - t0}))\n")
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
    try:
        out = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                             timeout=300, cwd=ROOT)
        secs = json.loads(out.stdout.strip().splitlines()[-1])["s"]
    except Exception as e:  # a reported figure, not a gate: say why it is missing
        return {"value": None, "error": f"one-core oracle run failed: {e}"[:200]}
    flops = 12.0 * d * rows * (rows + 1) / 2
    return {"value": flops / secs / 1e12, "unit": "TFLOP/s", "cores": 1, "seconds": secs,
            "pairs_per_s": rows * (rows + 1) / 2 / secs,
            "sample": f"fp64 attention fwd+bwd of 1 query head over a {rows}-token segment, BLAS on one thread"}


def lpt_partition(costs, world: int):
    """Longest-processing-time assignment of units to ranks: the units in order of decreasing
    cost, each to the rank with the least cost so far (the lowest rank on ties).  Returns each
    rank's unit indices in increasing order."""
    order = sorted(range(len(costs)), key=lambda i: (-costs[i], i))
    load = [0.0] * world
    parts = [[] for _ in range(world)]
    for i in order:
        r = min(range(world), key=lambda j: (load[j], j))
        parts[r].append(i)
        load[r] += costs[i]
    return [sorted(p) for p in parts]


def rank_batch(w, window: int, keep: int, rank: int, world: int):
    """The trajectories rank `rank` runs, as (cu_steps, step_img, step_txt, global indices).

    Segments of different trajectories are independent, so ranks shard trajectories with no
    data-path exchange.  The job draws the workload's distribution for world x its trajectory
    count (the first w.num_traj trajectories are exactly the one-GPU batch) and splits them by
    longest processing time on each trajectory's attention cost, the sum over its segments of
    L(L+1)/2 causal pairs: weak scaling, each rank getting about one workload's worth."""
    import dataclasses
    cu, img, txt = workloads.draw_steps(dataclasses.replace(w, num_traj=w.num_traj * world))
    ntraj = len(cu) - 1
    if world == 1:
        return cu, img, txt, list(range(ntraj))
    seg_lens, seg_traj = layout_stats(cu, img, txt, window, keep)
    cost = np.zeros(ntraj)
    np.add.at(cost, seg_traj, (seg_lens * (seg_lens + 1) // 2).astype(np.float64))
    mine = lpt_partition(cost.tolist(), world)[rank]
    steps = [(int(cu[b]), int(cu[b + 1])) for b in mine]
    rcu = np.concatenate([[0], np.cumsum([g1 - g0 for g0, g1 in steps])]).astype(np.int32)
    rimg = np.concatenate([img[g0:g1] for g0, g1 in steps] or [np.zeros(0, np.int32)]).astype(np.int32)
    rtxt = np.concatenate([txt[g0:g1] for g0, g1 in steps] or [np.zeros(0, np.int32)]).astype(np.int32)
    return rcu, rimg, rtxt, mine


def max_over_ranks(value: float, device) -> float:
    """The slowest rank's time (the job's time), over the default process group if there is one."""
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() == 1:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value: float, device) -> float:
    """The job's total of a per-rank quantity (flops, tokens), over the default process group."""
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() == 1:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def line_config(w, window, keep, cu, img, txt, world):
    """The workload a line was measured on (the same for both arms): sizes of the layout this rank
    runs, from the closed form on the host."""
    seg_lens, seg_traj = layout_stats(cu, img, txt, window, keep)
    chunks = make_chunks(seg_lens, seg_traj, len(cu) - 1, w.hq, w.hkv, w.d)
    return {"workload": w.name, "window": window, "keep": keep, "num_traj": w.num_traj, "hq": w.hq, "hkv": w.hkv,
            "d": w.d, "segments": int(len(seg_lens)), "segment_tokens": int(seg_lens.sum()),
            "max_seqlen": int(seg_lens.max()) if len(seg_lens) else 0, "chunks": len(chunks),
            "l2": "inputs larger than L2 (trajectory Q/K/V and dO resident, > 129 MB)",
            **({"sharding": f"{world * w.num_traj} trajectories over {world} ranks by longest processing "
                            f"time on sum L(L+1)/2; segments, tokens and chunks above are rank 0's"}
               if world > 1 else {})}


def run_reference(args, w, window, keep, rank, world):
    if rank != 0:
        return
    vals = []
    for i in range(args.warmup + args.steps):
        r = oracle_sample(w, window, keep)
        if i >= args.warmup:
            vals.append(r)
    v = statistics.median(x["value"] for x in vals)
    secs = statistics.median(x["seconds"] for x in vals)
    cpu = dict(vals[-1], value=v, seconds=secs)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "TFLOP/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": secs * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": line_config(w, window, keep, *rank_batch(w, window, keep, rank, world)[:3], world),
            "cpu_baseline": cpu,
            "e2e": {"value": v, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="traj16x50_w8", choices=list(workloads.WORKLOADS))
    ap.add_argument("--layout", default=None, choices=[None, *workloads.COMPARISON_LAYOUTS],
                    help="lay the workload's draw out as one of the comparison layouts (window, keep)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-next-rows", action="store_true", help="skip the stream-field / loss kernel timings")
    ap.add_argument("--no-fused", action="store_true", help="skip the gathered-attention (fused gather) timing")
    ap.add_argument("--no-reuse", action="store_true", help="skip the prefix-reuse forward timing")
    ap.add_argument("--no-hbm-kernels", action="store_true", help="skip the builder / gather timings")
    ap.add_argument("--builder-stress-traj", type=int, default=4096,
                    help="trajectories of the builder stress batch (a smaller one for profiler captures)")
    ap.add_argument("--num-traj", type=int, default=None,
                    help="run the first NUM_TRAJ trajectories of the workload's draw instead of all (a small case "
                         "of the same segment shapes, for profiler captures); the line's config says so")
    args = ap.parse_args()

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    w = workloads.WORKLOADS[args.workload]
    if args.num_traj is not None:
        import dataclasses
        w = dataclasses.replace(w, num_traj=args.num_traj)
    window, keep = w.window, w.keep
    if args.layout is not None:
        window, keep = workloads.COMPARISON_LAYOUTS[args.layout]

    if args.impl == "reference":
        run_reference(args, w, window, keep, rank, world)
        return

    if world > 1:
        import torch.distributed as dist
        local = int(os.environ.get("LOCAL_RANK", rank))
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", torch.cuda.current_device())

    # the CPU baseline runs before any GPU work so that no process pool or
    # thread state is shared with the CUDA context
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = oracle_sample(w, window, keep)

    path = Path(w, window, keep, dev, steps=rank_batch(w, window, keep, rank, world)[:3])
    stream = torch.cuda.current_stream()
    flops, f_fwd, f_bwd = credited_flops(path.seg_lens, w.hq, w.d)
    for _ in range(args.warmup):
        path.step(stream)
    torch.cuda.synchronize()
    st = path.device_status()
    assert st == (0, 0, 0), f"device status {st}"
    path.verify_sizes()

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    clocks = ClockSampler()
    clocks.start()
    ev = []
    barrier()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        path.step(stream, ev)
    t1.record(stream)
    barrier()
    ck = clocks.stop()
    path.verify_sizes()
    ms = t0.elapsed_time(t1) / args.steps
    ms = max_over_ranks(ms, dev)
    # per chunk: [0]-[1] build, (host reads the sizes), [2]-[3] gather, [3]-[4] fwd, [4]-[5] bwd
    build_ms = sum(e[0].elapsed_time(e[1]) for e, _ in ev) / args.steps
    gather_ms = sum(e[2].elapsed_time(e[3]) for e, _ in ev) / args.steps
    fwd_ms = sum(e[3].elapsed_time(e[4]) for e, _ in ev) / args.steps
    bwd_ms = sum(e[4].elapsed_time(e[5]) for e, _ in ev) / args.steps
    bwd_launch_ms = statistics.mean(e[4].elapsed_time(e[5]) for e, _ in ev)
    gather_bytes = path.num_tokens * 2 * (w.hq + 2 * w.hkv) * w.d * 2     # rows read once + written once
    bwd_launch_flops = f_bwd / len(path.chunk_in)

    job_flops = sum_over_ranks(flops, dev)               # every rank's own batch
    job_tokens = sum_over_ranks(float(path.num_tokens), dev)
    value = job_flops / (ms / 1e3) / 1e12
    burst, sustained, hbm, src = peaks()

    # end to end through the public API with host buffers: pinned host -> device copies of the
    # step's inputs and a device -> host read of its result, inside the timed region
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(path, args, job_flops, stream)

    next_rows = None if args.no_next_rows else run_next_rows(path, stream, hbm)
    fused = None if args.no_fused else run_fused(path, stream)
    reuse = None if args.no_reuse else run_reuse(path, stream)
    hbm_kernels = None if args.no_hbm_kernels else run_hbm_kernels(path, stream, hbm, args.builder_stress_traj)

    ach_bwd = bwd_launch_flops / (bwd_launch_ms / 1e3) / 1e12
    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": line_config(w, window, keep, path.cu, path.img, path.txt, world),
        "attn_tflop_credited": flops / 1e12,
        "builder_ms": build_ms, "gather_ms": gather_ms, "gather_gbs": gather_bytes / (gather_ms / 1e3) / 1e9,
        "attn_fwd_ms": fwd_ms, "attn_bwd_ms": bwd_ms,
        "attn_fwd_tflops": f_fwd / (fwd_ms / 1e3) / 1e12, "attn_bwd_tflops": f_bwd / (bwd_ms / 1e3) / 1e12,
        "attn_fwdbwd_tflops": flops / ((fwd_ms + bwd_ms) / 1e3) / 1e12,
        # the job's rate against the job's peak: N GPUs' worth
        "frac_of_bf16_burst": value / (world * burst), "frac_of_bf16_sustained": value / (world * sustained),
        "flash_convention_tflops": value * 14.0 / 12.0,
        "segment_tokens_per_s": job_tokens / (ms / 1e3),
        "roofline": {"bound": "tensor", "kernel": "vcs_attn_bwd (bwd_pre + bwd_main + bwd_dq_cvt)",
                     "achieved": ach_bwd, "peak": sustained, "unit": "TFLOP/s", "frac": ach_bwd / sustained,
                     "peak_source": f"{src} bf16 sustained",
                     "traffic": measured_traffic(path.chunk_in[0]["b1"] - path.chunk_in[0]["b0"])
                     if w.name == "traj16x50_w8" and (window, keep) == (w.window, w.keep) else None,
                     "traffic_source": "ncu DRAM bytes of a one-trajectory small case x the trajectories of a "
                                       "launch (profiles/attn_traffic_traj16x50_w8_1traj.md)"},
        "cpu_baseline": cpu,
        "e2e": e2e,
        "next_rows": next_rows,
        "fused_gather": fused,
        "prefix_reuse": reuse,
        "hbm_kernels": hbm_kernels,
        "gpu_launches": int(sum_over_ranks(float(path.launches_per_step * args.steps), dev)),  # every rank's
        "clocks": ck,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def run_next_rows(path, stream, hbm_gbs):
    """The stream fields, trainable-token compaction and RL objective (App. C.1-C.2) on the
    largest chunk's layout, each launch timed alone with L2 flushed before it (CUDA events on
    the launching stream, 3 warm-up + 10 timed launches).  HBM-bound: algorithmic bytes / time."""
    vcs, w = path.vcs, path.w
    ci = path.chunk_in[0]
    lay = vcs.build_segments(ci["cu"], ci["img"], ci["txt"], path.window, path.keep, stream=stream)
    nt, ntraj = lay["num_tokens"], ci["b1"] - ci["b0"]
    ttok = ci["ttok1"] - ci["ttok0"]
    gen = torch.Generator(path.dev).manual_seed(w.seed + 300)
    traj_ids = torch.randint(0, 150000, (ttok,), generator=gen, device=path.dev, dtype=torch.int32)
    traj_lp = -torch.rand(ttok, generator=gen, device=path.dev) * 6
    ids = torch.empty(nt, dtype=torch.int32, device=path.dev)
    old = torch.empty(nt, dtype=torch.float32, device=path.dev)
    status = torch.zeros(1, dtype=torch.int32, device=path.dev)
    logp = -torch.rand(nt, generator=gen, device=path.dev) * 6
    ref = logp + torch.randn(nt, generator=gen, device=path.dev) * 0.1
    adv = torch.randn(ntraj, generator=gen, device=path.dev)
    loss = torch.empty(1, dtype=torch.float64, device=path.dev)
    dlogp = torch.empty(nt, dtype=torch.float32, device=path.dev)
    lws_bytes = vcs.vcs_grpo_loss_workspace_size(nt)
    lws = torch.empty(max(lws_bytes, 256), dtype=torch.uint8, device=path.dev)
    idx = torch.empty(nt, dtype=torch.int32, device=path.dev)
    count = torch.zeros(1, dtype=torch.int64, device=path.dev)
    cws_bytes = vcs.vcs_compact_workspace_size(nt)
    cws = torch.empty(max(cws_bytes, 256), dtype=torch.uint8, device=path.dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=path.dev)
    sp = stream.cuda_stream
    ntrain = int(lay["tok_loss_mask"].sum().item())
    calls = {
        "stream_fields": (lambda: vcs.vcs_stream_fields(traj_ids, traj_lp, ttok, lay["tok_gather"],
                                                        lay["tok_loss_mask"], nt, ids, old, status, sp),
                          nt * (4 + 1 + 4 + 4 + 4) + 4 * ntrain),
        "compact_trainable": (lambda: vcs.vcs_compact_trainable(lay["tok_loss_mask"], nt, idx, nt, count, cws,
                                                                cws_bytes, sp), nt * 1 + 4 * ntrain),
        "grpo_loss": (lambda: vcs.vcs_grpo_loss(logp, old, ref, lay["tok_loss_mask"], lay["cu_seqlens"],
                                                lay["seg_traj"], lay["num_segments"], nt, adv, ntraj, 0.2, 0.28, 3.0,
                                                1e-4, loss, dlogp, lws, lws_bytes, sp), nt * (4 + 4 + 4 + 1 + 4)),
    }
    out = {"tokens": nt, "trainable_tokens": ntrain, "l2": "flushed (256 MB write) before every timed launch"}
    for name, (fn, nbytes) in calls.items():
        times = []
        for i in range(13):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            st = fn()
            e1.record(stream)
            assert st == 0, (name, st)
            if i >= 3:
                times.append((e0, e1))
        torch.cuda.synchronize()
        ms = statistics.median(a.elapsed_time(b) for a, b in times)
        gbs = nbytes / (ms / 1e3) / 1e9
        out[name] = {"ms": ms, "bytes": int(nbytes), "gbs": gbs, "frac_of_hbm": gbs / hbm_gbs}
    assert int(status.item()) == 0 and int(lws[:4].view(torch.int32).item()) == 0
    return out


def _median_ms(fn, stream, flush, reps=10, warm=3):
    """Median of `reps` launches of fn (after `warm`), L2 flushed before each (CUDA events)."""
    times = []
    for i in range(warm + reps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        assert fn() == 0
        e1.record(stream)
        if i >= warm:
            times.append((e0, e1))
    torch.cuda.synchronize()
    return statistics.median(a.elapsed_time(b) for a, b in times)


def run_hbm_kernels(path, stream, hbm_gbs, stress_traj=4096):
    """Builder and gather timed alone (L2 flushed, 3 warm-up + median of 10): the builder on the
    largest chunk and on a 4,096-trajectory batch of the same step distribution (a size at
    which the builder's writes, not its launches, take the time), the gather on the largest
    chunk.  Algorithmic bytes: the builder writes 13 B per segment token (gather index, source
    step, position, loss mask) and 8 B per segment, and reads 8 B per step; the gather reads
    and writes 2 (Hq + 2 Hkv) d bytes per segment token."""
    vcs, w = path.vcs, path.w
    sp = stream.cuda_stream
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=path.dev)
    out = {"l2": "flushed (256 MB write) before every timed launch"}
    ci = path.chunk_in[0]
    nseg, ntok = ci["s1"] - ci["s0"], ci["tok1"] - ci["tok0"]

    def build(c, b, nsteps, img, txt, cu_seqlens, seg_traj, gi, src, pos, mask, sizes, ws, nb, ms, mt):
        return lambda: vcs.vcs_build_segments(c, b, nsteps, img, txt, path.window, path.keep, ms, mt, cu_seqlens,
                                              seg_traj, gi, src, pos, mask, sizes, ws, nb, sp)

    seg_traj = torch.empty(path.max_seg, dtype=torch.int32, device=path.dev)
    ms = _median_ms(build(ci["cu"], ci["b1"] - ci["b0"], ci["nsteps"], ci["img"], ci["txt"], path.cu_seqlens,
                          seg_traj, path.tok_gather, path.tok_src, path.tok_pos, path.tok_mask, path.sizes,
                          path.seg_ws, path.seg_ws_bytes, path.max_seg, path.max_tok), stream, flush)
    nbytes = 13 * ntok + 8 * nseg + 8 * ci["nsteps"]
    out["builder"] = {"us": ms * 1e3, "segment_tokens": ntok, "bytes": nbytes,
                      "gbs": nbytes / (ms / 1e3) / 1e9}
    # builder stress: 4,096 trajectories drawn like the workload's (its own seed)
    import dataclasses
    ws_ = dataclasses.replace(w, num_traj=stress_traj, seed=w.seed + 4096)
    cu, img, txt = workloads.draw_steps(ws_)
    seg_lens, _ = layout_stats(cu, img, txt, path.window, path.keep)
    S, N = int(len(seg_lens)), int(seg_lens.sum())
    if N < 2 ** 31 - 1 and N * 13 < (24 << 30):
        dev = path.dev
        T = lambda n, dt=torch.int32: torch.empty(max(n, 1), dtype=dt, device=dev)  # noqa: E731
        d_cu, d_img, d_txt = (torch.from_numpy(np.ascontiguousarray(x, dtype=np.int32)).to(dev) for x in (cu, img, txt))
        nb = vcs.vcs_segments_workspace_size(stress_traj, len(img))
        bufs = [T(S + 1), T(S), T(N), T(N), T(N), T(N, torch.uint8), torch.zeros(3, dtype=torch.int64, device=dev),
                T(nb, torch.uint8)]
        ms = _median_ms(build(d_cu, stress_traj, len(img), d_img, d_txt, *bufs[:7], bufs[7], nb, S, N), stream,
                        flush)
        nbytes = 13 * N + 8 * S + 8 * len(img)
        out["builder_stress"] = {"trajectories": stress_traj, "segments": S, "segment_tokens": N, "us": ms * 1e3,
                                 "bytes": nbytes, "gbs": nbytes / (ms / 1e3) / 1e9,
                                 "frac_of_hbm": nbytes / (ms / 1e3) / 1e9 / hbm_gbs}
        del bufs
    qt, kt, vt = (x[ci["ttok0"]:ci["ttok1"]] for x in (path.q_traj, path.k_traj, path.v_traj))
    ms = _median_ms(lambda: vcs.vcs_gather(qt, kt, vt, ci["ttok1"] - ci["ttok0"], path.tok_gather, ntok, w.hq, w.hkv,
                                           w.d, path.q, path.k, path.v, path.gstatus, sp), stream, flush)
    nbytes = ntok * 2 * (w.hq + 2 * w.hkv) * w.d * 2
    out["gather"] = {"ms": ms, "bytes": nbytes, "gbs": nbytes / (ms / 1e3) / 1e9,
                     "frac_of_hbm": nbytes / (ms / 1e3) / 1e9 / hbm_gbs}
    assert path.device_status() == (0, 0, 0)
    return out


def run_fused(path, stream, reps=2):
    """Attention reading Q/K/V straight from the trajectory tensors through the gather map
    (vcs_attn_fwd_gathered / vcs_attn_bwd_gathered: no materialised copies, the backward's
    gradients summed into trajectory layout) against gather + vcs_attn_fwd + vcs_attn_bwd, on
    the largest chunk: 1 warm-up + `reps` timed passes each, CUDA events on the stream."""
    vcs, w = path.vcs, path.w
    hq, hkv, d = w.hq, w.hkv, w.d
    ci = path.chunk_in[0]
    sp = stream.cuda_stream
    nseg, ntok, mx = ci["s1"] - ci["s0"], ci["tok1"] - ci["tok0"], ci["max_seqlen"]
    st = vcs.vcs_build_segments(ci["cu"], ci["b1"] - ci["b0"], ci["nsteps"], ci["img"], ci["txt"], path.window,
                                path.keep, path.max_seg, path.max_tok, path.cu_seqlens, None, path.tok_gather,
                                path.tok_src, path.tok_pos, path.tok_mask, path.sizes, path.seg_ws,
                                path.seg_ws_bytes, sp)
    assert st == 0
    ttok = ci["ttok1"] - ci["ttok0"]
    qt, kt, vt = (x[ci["ttok0"]:ci["ttok1"]] for x in (path.q_traj, path.k_traj, path.v_traj))
    dout = path.dout[ci["tok0"]:ci["tok1"]]
    gws_bytes = vcs.vcs_attn_bwd_gathered_workspace_size(nseg, ntok, mx, ttok, hq, hkv, d)
    gws = torch.empty(gws_bytes, dtype=torch.uint8, device=path.dev)
    dqt, dkt, dvt = torch.empty_like(qt), torch.empty_like(kt), torch.empty_like(vt)
    fl, f_fwd, f_bwd = credited_flops(path.seg_lens[ci["s0"]:ci["s1"]], hq, d)

    # each a list of (part, launch) with events recorded between the parts
    fused = [("fwd_ms", lambda: vcs.vcs_attn_fwd_gathered(qt, kt, vt, ttok, path.tok_gather, path.cu_seqlens, nseg,
                                                          ntok, mx, hq, hkv, d, 0.0, path.o, path.lse, path.fwd_ws,
                                                          path.fwd_ws_bytes, sp)),
             ("bwd_ms", lambda: vcs.vcs_attn_bwd_gathered(qt, kt, vt, ttok, path.tok_gather, path.o, path.lse, dout,
                                                          path.cu_seqlens, nseg, ntok, mx, hq, hkv, d, 0.0, dqt, dkt,
                                                          dvt, gws, gws_bytes, sp))]
    materialised = [("gather_ms", lambda: vcs.vcs_gather(qt, kt, vt, ttok, path.tok_gather, ntok, hq, hkv, d, path.q,
                                                         path.k, path.v, path.gstatus, sp)),
                    ("fwd_ms", lambda: vcs.vcs_attn_fwd(path.q, path.k, path.v, path.cu_seqlens, nseg, ntok, mx, hq,
                                                        hkv, d, 0.0, path.o, path.lse, path.fwd_ws,
                                                        path.fwd_ws_bytes, sp)),
                    ("bwd_ms", lambda: vcs.vcs_attn_bwd(path.q, path.k, path.v, path.o, path.lse, dout,
                                                        path.cu_seqlens, nseg, ntok, mx, hq, hkv, d, 0.0, path.dq,
                                                        path.dk, path.dv, path.bwd_ws, path.bwd_ws_bytes, sp))]

    out = {"chunk_segment_tokens": ntok, "chunk_trajectory_tokens": ttok}
    for name, parts in (("fused", fused), ("materialised", materialised)):
        runs = []
        for i in range(1 + reps):
            e = [torch.cuda.Event(enable_timing=True) for _ in range(len(parts) + 1)]
            e[0].record(stream)
            for j, (_, fn) in enumerate(parts):
                assert fn() == 0, (name, parts[j][0])
                e[j + 1].record(stream)
            if i > 0:
                runs.append(e)
        torch.cuda.synchronize()
        ms = statistics.mean(e[0].elapsed_time(e[-1]) for e in runs)
        out[name] = {"ms": ms, "tflops": fl / (ms / 1e3) / 1e12}
        for j, (part, _) in enumerate(parts):
            out[name][part] = statistics.mean(e[j].elapsed_time(e[j + 1]) for e in runs)
    assert int(gws[:4].view(torch.int32).item()) == 0 and path.device_status() == (0, 0, 0)
    out["fused"]["note"] = ("forward + backward with dQ, dK, dV scattered into trajectory layout "
                            "(fp32 sums over each token's copies)")
    out["materialised"]["note"] = "gather + forward + backward, gradients left in segment layout"
    del gws, dqt, dkt, dvt
    return out


def run_reuse(path, stream, reps=3):
    """Forward with prefix reuse (each query-tile pair whose rows a trajectory's previous
    segment shares is copied, not computed) against the plain forward, on the largest
    chunk: vcs_shared_prefix, vcs_attn_fwd_reuse and vcs_attn_fwd timed with CUDA events,
    1 warm-up + `reps` timed launches each.  TFLOP/s are the plain forward's credited flops
    over each time, so the ratio is the speed-up."""
    vcs, w = path.vcs, path.w
    hq, hkv, d = w.hq, w.hkv, w.d
    ci = path.chunk_in[0]
    sp = stream.cuda_stream
    nseg, ntok, mx = ci["s1"] - ci["s0"], ci["tok1"] - ci["tok0"], ci["max_seqlen"]
    seg_traj = torch.empty(path.max_seg, dtype=torch.int32, device=path.dev)
    assert vcs.vcs_build_segments(ci["cu"], ci["b1"] - ci["b0"], ci["nsteps"], ci["img"], ci["txt"], path.window,
                                  path.keep, path.max_seg, path.max_tok, path.cu_seqlens, seg_traj, path.tok_gather,
                                  path.tok_src, path.tok_pos, path.tok_mask, path.sizes, path.seg_ws,
                                  path.seg_ws_bytes, sp) == 0
    qt, kt, vt = (x[ci["ttok0"]:ci["ttok1"]] for x in (path.q_traj, path.k_traj, path.v_traj))
    assert vcs.vcs_gather(qt, kt, vt, ci["ttok1"] - ci["ttok0"], path.tok_gather, ntok, hq, hkv, d, path.q, path.k,
                          path.v, path.gstatus, sp) == 0
    shared = torch.empty(nseg, dtype=torch.int32, device=path.dev)
    status = torch.zeros(1, dtype=torch.int32, device=path.dev)
    calls = {
        "shared_prefix_ms": lambda: vcs.vcs_shared_prefix(path.cu_seqlens, seg_traj, path.tok_gather, nseg, ntok,
                                                          shared, status, sp),
        "fwd_reuse_ms": lambda: vcs.vcs_attn_fwd_reuse(path.q, path.k, path.v, path.cu_seqlens, shared, nseg, ntok, mx,
                                                       hq, hkv, d, 0.0, path.o, path.lse, path.fwd_ws,
                                                       path.fwd_ws_bytes, sp),
        "fwd_ms": lambda: vcs.vcs_attn_fwd(path.q, path.k, path.v, path.cu_seqlens, nseg, ntok, mx, hq, hkv, d, 0.0,
                                           path.o, path.lse, path.fwd_ws, path.fwd_ws_bytes, sp),
    }
    out = {"chunk_segment_tokens": ntok}
    for name, fn in calls.items():
        times = []
        for i in range(1 + reps):
            e = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
            e[0].record(stream)
            assert fn() == 0, name
            e[1].record(stream)
            if i > 0:
                times.append(e)
        torch.cuda.synchronize()
        out[name] = statistics.mean(a.elapsed_time(b) for a, b in times)
    assert int(status.item()) == 0 and path.device_status() == (0, 0, 0)
    # credited forward flops of the skipped pairs (their rows are copied) against the chunk's
    lens = path.seg_lens[ci["s0"]:ci["s1"]].astype(np.int64)
    skip = shared.cpu().numpy().astype(np.int64) // 256 * 256
    _, f_all, _ = credited_flops(lens, hq, d)
    _, f_skip, _ = credited_flops(skip, hq, d)
    out["skipped_flop_frac"] = f_skip / f_all
    out["fwd_tflops"] = f_all / (out["fwd_ms"] / 1e3) / 1e12
    out["fwd_reuse_tflops_equiv"] = f_all / (out["fwd_reuse_ms"] / 1e3) / 1e12
    return out


def run_e2e(path, args, flops, stream):
    """Same metric through the public API with host buffers: every step's inputs copied from
    pinned host memory and every step's result (dQ, dK, dV of every chunk) copied back to
    pinned host memory, inside the timed region."""
    srcs = {"q": path.q_traj, "k": path.k_traj, "v": path.v_traj, "do": path.dout}
    w = path.w
    res_shapes = {"dq": (path.num_tokens, w.hq, w.d), "dk": (path.num_tokens, w.hkv, w.d),
                  "dv": (path.num_tokens, w.hkv, w.d)}
    need_in = sum(t.numel() * t.element_size() for t in srcs.values())
    try:
        avail = int(next(l for l in open("/proc/meminfo") if l.startswith("MemAvailable")).split()[1]) * 1024
    except Exception:
        avail = 0
    # every rank of this node pins its own copy at the same time, so the node's need is checked;
    # every rank takes the same branch (the decisions are reduced over ranks), so that the
    # collectives below are entered by all of them or by none.  The result buffers hold the
    # whole step's gradients when they fit beside the inputs; otherwise one chunk's, which every
    # chunk's gradients pass through in turn (the bytes copied back per step are the same).
    local_ranks = int(os.environ.get("LOCAL_WORLD_SIZE", "1"))
    res_rows = path.num_tokens
    if sum_over_ranks(float((need_in + sum(2 * math.prod(sh) for sh in res_shapes.values())) * local_ranks
                            > 0.6 * avail), path.dev) > 0:
        res_rows = path.max_tok
        res_shapes = {k: (res_rows,) + sh[1:] for k, sh in res_shapes.items()}
    need = need_in + sum(2 * math.prod(sh) for sh in res_shapes.values())
    if sum_over_ranks(float(need * local_ranks > 0.6 * avail), path.dev) > 0:
        return {"value": None, "unit": "TFLOP/s",
                "error": f"pinned staging of {local_ranks} x {need / 2**30:.0f} GiB exceeds 60% of available "
                         f"host memory ({avail / 2**30:.0f} GiB)"}
    host, res, err = {}, {}, None
    try:
        for name, t in srcs.items():
            host[name] = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
            host[name].copy_(t)
        for name, sh in res_shapes.items():
            res[name] = torch.empty(sh, dtype=torch.bfloat16, pin_memory=True)
    except RuntimeError as e:
        err = f"pinned staging failed: {e}"[:200]
    if sum_over_ranks(float(err is not None), path.dev) > 0:
        return {"value": None, "unit": "TFLOP/s", "error": err or "pinned staging failed on another rank"}
    h2d = sum(t.numel() * t.element_size() for t in host.values())
    d2h = path.num_tokens * (w.hq + 2 * w.hkv) * w.d * 2          # every chunk's dQ, dK, dV
    whole = res_rows == path.num_tokens
    # Each step's inputs are copied from pinned host memory on a second stream, chunk by
    # chunk: a chunk's copy for the next step starts once its launches of this step are done,
    # so it overlaps the other chunk's compute.  A chunk's builder, gather and forward wait
    # for its Q/K/V; its backward for its dO (copied after them, under the forward).  Each
    # chunk's dQ, dK, dV go back to the host on a third stream as soon as its backward is
    # done (under the next chunk's builder, gather and forward); the next backward, which
    # overwrites the device buffers, waits for that copy.
    cs = torch.cuda.Stream(device=path.dev)
    rs = torch.cuda.Stream(device=path.dev)
    nch = len(path.chunk_in)
    # chunks alternate between two sets of device gradient buffers, so that a chunk's backward
    # never waits for the previous chunk's gradients to reach the host
    gsets = [(path.dq, path.dk, path.dv), tuple(torch.empty_like(t) for t in (path.dq, path.dk, path.dv))]
    chunk_no = {"n": 0}
    set_of = {}
    copied = [torch.cuda.Event() for _ in range(nch)]
    copied_do = [torch.cuda.Event() for _ in range(nch)]
    done = [torch.cuda.Event() for _ in range(nch)]
    state = {"step": 0, "returned": [None, None]}

    def copy_chunk(i):
        ci = path.chunk_in[i]
        a, b, t0_, t1_ = ci["ttok0"], ci["ttok1"], ci["tok0"], ci["tok1"]
        with torch.cuda.stream(cs):
            path.q_traj[a:b].copy_(host["q"][a:b], non_blocking=True)
            path.k_traj[a:b].copy_(host["k"][a:b], non_blocking=True)
            path.v_traj[a:b].copy_(host["v"][a:b], non_blocking=True)
            copied[i].record(cs)
            path.dout[t0_:t1_].copy_(host["do"][t0_:t1_], non_blocking=True)
            copied_do[i].record(cs)

    def before(i):
        stream.wait_event(copied[i])

    def grads(i):
        k = chunk_no["n"] % 2                        # this chunk's gradient buffer set
        set_of[i] = k
        chunk_no["n"] += 1
        return gsets[k]

    def before_bwd(i):
        stream.wait_event(copied_do[i])
        k = chunk_no["n"] % 2
        if state["returned"][k] is not None:        # that set's last gradients are still being read
            stream.wait_event(state["returned"][k])

    def after(i):
        done[i].record(stream)
        ci = path.chunk_in[i]
        n = ci["tok1"] - ci["tok0"]
        k = set_of[i]
        rs.wait_event(done[i])
        r0 = ci["tok0"] if whole else 0              # copies on rs run in order: a shared buffer is free
        with torch.cuda.stream(rs):
            for name, t in zip(("dq", "dk", "dv"), gsets[k]):
                res[name][r0:r0 + n].copy_(t[:n], non_blocking=True)
            ev = torch.cuda.Event()
            ev.record(rs)
        state["returned"][k] = ev
        state["last"] = (ev, k)
        if state["step"] + 1 < args.steps:           # the next step's inputs for this chunk
            cs.wait_event(done[i])
            copy_chunk(i)

    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    cs.wait_event(t0)
    for i in range(nch):
        copy_chunk(i)
    for s_ in range(args.steps):
        state["step"] = s_
        path.step(stream, before_chunk=before, after_chunk=after, before_bwd=before_bwd, grads=grads)
    stream.wait_event(state["last"][0])              # the last chunk's gradients are on the host
    t1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(t0.elapsed_time(t1) / args.steps, path.dev)
    path.verify_sizes()
    # the host copy holds the step's gradients: spot-check one row of each against the device
    ci = path.chunk_in[-1]
    n = ci["tok1"] - ci["tok0"]
    r0 = ci["tok0"] if whole else 0
    for name, dev_t in zip(("dq", "dk", "dv"), gsets[state["last"][1]]):
        assert torch.equal(res[name][r0 + n - 1], dev_t[n - 1].cpu()), name
    # the bytes every rank copies (the whole job's, like the value)
    h2d = sum_over_ranks(float(h2d), path.dev)
    d2h = sum_over_ranks(float(d2h), path.dev)
    return {"value": flops / (ms / 1e3) / 1e12, "unit": "TFLOP/s", "ms_per_step": ms,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "result": "dQ, dK, dV of every segment token (bf16) copied to pinned host memory every step, into "
                      + ("buffers holding the whole step" if whole else
                         "one chunk-sized buffer per tensor that each chunk's gradients pass through (the whole "
                         "step's would not fit beside the pinned inputs in 60% of the host's available memory)")}


if __name__ == "__main__":
    main()
