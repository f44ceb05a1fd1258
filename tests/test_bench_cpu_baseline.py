"""The bench's CPU-baseline leg on the host (no GPU): the oracle sample's fields, the
one-core run in its own interpreter, and the extrapolation to the whole workload."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def test_one_core_run_reports_its_sample():
    import bench
    r = bench.oracle_one_core(64, 300, 5)
    assert r["value"] is not None and r["value"] > 0, r
    assert r["cores"] == 1 and r["seconds"] > 0
    assert r["pairs_per_s"] == pytest.approx(300 * 301 / 2 / r["seconds"])


def test_oracle_sample_fields_and_extrapolation():
    import numpy as np
    import bench
    from oracle import segments as oseg
    from paper_2607_11185_gb300 import workloads
    w = workloads.WORKLOADS["tiny"]
    r = bench.oracle_sample(w, w.window, w.keep)
    assert r["kind"] == "oracle" and r["unit"] == "TFLOP/s" and r["cores"] == os.cpu_count()
    assert r["value"] > 0 and r["seconds"] > 0 and r["one_core"]["cores"] == 1
    # the extrapolation is the whole workload's credited flops at the sample's rate
    cu, img, txt = workloads.draw_steps(w)
    lens = np.diff(oseg.build(cu, img, txt, w.window, w.keep, method="closed")["cu_seqlens"]).astype(np.int64)
    job = 12.0 * w.d * w.hq * float((lens * (lens + 1) // 2).sum())
    assert r["extrapolated_full_workload_s"] == pytest.approx(job / (r["value"] * 1e12), rel=1e-9)
