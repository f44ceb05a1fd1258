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


def test_reference_arm_prints_one_contract_line():
    import contextlib
    import io
    import json
    import types
    import bench
    from paper_2607_11185_gb300 import workloads
    w = workloads.WORKLOADS["tiny"]
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        bench.run_reference(types.SimpleNamespace(warmup=0, steps=1, gpus=1), w, w.window, w.keep, 0, 1)
    lines = [ln for ln in buf.getvalue().splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "TFLOP/s" and d["higher_is_better"] is True
    assert d["metric"] == bench.METRIC and d["value"] > 0 and d["steps"] == 1 and d["warmup"] == 0
    assert d["cpu_baseline"]["value"] == d["value"] and d["cpu_baseline"]["kind"] == "oracle"
    assert d["e2e"] == {"value": d["value"], "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert d["config"]["workload"] == "tiny"
