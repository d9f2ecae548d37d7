"""bench.py's reference arm (the float64 oracle on the host cores) prints the
same one-line JSON contract as the CUDA arm: one line on rank 0, the same
metric, unit and workload, impl = "reference", and its own cpu_baseline and
e2e objects.  Runs on the CPU with the 8-query tiny workload."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run_reference(*extra):
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "tiny_f32_1k",
                        "--steps", "2", "--warmup", "1", "--ref-seconds", "1.5", *extra],
                       cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    return [json.loads(line) for line in r.stdout.splitlines() if line.startswith("{")]


def test_reference_arm_prints_one_contract_line():
    import bench

    lines = _run_reference()
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference"
    assert d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["higher_is_better"] is True and d["scaling"] == "weak"
    assert (d["n_gpus"], d["steps"], d["warmup"]) == (1, 2, 1)
    assert d["config"]["workload"] == "tiny_f32_1k"
    assert d["config"]["queries_per_step"] >= 1
    assert d["value"] > 0 and d["ms_per_step"] > 0
    # value = queries per step / mean step time
    assert d["value"] == pytest.approx(d["config"]["queries_per_step"] / (d["ms_per_step"] / 1e3), rel=1e-9)
    assert d["vs_baseline"] is None and d["data"] == "synthetic" and d["dtype"] == "f64"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["unit"] == d["unit"]
    assert cb["cores"] >= 1 and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_flat_scan_line():
    lines = _run_reference("--flat")
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference" and d["config"].get("flat") is True
    assert d["value"] > 0 and "flat retrieval" in d["cpu_baseline"]["sample"]


def test_algorithmic_work_by_hand():
    """The roofline's algorithmic bytes and flops (each selected group's
    entries read once, the queries once, the group keys as bf16 hi + lo,
    the outputs; 2*D flops per (query, candidate) pair and per (query,
    group) pair) on a selection small enough to count by hand: 3 queries,
    groups of 5 / 0 / 7 / 2 entries, D = 8, bf16, buckets of >= 2 queries on
    the tensor cores."""
    import dataclasses

    import numpy as np

    import bench
    from paper_2605_29734_gb300 import workloads

    w = dataclasses.replace(workloads.WORKLOADS["tiny_f32_1k"], dtype="bf16", d=8, g=4, b=3, k_groups=2,
                            k_entries=3)
    counts = np.array([5, 0, 7, 2])
    group_idx = np.array([[0, 2], [2, 3], [0, -1]])
    wk = bench.step_work(w, counts, group_idx, tc_min=2)
    # buckets: group 0 <- 2 queries, group 2 <- 2, group 3 <- 1
    assert wk["kernels"]["fine"] == {"bytes": 2 * 8 * 2 + 1 * 8 * 2, "flops": 2 * 8 * (1 * 2)}
    assert wk["kernels"]["fine_tc"] == {"bytes": (5 + 7) * 8 * 2 + 3 * 8 * 2, "flops": 2 * 8 * (2 * 5 + 2 * 7)}
    out_bytes = 3 * (2 * 8 + 3 * 12 + 4)  # group id + score, entry id + score + weight, lse
    assert wk["step_bytes"] == (5 + 7 + 2) * 8 * 2 + 3 * 8 * 2 + 4 * 8 * 4 + out_bytes
    assert wk["step_flops"] == 2 * 8 * (12 + 9 + 5) + 2 * 8 * 3 * 4
    assert wk["mean_candidates"] == pytest.approx(26 / 3)
    flat = bench.step_work(w, counts, group_idx, tc_min=2, flat=True)
    assert flat["step_bytes"] == (5 + 7 + 2) * 8 * 2 + 3 * 8 * 2 + 3 * (3 * 12 + 4)
    assert flat["step_flops"] == 2 * 8 * (12 + 9 + 5)
    # tensor cores off (tc_min above the batch): everything on the CUDA cores
    off = bench.step_work(w, counts, group_idx, tc_min=1 << 30)
    assert off["kernels"]["fine_tc"]["bytes"] == 0 and off["kernels"]["fine"]["flops"] == 2 * 8 * 26
