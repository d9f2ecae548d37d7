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
