"""The benchmark's reference arm on CPU: `bench.py --impl reference` times the oracle on a bounded
sample of the benchmark workload and prints one JSON line with the GPU arm's metric, unit,
direction and workload description, a `cpu_baseline` describing the run and an end-to-end entry
with no host-device copies.  Also the helpers that describe the workload."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_dense_params_counts_weights_and_biases():
    # 3072 x 1024 + 1024, 1024 x 1024 + 1024, 1024 x 10 + 10
    assert bench.dense_params((3072, 1024, 1024, 10)) == 4206602
    assert bench.dense_params((3072, 10)) == 30730
    assert bench.dense_params((5, 1)) == 6


def test_job_and_workload_config():
    w = bench.WORKLOAD
    # ceil(2 epochs x 50,000 / (16 x 128)) = 49 local steps
    assert bench.job_steps(w) == 49
    cfg = bench.workload_config(w, 16, 1)
    assert cfg["workload"] == "mlp_3072-1024-1024-10_K16_B128_H16_bf16"
    assert cfg["global_batch"] == 2048 and cfg["K"] == 16 and cfg["B_loc"] == 128
    assert cfg["params_per_replica"] == 4206602 and cfg["parallelism"] == "single"
    assert bench.workload_config(w, 16, 4)["parallelism"] == "replicas"
    assert bench.workload_config(w, 8, 1)["workload"].endswith("K8_B128_H16_bf16")


def test_reference_arm_prints_one_contract_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1",
                        "--warmup", "3"], cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    assert d["metric"] == "samples/s over K simulated workers (1 GB300)"
    assert d["unit"] == "samples/s" and d["higher_is_better"] is True
    assert d["steps"] == 1 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["value"] > 0 and d["ms_per_step"] > 0
    assert d["config"] == bench.workload_config(bench.WORKLOAD, 16, 1)
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
