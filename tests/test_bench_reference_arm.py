"""The benchmark's reference arm on CPU: `bench.py --impl reference` times the oracle on a bounded
sample of the benchmark workload and prints one JSON line with the GPU arm's metric, unit,
direction and workload description, a `cpu_baseline` describing the run and an end-to-end entry
with no host-device copies.  Also the helpers that describe the workload and summarise the
nvidia-smi clock samples taken during a timed region."""
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
    # ceil(10 epochs x 50,000 / (16 x 128)) = 245 local steps; t' = floor(0.5 x 245) = 122
    assert bench.job_steps(w) == 245 and bench.switch_step(w) == 122
    cfg = bench.workload_config(w, 16, 1)
    assert cfg["workload"] == "mlp_3072-4096x3-100_K16_B128_postlocal_H16_bf16"
    assert cfg["global_batch"] == 2048 and cfg["K"] == 16 and cfg["B_loc"] == 128
    assert cfg["params_per_replica"] == 46559332 and cfg["parallelism"] == "single"
    assert cfg["schedule"] == "post-local: H = 1 before t' = 122, H = 16 after"
    assert bench.workload_config(w, 16, 4)["parallelism"] == "replicas"
    assert bench.workload_config(w, 8, 1)["workload"].endswith("K8_B128_postlocal_H16_bf16")
    # the MLP 3072-1024-1024-10 configuration: ceil(2 x 50,000 / 2048) = 49 steps, no switch
    assert bench.job_steps(bench.CONFIG2) == 49 and bench.switch_step(bench.CONFIG2) == -1
    assert bench.dense_params(bench.CONFIG2["widths"]) == 4206602
    assert bench.job_steps(bench.SOFTMAX) == 64


def test_reference_arm_prints_one_contract_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1",
                        "--warmup", "1"], cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    assert d["metric"] == "samples/s over K simulated workers (1 GB300)"
    assert d["unit"] == "samples/s" and d["higher_is_better"] is True
    assert d["steps"] == 1 and d["warmup"] == 1 and d["n_gpus"] == 1
    assert d["value"] > 0 and d["ms_per_step"] > 0
    assert d["config"] == bench.workload_config(bench.WORKLOAD, 16, 1)
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_clock_summary_reads_nvidia_smi_rows():
    rows = [
        "0, 2070, 2070, 812.31, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n",
        "0, 1980, 2070, 1391.02, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n",
        "0, 2070, 2070, 1020.50, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n",
        "0, [N/A], 2070, 1.0, 0x0, Not Active, Not Active, Not Active, Not Active\n",  # unusable
        "garbage\n",
    ]
    c = bench.summarise_clocks(rows)
    assert c == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    hot = rows[:1] + ["0, 1500, 2070, 900.0, 0x48, Active, Not Active, Active, Not Active\n"]
    c = bench.summarise_clocks(hot)
    assert c["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"] and c["sm_mhz"] == 1785.0
    assert bench.summarise_clocks(["garbage\n"]) is None
