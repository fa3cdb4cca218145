#!/usr/bin/env python3
"""Throughput of post-local SGD over K simulated workers on one GB300 (samples/s).

Workload (the largest configuration): post-local SGD on MLP 3072-4096-4096-4096-100 (ReLU,
He-normal init), bf16 GEMM operands with fp32 accumulation and fp32 master weights, K = 16 workers,
B_loc = 128, 10 epochs of N = 50,000 synthetic CIFAR-100-shaped Gaussian-mixture points (32x32x3,
100 classes) = a 245-step job; H = 1 (an average after every step) before t' = floor(T / 2) = 122
and H = 16 after it (Sec. 3, Algorithm 2); Nesterov momentum 0.9 kept local, weight decay 5e-4,
learning rate 0.1 decayed 10x at 50 % and 75 % of the job.  One timed step = one local step of all
K replicas (sampling, gather + cast, forward, loss, backward, fused update) plus the K-way average
when the schedule ends a round there.  `value` is device-timed with inputs resident in HBM; `e2e`
drives the same steps through lsgd_local_step_batch with each step's mini-batch copied from pinned
host memory and its losses read back.  The MLP 3072-1024-1024-10 configuration (H = 16, lr 0.1
scaled by K with warm-up) is timed as well and reported under "config2".

--impl reference times the oracle (single-threaded C++, fp64) on the host cores instead, on the
same bounded sample as the GPU line's cpu_baseline.  Under torchrun (N > 1) every rank runs an
independent replica of the workload (no collective on the data path); the time is the maximum
over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import platform
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

# The benchmark workloads.  Learning-rate readings: config 2 states "lr 0.1 scaled by K with
# 5-epoch linear warmup"; config 3 states only the decays, so its rate is 0.1 without K scaling or
# warm-up (the scaled rate, 1.6, drives this deep MLP to NaN in its H = 1 phase).
WORKLOAD = dict(name="mlp_3072-4096x3-100_K16_B128_postlocal_H16_bf16",
                widths=(3072, 4096, 4096, 4096, 100), K=16, B=128, H=16, N=50000, C=100,
                epochs=10.0, t_switch_frac=0.5, base_lr=0.1, scale_by_K=False, warmup_epochs=0.0,
                milestones=(0.5, 0.75), momentum=0.9, nesterov=True, weight_decay=5e-4, seed=0,
                data_seed=1234, bf16=True, init="he")
CONFIG2 = dict(name="mlp_3072-1024-1024-10_K16_B128_H16_bf16", widths=(3072, 1024, 1024, 10),
               K=16, B=128, H=16, N=50000, C=10, epochs=2.0, t_switch_frac=None, base_lr=0.1,
               scale_by_K=True, warmup_epochs=5.0, milestones=(), momentum=0.9, nesterov=True,
               weight_decay=5e-4, seed=0, data_seed=1234, bf16=True, init="he")
SOFTMAX = dict(name="softmax_3072-10_K4_B32_H4_fp32", widths=(3072, 10), K=4, B=32, H=4, N=8192,
               C=10, epochs=1.0, t_switch_frac=None, base_lr=0.1, scale_by_K=False,
               warmup_epochs=0.0, milestones=(), momentum=0.0, nesterov=False, weight_decay=0.0,
               seed=0, data_seed=1234, bf16=False, init="zero", T=64)
SWEEP = dict(name="mlp_3072-512-512-10_B32", widths=(3072, 512, 512, 10), K=8, B=32, H=1,
             N=50000, C=10, epochs=1.0, t_switch_frac=None, base_lr=0.1, scale_by_K=False,
             warmup_epochs=0.0, milestones=(), momentum=0.9, nesterov=False, weight_decay=0.0,
             seed=0, data_seed=1234, bf16=True, init="he", T=500)
RESNET_WORKLOAD = dict(name="resnet20_K16_B128_postlocal_H16_bf16", K=16, B=128, H=16, N=50000,
                       C=10, base_lr=0.2, scale_by_K=True, warmup_epochs=5.0, momentum=0.9,
                       nesterov=True, weight_decay=1e-4, seed=0, data_seed=1234, epochs=1.0)
DENSE_CONFIGS = {"softmax": SOFTMAX, "mlp1024": CONFIG2, "mlp4096": WORKLOAD}


def job_steps(w, K=None):
    """T of one training job: ceil(epochs * N / (K * B_loc)) local steps (245 for the workload)."""
    if "T" in w:
        return w["T"]
    K = K or w["K"]
    return -(-int(w["epochs"] * w["N"]) // (K * w["B"]))


def switch_step(w, K=None):
    """The post-local switch t' = floor(frac * T) (the first learning-rate decay), or -1."""
    f = w.get("t_switch_frac")
    return -1 if f is None else int(f * job_steps(w, K))


# Bytes the algorithm moves per parameter and replica (fp32 w, u, g; bf16 shadow):
#   stand-alone update           = read g, w, u + write w, u (4 B each) + write the shadow (2 B) = 22
#   update fused into the weight-gradient epilogue = read w, u + write w, u + write shadow = 18,
#     plus the bf16 operands it reads (activations and output gradients, 2 B each)
#   average = read w + write w (4 B each) + write bf16 shadow (2 B) = 10
UPDATE_BYTES_PER_PARAM = 22
FUSED_UPDATE_BYTES_PER_PARAM = 18
AVERAGE_BYTES_PER_PARAM = 10
# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) of one step's update launches by step
# kind, from single-pass ncu captures of the current kernels at the benchmark's size:
#   MLP 3072-4096x3-100, K = 16, B_loc = 128 (2 launches per step: layer 2, then layers 1, 0 and
#   the 100-class layer):
#     "avg_synced" -- a step of the H = 1 phase (the replicas agree at its start, it ends with
#                     the average): 6,695,380,736 B (step 3 of the job);
#     "plain"      -- an H = 16 step that neither starts synced nor ends a round:
#                     13,583,207,680 B (step 126);
#   MLP 3072-1024-1024-10, K = 16, B_loc = 128: "plain" 1,187,127,808 B (the classifier head's
#     backward plus the one launch of both hidden layers).
# A traced window with a step of another kind reports no traffic.
UPDATE_TRAFFIC_PER_STEP = {
    WORKLOAD["name"]: {"avg_synced": 6695380736, "plain": 13583207680},
    CONFIG2["name"]: {"plain": 1187127808},
}

FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0

# The oracle's bounded sample (both arms): one replica's local step on the first ORACLE_ROWS rows
# of its mini-batch (forward, backward) plus the update of all its parameters.
ORACLE_ROWS = 16


def dense_params(widths):
    """Parameters per replica of a dense network: weights and biases of every layer."""
    return sum(a * b + b for a, b in zip(widths[:-1], widths[1:]))


def workload_config(w, K, world, fused=True):
    """The workload description both arms print, identically."""
    B, H, T_job = w["B"], w["H"], job_steps(w, K)
    ts = switch_step(w, K)
    name = w["name"] if K == w["K"] else w["name"].replace(f"K{w['K']}", f"K{K}")
    sched = (f"post-local: H = 1 before t' = {ts}, H = {H} after" if ts >= 0 else f"H = {H}")
    return {"workload": name, "global_batch": K * B, "K": K, "B_loc": B, "H": H,
            "schedule": sched, "fused_update": fused,
            "job": f"{T_job}-step schedule ({w['epochs']:g} epochs of N = {w['N']}), "
                   "repeated from its end state",
            "params_per_replica": dense_params(w["widths"]),
            "parallelism": "replicas" if world > 1 else "single",
            "l2": "inputs larger than L2: the per-step working set (w, u, shadow) is "
                  f"{(10 * K * dense_params(w['widths'])) / 1e9:.1f} GB against the 129 MB L2"}


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops_sustained"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, "fallback"


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(x: float, world: int) -> float:
    """The largest value of x over all ranks (every rank gets it); x itself with one rank.  The
    tensor lives where the process group's backend wants it (GPU for NCCL, host for gloo)."""
    if world == 1:
        return float(x)
    import torch
    import torch.distributed as dist

    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_throughput(units_per_rank: float, seconds: float, world: int) -> float:
    """Units all ranks processed over the slowest rank's time (replicas only: every rank runs the
    same fixed work, so the job ends when the slowest does)."""
    return world * units_per_rank / max_over_ranks(seconds, world)


def host_info():
    """Host cores and CPU model of the machine the oracle is timed on."""
    model = platform.processor() or platform.machine()
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                model = line.split(":", 1)[1].strip()
                break
    except Exception:
        pass
    return {"nproc": os.cpu_count(), "cpu_model": model, "machine": platform.machine()}


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons; mark() brackets the timed region so
    that only the samples taken inside it are summarised."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.path = None
        self.lines = []

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "20", "-i", str(self.dev)],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def count(self) -> int:
        """Rows written so far (the sampler's position, to bracket a region)."""
        if not self.proc:
            return 0
        with open(self.path) as f:
            return sum(1 for _ in f)

    def stop(self, first: int = 0, last: int | None = None):
        """Summary of rows [first, last) (all rows by default)."""
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        with open(self.path) as f:
            lines = f.readlines()
        os.unlink(self.path)
        sel = lines[first:last] if last is not None else lines[first:]
        return summarise_clocks(sel or lines)


def summarise_clocks(lines):
    """Median SM clock, highest maximum clock and every throttle reason seen Active in nvidia-smi
    CSV rows of ClockSampler.FIELDS (no header, no units); None without a usable row."""
    rows = []
    for line in lines:
        parts = [p.strip() for p in line.split(",")]
        if len(parts) < 9:
            continue
        try:
            rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
        except ValueError:
            continue
    if not rows:
        return None
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    reasons = sorted({names[i] for _, _, r in rows for i, v in enumerate(r) if v.lower() == "active"})
    return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
            "reasons": reasons, "samples": len(rows)}


def make_gpu_cfg(P, w, fused=True, K=None):
    K = K or w["K"]
    return P.make_config(K=K, B_loc=w["B"], H=w["H"], t_switch=switch_step(w, K),
                         total_steps=job_steps(w, K), N=w["N"], widths=w["widths"],
                         init=P.INIT_ZERO if w["init"] == "zero" else P.INIT_HE,
                         base_lr=w["base_lr"], scale_by_K=w["scale_by_K"],
                         warmup_epochs=w["warmup_epochs"], milestones=w["milestones"],
                         momentum=w["momentum"], nesterov=w["nesterov"],
                         weight_decay=w["weight_decay"], seed=w["seed"],
                         precision=P.BF16 if w["bf16"] else P.FP32,
                         fused_update=fused and w["bf16"])


def make_oracle_cfg(oracle, w, K=None, T=None):
    K = K or w["K"]
    return oracle.make_cfg(widths=w["widths"], bf16=w["bf16"], K=K, B=w["B"], H=w["H"],
                           t_switch=switch_step(w, K), T=T or job_steps(w, K), N=w["N"],
                           base_lr=w["base_lr"], scale_by_K=w["scale_by_K"],
                           warmup_epochs=w["warmup_epochs"], milestones=w["milestones"],
                           momentum=w["momentum"], nesterov=w["nesterov"],
                           weight_decay=w["weight_decay"], seed=w["seed"])


def oracle_sample(w, X, y, n_steps: int, rows: int, budget_s: float):
    """Time the oracle on up to `n_steps` local steps of single replicas of workload w (the first
    `rows` rows of each worker's mini-batch, forward and backward, then the update of all the
    replica's parameters), stopping once budget_s has passed.  Returns (seconds, samples, steps)."""
    import numpy as np

    import oracle

    o = make_oracle_cfg(oracle, w)
    wt = oracle.init_params(o, oracle.INIT_ZERO if w["init"] == "zero" else oracle.INIT_HE)
    u = np.zeros_like(wt)
    t0 = time.perf_counter()
    done = 0
    for i in range(n_steps):
        idx = oracle.sample_indices(o, i % o.K, i // o.K)[:rows]
        _, g = oracle.loss_grad(o, wt, X, y=y, idx=idx)
        wt, u = oracle.sgd_update(o, oracle.lr(o, i // o.K), wt, u, g)
        done += 1
        if time.perf_counter() - t0 > budget_s:
            break
    return time.perf_counter() - t0, done * rows, done


def oracle_sample_text(w, steps, rows):
    return (f"{steps} single-replica local steps of {w['name']}, each on the first {rows} of the "
            f"worker's {w['B']} mini-batch rows (forward, backward) plus the update of all "
            f"{dense_params(w['widths'])} parameters, on one host core")


def oracle_other_configs(budget_s: float = 6.0):
    """The oracle timed on the other configurations, one host core each: softmax regression's
    whole 64-step job (K = 4), config 2 and ResNet-20 on bounded single-replica samples, and the
    K x H sweep network's first 4 local steps + 1 average at K = 8."""
    import numpy as np

    import oracle
    import synthdata

    out = {}
    # softmax regression: the whole job
    w = SOFTMAX
    X, y = synthdata.gaussian_mixture_cached(w["N"], 3072, w["C"], w["data_seed"])
    o = make_oracle_cfg(oracle, w)
    W0 = np.zeros((w["K"], oracle.num_params(o)))
    t0 = time.perf_counter()
    _, _, _, syncs = oracle.run(o, X, y=y, W=W0)
    t = time.perf_counter() - t0
    out["softmax"] = {"workload": w["name"], "samples_per_s": w["T"] * w["K"] * w["B"] / t,
                      "ms_per_step": 1000 * t / w["T"], "sample": f"the whole {w['T']}-step job "
                      f"({syncs} averages)"}
    # config 2: bounded single-replica sample
    w = CONFIG2
    X, y = synthdata.gaussian_mixture_cached(w["N"], 3072, w["C"], w["data_seed"])
    t, samples, steps = oracle_sample(w, X, y, 64, 32, budget_s)
    out["mlp1024"] = {"workload": w["name"], "samples_per_s": samples / t,
                      "sample": oracle_sample_text(w, steps, 32)}
    # the sweep network at K = 8, B = 32: the first 4 local steps and the average that ends them
    w = SWEEP
    o = make_oracle_cfg(oracle, w, T=4)
    o.H = 4
    t0 = time.perf_counter()
    _, _, _, syncs = oracle.run(o, X, y=y, n_steps=4)
    t = time.perf_counter() - t0
    out["mlp512"] = {"workload": w["name"] + "_K8_H4", "samples_per_s": 4 * w["K"] * w["B"] / t,
                     "ms_per_step": 1000 * t / 4,
                     "sample": f"the first 4 local steps of all 8 replicas + {syncs} average"}
    # ResNet-20: one replica's step on 8 images + its update
    w = RESNET_WORKLOAD
    X10, y10 = synthdata.gaussian_mixture_cached(w["N"], 3072, w["C"], w["data_seed"])
    o = oracle.make_cfg(kind=oracle.RESNET20, bf16=True, K=w["K"], B=w["B"], H=w["H"], T=25,
                        t_switch=12, N=w["N"], base_lr=w["base_lr"], scale_by_K=True,
                        warmup_epochs=5.0, milestones=(0.5, 0.75), momentum=0.9, nesterov=True,
                        weight_decay=w["weight_decay"], seed=w["seed"])
    wt = oracle.init_params(o)
    u = np.zeros_like(wt)
    t0 = time.perf_counter()
    steps = 0
    while True:
        idx = oracle.sample_indices(o, steps % o.K, 0)[:8]
        _, g = oracle.loss_grad(o, wt, X10, y=y10, idx=idx)
        wt, u = oracle.sgd_update(o, oracle.lr(o, 0), wt, u, g)
        steps += 1
        if time.perf_counter() - t0 > budget_s / 2:
            break
    t = time.perf_counter() - t0
    out["resnet20"] = {"workload": w["name"], "samples_per_s": 8 * steps / t,
                       "sample": f"{steps} single-replica local steps on 8 of the worker's 128 "
                                 "images plus the update of all parameters"}
    out["host"] = host_info()
    return out


def run_reference(args, world, rank):
    if rank != 0:
        return
    import synthdata

    w = WORKLOAD
    X, y = synthdata.gaussian_mixture_cached(w["N"], w["widths"][0], w["C"], w["data_seed"])
    for _ in range(args.warmup):
        oracle_sample(w, X, y, 1, ORACLE_ROWS, 1e9)
    t, samples, steps = oracle_sample(w, X, y, args.steps, ORACLE_ROWS, 1e9)
    v = samples / t
    line = {
        "impl": "reference", "metric": "samples/s over K simulated workers (1 GB300)",
        "value": v, "unit": "samples/s", "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1000.0 * t / steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(w, w["K"], world),
        "cpu_baseline": {"value": v, "unit": "samples/s", "cores": 1, "kind": "oracle",
                         "sample": oracle_sample_text(w, steps, ORACLE_ROWS)},
        "e2e": {"value": v, "unit": "samples/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_sweep(args):
    """Sync / compute trade-off: MLP 3072-512-512-10, B_loc = 32, heavy-ball momentum 0.9, 500
    local steps per (K, H) on the synthetic 10-class data; one JSON line per point with samples/s
    (device time) and the fraction of step time spent in the K-way average."""
    import torch

    import synthdata
    from paper_1808_07217_gb300 import _build

    _build.build()
    import paper_1808_07217_gb300 as P

    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream()
    N, B, widths, T = 50000, 32, (3072, 512, 512, 10), 500
    X, y = synthdata.gaussian_mixture_cached(N, 3072, 10, 1234)
    for K in (8, 32, 64):
        for H in (1, 2, 4, 8, 16, 32):
            cfg = P.make_config(K=K, B_loc=B, H=H, total_steps=T + 20, N=N, widths=widths,
                                base_lr=0.1, momentum=0.9, seed=0, precision=P.BF16,
                                fused_update=True)
            ctx = P.lsgd_create(cfg, stream=stream.cuda_stream)
            P.lsgd_set_dataset(ctx, X, y)
            P.lsgd_run(ctx, 20)
            torch.cuda.synchronize()
            P.lsgd_profile_enable(ctx, True)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            P.lsgd_run(ctx, T)
            e1.record(stream)
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1)
            prof = P.lsgd_profile_read(ctx)
            tot = sum(v[1] for v in prof.values())
            print(json.dumps({"sweep": "mlp_3072-512-512-10_B32", "K": K, "H": H, "steps": T,
                              "samples_per_s": T * K * B / (ms / 1000.0), "ms_per_step": ms / T,
                              "sync_frac": prof["average"][1] / tot,
                              "syncs": prof["average"][0]}), flush=True)
            P.lsgd_destroy(ctx)


# Algorithmic bytes per parameter and replica of one synchronisation (fp32 state, bf16 shadow),
# plus bytes per parameter of the shared vectors (w_ref, u_g: fp32):
#   plain average          : read w, write w + shadow                           = 10 | 0
#   global momentum        : the same, plus read + write w_ref and u_g          = 10 | 16
#   sign (two passes)      : read w (L1 norms), read w + write w + shadow       = 14 | 12 (w_ref read
#                            twice, written once)
#   EF-sign (two passes)   : sign's, plus read e (twice) and write e            = 26 | 12
SYNC_VARIANT_BYTES = {"plain": (10, 0), "global_momentum": (10, 16), "sign": (14, 12),
                      "ef_sign": (26, 12)}


def run_sync_variants(args):
    """Time one synchronisation of each averaging variant on the MLP 3072-1024-1024-10 parameter
    arena (K = 16 replicas of d = 4.2 M parameters; 268 MB of fp32 replicas, larger than L2): one
    JSON line per variant with ms per sync and algorithmic GB/s against the HBM peak."""
    import torch

    from paper_1808_07217_gb300 import _build

    _build.build()
    import paper_1808_07217_gb300 as P

    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream()
    hbm, _, src = _peaks()
    w = CONFIG2
    K = args.replicas or w["K"]
    n_sync = max(args.steps, 8)
    for name, extra in (("plain", {}), ("global_momentum", dict(global_momentum=0.9)),
                        ("sign", dict(compress=P.COMPRESS_SIGN)),
                        ("ef_sign", dict(compress=P.COMPRESS_EF_SIGN))):
        cfg = P.make_config(K=K, B_loc=w["B"], H=w["H"], total_steps=16, N=w["N"],
                            widths=w["widths"], base_lr=w["base_lr"], momentum=w["momentum"],
                            nesterov=w["nesterov"], weight_decay=w["weight_decay"], seed=w["seed"],
                            precision=P.BF16, **extra)
        ctx = P.lsgd_create(cfg, stream=stream.cuda_stream)
        d = P.lsgd_num_params(ctx)
        for _ in range(max(3, args.warmup)):
            P.lsgd_sync_average(ctx)
        torch.cuda.synchronize()
        n1 = P.lsgd_kernel_launches(ctx)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(n_sync):
            P.lsgd_sync_average(ctx)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / n_sync
        per_rep, shared = SYNC_VARIANT_BYTES[name]
        nbytes = per_rep * K * d + shared * d
        gbs = nbytes / (ms * 1e6)
        print(json.dumps({"sync_variant": name, "K": K, "d": d, "ms_per_sync": ms,
                          "launches_per_sync": (P.lsgd_kernel_launches(ctx) - n1) / n_sync,
                          "algorithmic_bytes": nbytes, "achieved_gbs": gbs,
                          "peak_gbs": hbm, "frac": gbs / hbm, "peak_source": src}), flush=True)
        P.lsgd_destroy(ctx)


class DenseRun:
    """A dense workload's context on the device, stepped along its job schedule: a run past the
    job's last step restarts the schedule from the model it ended with (lsgd_set_step(0) after
    the job's final average), so every timed step is a step of the configured schedule."""

    def __init__(self, P, w, stream, fused=True, K=None):
        import synthdata

        self.P, self.w = P, w
        self.K = K or w["K"]
        self.T = job_steps(w, self.K)
        self.cfg = make_gpu_cfg(P, w, fused, self.K)
        self.X, self.y = synthdata.gaussian_mixture_cached(w["N"], w["widths"][0], w["C"],
                                                           w["data_seed"])
        self.ctx = P.lsgd_create(self.cfg, stream=stream.cuda_stream)
        P.lsgd_set_dataset(self.ctx, self.X, self.y)
        self.d = P.lsgd_num_params(self.ctx)
        _, self.kinds = P.lsgd_schedule(self.cfg, self.T)
        # round-ending steps form the average inside their update launches (fused bf16 path)
        self.fuse_avg = fused and w["bf16"]
        self.fused = fused and w["bf16"]
        self.traced_steps = []

    def run_steps(self, n):
        P = self.P
        while n > 0:
            m = min(n, self.T - P.lsgd_step_count(self.ctx))
            P.lsgd_run(self.ctx, m)
            n -= m
            if P.lsgd_step_count(self.ctx) == self.T:
                P.lsgd_set_step(self.ctx, 0)

    def losses_finite(self, n):
        import numpy as np

        n = min(self.P.lsgd_step_count(self.ctx), n)
        return (not n) or bool(np.isfinite(self.P.lsgd_losses(self.ctx, n, self.K)).all())

    def time_steps(self, n, stream):
        """Device time (ms) of n steps, their kernel launches and averages."""
        import torch

        P = self.P
        n0, s0 = P.lsgd_kernel_launches(self.ctx), P.lsgd_sync_count(self.ctx)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        self.run_steps(n)
        e1.record(stream)
        torch.cuda.synchronize()
        return (e0.elapsed_time(e1), P.lsgd_kernel_launches(self.ctx) - n0,
                P.lsgd_sync_count(self.ctx) - s0)

    def traced(self, n):
        """Per-phase device times of n further steps (CUDA events around every phase)."""
        import torch

        P = self.P
        s0 = P.lsgd_step_count(self.ctx)
        self.traced_steps = [(s0 + i) % self.T for i in range(n)]
        P.lsgd_profile_enable(self.ctx, True)
        self.run_steps(n)
        torch.cuda.synchronize()
        prof = P.lsgd_profile_read(self.ctx)
        P.lsgd_profile_enable(self.ctx, False)
        return prof

    def step_bytes(self, s):
        """Algorithmic bytes of step s's update launches and of its averaging launches, per
        parameter and replica of the weight matrices (fp32 w, u; bf16 shadow):
          * plain fused update: read w, u; write w, u and the shadow = 18 B; when the replicas
            agree at the step's start (after an average) w is read once per tile: 14 + 4 / K;
          * a step that ends with the average forms it in the same launches: u read and written
            (8 B) per replica, the mean and its shadow written once (to the replica every kernel
            of the next step reads): 8 + 10 / K with the replicas agreeing at the start, else
            w read per replica: 12 + 6 / K;
        plus 2 B per element of the bf16 operands (output gradient and layer input).  A separate
        average moves 10 B per parameter and replica (read w, write w and shadow); in a fused step
        only the biases (and a classifier head updated by its own kernels) take it."""
        w, K, B = self.w, self.K, self.w["B"]
        widths = w["widths"]
        L = len(widths) - 1
        if not self.fused:
            upd = UPDATE_BYTES_PER_PARAM * K * self.d
            return upd, (AVERAGE_BYTES_PER_PARAM * K * self.d if self.kinds[s] == 2 else 0)
        head = w["bf16"] and widths[-1] <= 16
        ends = self.kinds[s] == 2 and self.fuse_avg
        synced = K > 1 and (s == 0 or self.kinds[s - 1] == 2)
        upd = 0
        for l in range(L):
            n_w = widths[l] * widths[l + 1]
            if head and l == L - 1:
                upd += FUSED_UPDATE_BYTES_PER_PARAM * K * n_w
            elif ends:
                upd += (8 * K + 10) * n_w if synced else (12 * K + 6) * n_w
            else:
                upd += (14 * K + 4) * n_w if synced else FUSED_UPDATE_BYTES_PER_PARAM * K * n_w
            upd += 2 * K * B * (widths[l] + widths[l + 1])
        if self.kinds[s] != 2:
            return upd, 0
        if not self.fuse_avg:
            return upd, AVERAGE_BYTES_PER_PARAM * K * self.d
        seg = sum(widths[1:]) + (widths[-2] * widths[-1] if head else 0)
        return upd, AVERAGE_BYTES_PER_PARAM * K * seg

    def step_kind(self, s):
        """'avg' / 'plain' (whether step s ends with the average formed in its update launches),
        with '_synced' when the replicas agree at its start."""
        ends = self.fused and self.kinds[s] == 2 and self.fuse_avg
        synced = self.K > 1 and (s == 0 or self.kinds[s - 1] == 2)
        return ("avg" if ends else "plain") + ("_synced" if synced else "")

    def traced_traffic(self):
        """Measured DRAM bytes of the traced steps' update launches (UPDATE_TRAFFIC_PER_STEP),
        or None if a step's kind has no capture."""
        table = UPDATE_TRAFFIC_PER_STEP.get(self.w["name"], {})
        if not self.fused or self.K != self.w["K"]:
            return None
        tot = 0
        for s in self.traced_steps:
            b = table.get(self.step_kind(s))
            if b is None:
                return None
            tot += b
        return tot

    def traced_bytes(self):
        """(update, average) algorithmic bytes summed over the traced steps."""
        tot = [0, 0]
        for s in self.traced_steps:
            u, a = self.step_bytes(s)
            tot[0] += u
            tot[1] += a
        return tot

    def destroy(self):
        self.P.lsgd_destroy(self.ctx)


def roofline(run, prof, steps, hbm, peak_src, fused=True):
    """The update launches' algorithmic GB/s over the traced steps, against the HBM peak."""
    upd_n, upd_ms = prof["update"]
    upd_bytes, _ = run.traced_bytes()
    upd_gbs = upd_bytes / (upd_ms / 1000.0) / 1e9
    traffic = run.traced_traffic()
    if traffic is not None:
        traffic /= steps
    n_avg = sum(1 for s in run.traced_steps if run.kinds[s] == 2)
    return {"kernel": ("wgrad_update_kernel (weight gradient + fused local update, and the K-way "
                       "average on round-ending steps)" if fused else "sgd_update_kernel"),
            "bound": "hbm", "achieved": upd_gbs, "peak": hbm, "unit": "GB/s",
            "frac": upd_gbs / hbm, "peak_source": f"{peak_src} hbm_gbs", "traffic": traffic,
            "unit_of_work": ("one step's weight-gradient + update launches (all layers), averaged "
                             f"over {steps} steps of which {n_avg} end with the K-way average"
                             if fused else "one launch over the whole K x d buffer"),
            "algorithmic_bytes": upd_bytes / steps, "launches_per_unit": upd_n // steps}


def average_phase(run, prof, hbm):
    """The averaging launches' algorithmic GB/s over the traced steps (the separate K-way average,
    or in fused steps the bias / head segments; the rest of the average is in the update)."""
    avg_n, avg_ms = prof["average"]
    _, avg_bytes = run.traced_bytes()
    if not avg_n or not avg_ms:
        return {"gbs": None, "frac_of_hbm": None, "ms_per_sync": None}
    gbs = avg_bytes / (avg_ms / 1000.0) / 1e9
    return {"gbs": gbs, "frac_of_hbm": gbs / hbm, "ms_per_sync": avg_ms / avg_n,
            "bytes_per_sync": avg_bytes / avg_n}


def run_dense_config(args, key):
    """Time one of DENSE_CONFIGS on its job schedule: W warm-up steps, S timed steps, then a
    traced pass for the per-phase split.  One JSON line."""
    import torch

    from paper_1808_07217_gb300 import _build

    _build.build()
    import paper_1808_07217_gb300 as P

    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream()
    w = DENSE_CONFIGS[key]
    if args.widths:
        # the same schedule on other layer widths (smaller cases of the same kernels for profiler
        # captures)
        widths = tuple(int(v) for v in args.widths.split(","))
        if widths[0] != w["widths"][0] or widths[-1] != w["widths"][-1]:
            raise SystemExit("--widths must keep the input width and the number of classes")
        w = dict(w, widths=widths, name=w["name"] + "_widths_" + "-".join(map(str, widths)))
    fused = w["bf16"] and not args.unfused
    run = DenseRun(P, w, stream, fused, args.replicas or None)
    S_ = args.steps
    run.run_steps(max(3, args.warmup))
    torch.cuda.synchronize()
    ms, launches, syncs = run.time_steps(S_, stream)
    finite = run.losses_finite(8)
    prof = run.traced(S_)
    hbm, _, src = _peaks()
    print(json.dumps({"workload": w["name"], "value": S_ * run.K * w["B"] / (ms / 1000.0),
                      "unit": "samples/s", "steps": S_, "ms_per_step": ms / S_,
                      "job": f"{run.T}-step schedule, repeated from its end state",
                      "syncs_in_timed_region": syncs, "gpu_launches": launches,
                      "params_per_replica": run.d, "losses_finite": finite,
                      "roofline": roofline(run, prof, S_, hbm, src, fused),
                      "sync_average": average_phase(run, prof, hbm),
                      "phase_ms_per_step": {k: v[1] / S_ for k, v in prof.items()}}), flush=True)
    run.destroy()


def run_resnet(args):
    """Post-local ResNet-20 (K = 16, B_loc = 128): the 25-step job of one epoch, H = 1 before
    t' = floor(T / 2) and H = 16 after, learning rate decayed at 50 % and 75 % of T, repeated from
    its end state; samples/s over whole jobs' steps, then the per-phase split from a traced pass.
    One JSON line."""
    import numpy as np
    import torch

    import synthdata
    from paper_1808_07217_gb300 import _build

    _build.build()
    import paper_1808_07217_gb300 as P

    torch.cuda.set_device(0)
    w = RESNET_WORKLOAD
    K, B = args.replicas or w["K"], w["B"]
    X, y = synthdata.gaussian_mixture_cached(w["N"], 3072, w["C"], w["data_seed"])
    W_, S_ = max(3, args.warmup), args.steps
    T_job = job_steps(w, K)
    stream = torch.cuda.current_stream()
    cfg = P.make_config(K=K, B_loc=B, H=w["H"], t_switch=T_job // 2, total_steps=T_job, N=w["N"],
                        kind=P.RESNET20, in_hwc=(32, 32, 3), n_classes=w["C"], base_ch=16,
                        res_blocks=3, base_lr=w["base_lr"], scale_by_K=w["scale_by_K"],
                        warmup_epochs=w["warmup_epochs"], milestones=(0.5, 0.75),
                        momentum=w["momentum"], nesterov=w["nesterov"],
                        weight_decay=w["weight_decay"], seed=w["seed"], precision=P.BF16)
    ctx = P.lsgd_create(cfg, stream=stream.cuda_stream)
    P.lsgd_set_dataset(ctx, X, y)

    def run_steps(n):
        while n > 0:
            m = min(n, T_job - P.lsgd_step_count(ctx))
            P.lsgd_run(ctx, m)
            n -= m
            if P.lsgd_step_count(ctx) == T_job:
                P.lsgd_set_step(ctx, 0)

    run_steps(W_)
    torch.cuda.synchronize()
    n0, sy0 = P.lsgd_kernel_launches(ctx), P.lsgd_sync_count(ctx)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    run_steps(S_)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    launches, syncs = P.lsgd_kernel_launches(ctx) - n0, P.lsgd_sync_count(ctx) - sy0
    n_chk = min(P.lsgd_step_count(ctx), 8)
    if n_chk and not np.isfinite(P.lsgd_losses(ctx, n_chk, K)).all():
        raise RuntimeError("non-finite loss in the timed steps")
    P.lsgd_profile_enable(ctx, True)
    run_steps(S_)
    torch.cuda.synchronize()
    prof = P.lsgd_profile_read(ctx)
    print(json.dumps({"workload": w["name"], "value": S_ * K * B / (ms / 1000.0),
                      "unit": "samples/s", "steps": S_, "ms_per_step": ms / S_,
                      "job": f"{T_job}-step schedule (t' = {T_job // 2}), repeated from its end state",
                      "syncs_in_timed_region": syncs, "gpu_launches": launches,
                      "phase_ms_per_step": {k: v[1] / S_ for k, v in prof.items()},
                      "params_per_replica": P.lsgd_num_params(ctx)}), flush=True)
    P.lsgd_destroy(ctx)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=245)
    ap.add_argument("--warmup", type=int, default=16)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="K x H sync / compute sweep of the MLP 3072-512-512-10 workload")
    ap.add_argument("--sync-variants", action="store_true",
                    help="time one synchronisation of each averaging variant (plain, global "
                         "momentum, sign, EF-sign) on the MLP 3072-1024-1024-10 K x d arena")
    ap.add_argument("--config", choices=sorted(DENSE_CONFIGS),
                    help="time one dense configuration alone (softmax regression, MLP "
                         "3072-1024-1024-10, post-local MLP 3072-4096x3-100) on its job schedule")
    ap.add_argument("--resnet", action="store_true",
                    help="post-local ResNet-20 workload (K = 16, B_loc = 128) instead of the MLP")
    ap.add_argument("--unfused", action="store_true",
                    help="apply the update with the stand-alone kernel over the whole K x d buffer "
                         "instead of the weight-gradient epilogue (same arithmetic)")
    ap.add_argument("--widths", default="",
                    help="with --config: other layer widths, e.g. 3072,2048,2048,2048,100 "
                         "(smaller cases of the same kernels for profiler captures)")
    ap.add_argument("--replicas", type=int, default=0,
                    help="override K (smaller cases for profiler captures); 0 = the workload's K")
    args = ap.parse_args()
    world, rank, local = _dist()
    if args.sweep:
        run_sweep(args)
        return
    if args.resnet:
        run_resnet(args)
        return
    if args.config:
        run_dense_config(args, args.config)
        return
    if args.sync_variants:
        run_sync_variants(args)
        return

    if args.impl == "reference":
        run_reference(args, world, rank)
        return

    import numpy as np
    import torch

    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    from paper_1808_07217_gb300 import _build

    _build.build()
    import paper_1808_07217_gb300 as P

    w = WORKLOAD
    fused = not args.unfused
    W_, S_ = max(3, args.warmup), args.steps
    e2e_warm = 2
    stream = torch.cuda.current_stream()
    run = DenseRun(P, w, stream, fused, args.replicas or None)
    K, B, T_job, ctx = run.K, w["B"], run.T, run.ctx
    _, kinds = P.lsgd_schedule(run.cfg, T_job)

    # ---- device-resident timing ----
    run.run_steps(W_)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    c0 = clocks.count()
    t_ms, launches, n_syncs = run.time_steps(S_, stream)
    if world > 1:
        torch.distributed.barrier()
    time.sleep(0.05)
    clk = clocks.stop(c0, clocks.count())
    if not run.losses_finite(16):
        raise RuntimeError("non-finite loss in the timed steps")

    # ---- the same number of steps again with per-phase CUDA events (the split and roofline) ----
    prof = run.traced(S_)
    samples_per_rank = S_ * K * B
    t_ms = max_over_ranks(t_ms, world)
    value = whole_job_throughput(samples_per_rank, t_ms / 1000.0, world)

    # ---- end to end through the C ABI with host buffers ----
    n_stage = 4
    xs, ys = [], []
    for i in range(n_stage):
        idx = P.lsgd_debug_indices(ctx, (P.lsgd_step_count(ctx) + i) % T_job, K, B).reshape(-1)
        xs.append(torch.from_numpy(run.X[idx].reshape(K, B, -1)).pin_memory())
        ys.append(torch.from_numpy(run.y[idx].reshape(K, B).copy()).pin_memory())
    # every step's K losses come back to pinned host memory; the reads are asynchronous, like the
    # host-to-device copies (which run on the library's copy stream, one batch ahead), and all
    # of them have landed when the timed region ends
    loss_host = torch.empty((max(S_, e2e_warm), K), dtype=torch.float32).pin_memory()

    def e2e_step(i):
        s = P.lsgd_step_count(ctx)
        # one step of the schedule on the host batch: the local step and the average ending it
        P.lsgd_run_batch(ctx, xs[i % n_stage], ys[i % n_stage])
        P.lsgd_losses_async(ctx, loss_host[i], 1)  # device -> host read of this step's losses
        if s + 1 == T_job:
            P.lsgd_set_step(ctx, 0)

    for i in range(e2e_warm):
        e2e_step(i)
    P.lsgd_synchronize(ctx)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    t0 = time.perf_counter()
    for i in range(S_):
        e2e_step(i)
    P.lsgd_synchronize(ctx)
    torch.cuda.synchronize()
    t_e2e = time.perf_counter() - t0
    if not bool(torch.isfinite(loss_host[:S_]).all()):
        raise RuntimeError("non-finite loss in the end-to-end steps")
    e2e_value = whole_job_throughput(samples_per_rank, t_e2e, world)
    h2d = K * B * w["widths"][0] * 4 + K * B * 4
    d2h = K * 4

    # ---- roofline of the dominant kernel (the fused update), the average, the GEMMs ----
    hbm, bf16_peak, peak_src = _peaks()
    widths = w["widths"]
    gemm_flops = 0
    for l in range(len(widths) - 1):
        mac = B * widths[l] * widths[l + 1]
        gemm_flops += 2 * mac * (3 if l > 0 else 2)
    gemm_flops *= K
    gemm_ms = (prof["forward"][1] + prof["backward"][1] + prof["update"][1]) / max(prof["forward"][0], 1)
    gemm_tflops = gemm_flops / (gemm_ms / 1000.0) / 1e12
    phase_ms = {k: v[1] for k, v in prof.items()}
    tot_phase = sum(phase_ms.values())
    run.destroy()

    # ---- config 2 (MLP 3072-1024-1024-10) on its own schedule, device time ----
    cfg2 = None
    if args.replicas == 0:
        r2 = DenseRun(P, CONFIG2, stream, fused)
        r2.run_steps(W_)
        torch.cuda.synchronize()
        ms2, launches2, syncs2 = r2.time_steps(S_, stream)
        finite2 = r2.losses_finite(16)
        prof2 = r2.traced(S_)
        cfg2 = {"workload": CONFIG2["name"], "value": S_ * r2.K * CONFIG2["B"] / (ms2 / 1000.0),
                "unit": "samples/s", "ms_per_step": ms2 / S_, "steps": S_,
                "syncs_in_timed_region": syncs2, "gpu_launches": launches2,
                "losses_finite": finite2, "roofline": roofline(r2, prof2, S_, hbm, peak_src, fused)}
        r2.destroy()

    cpu = None
    cpu_others = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        t_cpu, samples_cpu, steps_cpu = oracle_sample(w, run.X, run.y, 64, ORACLE_ROWS, 12.0)
        cpu = {"value": samples_cpu / t_cpu, "unit": "samples/s", "cores": 1, "kind": "oracle",
               "sample": oracle_sample_text(w, steps_cpu, ORACLE_ROWS)}
        cpu_others = oracle_other_configs()

    line = {
        "metric": "samples/s over K simulated workers (1 GB300)",
        "value": value, "unit": "samples/s", "n_gpus": world, "steps": S_, "warmup": W_,
        "ms_per_step": t_ms / S_, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": workload_config(w, K, world, fused),
        "syncs_in_timed_region": n_syncs,
        "first_timed_step": W_ % T_job,
        "e2e": {"value": e2e_value, "unit": "samples/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": launches,
        "roofline": roofline(run, prof, S_, hbm, peak_src, fused),
        "sync_average": average_phase(run, prof, hbm),
        "step_split": {"local_frac": 1.0 - phase_ms["average"] / tot_phase,
                       "sync_frac": phase_ms["average"] / tot_phase,
                       "phase_ms_per_step": {k: v / S_ for k, v in phase_ms.items()},
                       "note": "round-ending steps form the K-way average inside their update "
                               "launches; the average phase is then the bias / head segments"},
        "gemm": {"tflops": gemm_tflops, "frac_of_bf16_peak": gemm_tflops / bf16_peak,
                 "peak_source": f"{peak_src} bf16_tflops_sustained"},
        "clocks": clk,
        "cpu_baseline": cpu,
        "cpu_baseline_other_configs": cpu_others,
        "config2": cfg2,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
