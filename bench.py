#!/usr/bin/env python3
"""Throughput of local SGD over K simulated workers on one GB300 (samples/s).

Workload: MLP 3072-1024-1024-10 (ReLU, He-normal init), bf16 GEMM operands with fp32 accumulation
and fp32 master weights, K = 16 workers, B_loc = 128, H = 16, Nesterov momentum 0.9 kept local,
weight decay 5e-4, lr 0.1 scaled by K with 5-epoch linear warm-up, on N = 50,000 synthetic
CIFAR-shaped Gaussian-mixture points (32x32x3, 10 classes).  One timed step = one local step of all
K replicas (sampling, gather + cast, forward, loss, backward, fused update) plus, every H-th step,
the K-way average.  `value` is device-timed with inputs resident in HBM; `e2e` drives the same
steps through lsgd_local_step_batch with each step's mini-batch copied from pinned host memory and
its losses read back.

--impl reference times the oracle (single-threaded C++, fp64) on the host cores instead.
Under torchrun (N > 1) every rank runs an independent replica of the workload (no collective on the
data path); the time is the maximum over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = dict(name="mlp_3072-1024-1024-10_K16_B128_H16_bf16", widths=(3072, 1024, 1024, 10),
                K=16, B=128, H=16, N=50000, C=10, base_lr=0.1, scale_by_K=True, warmup_epochs=5.0,
                momentum=0.9, nesterov=True, weight_decay=5e-4, seed=0, data_seed=1234,
                epochs=2.0)


def job_steps(w, K=None):
    """T of one training job: ceil(epochs * N / (K * B_loc)) local steps (49 for the workload)."""
    K = K or w["K"]
    return -(-int(w["epochs"] * w["N"]) // (K * w["B"]))

# Bytes the algorithm moves per parameter and replica (fp32 w, u, g; bf16 shadow):
#   stand-alone update           = read g, w, u + write w, u (4 B each) + write the shadow (2 B) = 22
#   update fused into the weight-gradient epilogue = read w, u + write w, u + write shadow = 18,
#     plus the bf16 operands it reads (activations and output gradients, 2 B each)
#   average = read w + write w (4 B each) + write bf16 shadow (2 B) = 10
UPDATE_BYTES_PER_PARAM = 22
FUSED_UPDATE_BYTES_PER_PARAM = 18
AVERAGE_BYTES_PER_PARAM = 10
# DRAM bytes (read + write) per step of the update launches (the classifier head's backward and
# the weight-gradient + update launch of both hidden layers), from the ncu capture summarised in
# profiles/step_kernels_mlp3072_K16_B128.md (below the algorithmic bytes because part of the
# launch's writes is still in L2 when it ends).
UPDATE_TRAFFIC_PER_STEP = 1186195456

FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0


def dense_params(widths):
    """Parameters per replica of a dense network: weights and biases of every layer."""
    return sum(a * b + b for a, b in zip(widths[:-1], widths[1:]))


def workload_config(w, K, world, fused=True):
    """The workload description both arms print (the timed region's own facts are added by the
    GPU arm)."""
    B, H, T_job = w["B"], w["H"], job_steps(w, K)
    return {"workload": w["name"] if K == w["K"] else w["name"].replace("K16", f"K{K}"),
            "global_batch": K * B, "K": K, "B_loc": B, "H": H, "fused_update": fused,
            "job": f"{T_job}-step schedule ({w['epochs']:g} epochs of N = {w['N']}), "
                   "repeated from its end state",
            "params_per_replica": dense_params(w["widths"]),
            "parallelism": "replicas" if world > 1 else "single",
            "l2": "per-step working set (w, u, g, shadow: 1.0 GB) exceeds the 129 MB L2"}


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


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while a timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.dev)],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
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
        return summarise_clocks(lines)


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


def _make_cfg(P, total_steps, fused=True, K=None):
    w = WORKLOAD
    return P.make_config(K=K or w["K"], B_loc=w["B"], H=w["H"], total_steps=total_steps, N=w["N"],
                         widths=w["widths"], base_lr=w["base_lr"], scale_by_K=w["scale_by_K"],
                         warmup_epochs=w["warmup_epochs"], momentum=w["momentum"],
                         nesterov=w["nesterov"], weight_decay=w["weight_decay"], seed=w["seed"],
                         precision=P.BF16, fused_update=fused)


def _oracle_cfg(oracle, total_steps):
    w = WORKLOAD
    return oracle.make_cfg(widths=w["widths"], bf16=True, K=w["K"], B=w["B"], H=w["H"],
                           T=total_steps, N=w["N"], base_lr=w["base_lr"],
                           scale_by_K=w["scale_by_K"], warmup_epochs=w["warmup_epochs"],
                           momentum=w["momentum"], nesterov=w["nesterov"],
                           weight_decay=w["weight_decay"], seed=w["seed"])


def oracle_sample(X, y, replica_steps: int, rows: int, budget_s: float):
    """Time the oracle on `replica_steps` local steps of single replicas (first `rows` rows of each
    worker's mini-batch, then the update of all parameters).  Returns (seconds, samples, steps)."""
    import numpy as np

    import oracle

    o = _oracle_cfg(oracle, 1 << 20)
    w = oracle.init_params(o)
    u = np.zeros_like(w)
    t0 = time.perf_counter()
    done = 0
    for i in range(replica_steps):
        idx = oracle.sample_indices(o, i % o.K, i // o.K)[:rows]
        _, g = oracle.loss_grad(o, w, X, y=y, idx=idx)
        w, u = oracle.sgd_update(o, oracle.lr(o, i // o.K), w, u, g)
        done += 1
        if time.perf_counter() - t0 > budget_s:
            break
    return time.perf_counter() - t0, done * rows, done


def run_reference(args, world, rank):
    if rank != 0:
        return
    import synthdata

    w = WORKLOAD
    X, y = synthdata.gaussian_mixture_cached(w["N"], w["widths"][0], w["C"], w["data_seed"])
    rows = 32
    for _ in range(args.warmup):
        oracle_sample(X, y, 1, rows, 1e9)
    t, samples, steps = oracle_sample(X, y, args.steps, rows, 1e9)
    v = samples / t
    sample = (f"{steps} single-replica local steps, each on {rows} of the worker's {w['B']} "
              f"mini-batch rows plus the update of all parameters")
    line = {
        "impl": "reference", "metric": "samples/s over K simulated workers (1 GB300)",
        "value": v, "unit": "samples/s", "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1000.0 * t / steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(w, w["K"], world),
        "cpu_baseline": {"value": v, "unit": "samples/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
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
    """Time one synchronisation of each averaging variant on the MLP workload's parameter arena
    (K = 16 replicas of d = 4.2 M parameters; 268 MB of fp32 replicas, larger than L2): one JSON
    line per variant with ms per sync and algorithmic GB/s against the HBM peak."""
    import torch

    from paper_1808_07217_gb300 import _build

    _build.build()
    import paper_1808_07217_gb300 as P

    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream()
    hbm, _, src = _peaks()
    w = WORKLOAD
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


# The other dense configurations, timed on their own job schedules (one JSON line each):
#   softmax regression 3072 -> 10, fp32, zero init, K = 4 shards of 2,048 of N = 8,192 points,
#     B_loc = 32, H = 4, plain SGD lr 0.1, a 64-step job;
#   post-local MLP 3072-4096-4096-4096-100, bf16, K = 16, B_loc = 128, 10 epochs of N = 50,000
#     (245 steps), H = 1 before t' = 122 and 16 after, Nesterov 0.9, weight decay 5e-4, lr 0.1
#     scaled by K with a 5-epoch warm-up, decayed 10x at 50 % and 75 %.
DENSE_CONFIGS = {
    "softmax": dict(name="softmax_3072-10_K4_B32_H4_fp32", widths=(3072, 10), K=4, B=32, H=4,
                    N=8192, C=10, T=64, t_switch=-1, base_lr=0.1, scale_by_K=False,
                    warmup_epochs=0.0, milestones=(), momentum=0.0, nesterov=False,
                    weight_decay=0.0, init="zero", bf16=False, seed=0, data_seed=1234),
    "mlp4096": dict(name="mlp_3072-4096x3-100_K16_B128_postlocal_H16_bf16",
                    widths=(3072, 4096, 4096, 4096, 100), K=16, B=128, H=16, N=50000, C=100,
                    T=245, t_switch=122, base_lr=0.1, scale_by_K=True, warmup_epochs=5.0,
                    milestones=(0.5, 0.75), momentum=0.9, nesterov=True, weight_decay=5e-4,
                    init="he", bf16=True, seed=0, data_seed=1234),
}


def run_dense_config(args, key):
    """Time one of DENSE_CONFIGS: W warm-up steps, then S timed steps of its job schedule
    (repeated from its end state, as for the benchmark workload), then a traced pass for the
    per-phase split.  One JSON line with samples/s, ms per step, the syncs and launches in the
    timed region and the update phase's algorithmic HBM throughput."""
    import numpy as np
    import torch

    import synthdata
    from paper_1808_07217_gb300 import _build

    _build.build()
    import paper_1808_07217_gb300 as P

    torch.cuda.set_device(0)
    w = DENSE_CONFIGS[key]
    K, B, T = w["K"], w["B"], w["T"]
    X, y = synthdata.gaussian_mixture_cached(w["N"], w["widths"][0], w["C"], w["data_seed"])
    W_, S_ = max(3, args.warmup), args.steps
    fused = w["bf16"]
    cfg = P.make_config(K=K, B_loc=B, H=w["H"], t_switch=w["t_switch"], total_steps=T, N=w["N"],
                        widths=w["widths"], init=P.INIT_ZERO if w["init"] == "zero" else P.INIT_HE,
                        base_lr=w["base_lr"], scale_by_K=w["scale_by_K"],
                        warmup_epochs=w["warmup_epochs"], milestones=w["milestones"],
                        momentum=w["momentum"], nesterov=w["nesterov"],
                        weight_decay=w["weight_decay"], seed=w["seed"],
                        precision=P.BF16 if w["bf16"] else P.FP32, fused_update=fused)
    stream = torch.cuda.current_stream()
    ctx = P.lsgd_create(cfg, stream=stream.cuda_stream)
    P.lsgd_set_dataset(ctx, X, y)
    d = P.lsgd_num_params(ctx)

    def run_steps(n):
        while n > 0:
            m = min(n, T - P.lsgd_step_count(ctx))
            P.lsgd_run(ctx, m)
            n -= m
            if P.lsgd_step_count(ctx) == T:
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
    losses = P.lsgd_losses(ctx, n_chk, K) if n_chk else np.zeros(1)
    P.lsgd_profile_enable(ctx, True)
    run_steps(S_)
    torch.cuda.synchronize()
    prof = P.lsgd_profile_read(ctx)
    hbm, _, src = _peaks()
    widths = w["widths"]
    if fused:
        upd_bytes = sum(FUSED_UPDATE_BYTES_PER_PARAM * K * widths[l] * widths[l + 1]
                        + 2 * K * B * (widths[l] + widths[l + 1]) for l in range(len(widths) - 1))
    else:
        upd_bytes = UPDATE_BYTES_PER_PARAM * K * d
    upd_ms = prof["update"][1] / S_
    print(json.dumps({"workload": w["name"], "value": S_ * K * B / (ms / 1000.0),
                      "unit": "samples/s", "steps": S_, "ms_per_step": ms / S_,
                      "job": f"{T}-step schedule, repeated from its end state",
                      "syncs_in_timed_region": syncs, "gpu_launches": launches,
                      "params_per_replica": d, "losses_finite": bool(np.isfinite(losses).all()),
                      "update_phase": {"ms_per_step": upd_ms, "algorithmic_bytes": upd_bytes,
                                       "gbs": upd_bytes / (upd_ms * 1e6) if upd_ms else None,
                                       "frac_of_hbm": (upd_bytes / (upd_ms * 1e6) / hbm)
                                       if upd_ms else None, "peak_source": f"{src} hbm_gbs"},
                      "phase_ms_per_step": {k: v[1] / S_ for k, v in prof.items()}}), flush=True)
    P.lsgd_destroy(ctx)


RESNET_WORKLOAD = dict(name="resnet20_K16_B128_postlocal_H16_bf16", K=16, B=128, H=16, N=50000,
                       C=10, base_lr=0.2, scale_by_K=True, warmup_epochs=5.0, momentum=0.9,
                       nesterov=True, weight_decay=1e-4, seed=0, data_seed=1234, epochs=1.0)


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
    ap.add_argument("--steps", type=int, default=48)
    ap.add_argument("--warmup", type=int, default=16)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="K x H sync / compute sweep of the MLP 3072-512-512-10 workload")
    ap.add_argument("--sync-variants", action="store_true",
                    help="time one synchronisation of each averaging variant (plain, global "
                         "momentum, sign, EF-sign) on the MLP workload's K x d arena")
    ap.add_argument("--config", choices=sorted(DENSE_CONFIGS),
                    help="time another dense configuration (softmax regression, post-local "
                         "MLP 3072-4096x3-100) on its job schedule")
    ap.add_argument("--resnet", action="store_true",
                    help="post-local ResNet-20 workload (K = 16, B_loc = 128) instead of the MLP")
    ap.add_argument("--unfused", action="store_true",
                    help="apply the update with the stand-alone kernel over the whole K x d buffer "
                         "instead of the weight-gradient epilogue (same arithmetic)")
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

    import synthdata

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
    K, B, H = args.replicas or w["K"], w["B"], w["H"]
    fused = not args.unfused
    X, y = synthdata.gaussian_mixture_cached(w["N"], w["widths"][0], w["C"], w["data_seed"])
    W_, S_ = max(3, args.warmup), args.steps
    e2e_warm = 2
    # The workload is a T-step job (2 epochs: 49 steps, the learning rate still warming up toward
    # K x 0.1); longer runs repeat it from the model it ended with (lsgd_set_step(0) after the
    # job's last step and its final average), so every timed step is a step of that schedule.
    T_job = job_steps(w, K)
    cfg = _make_cfg(P, T_job, fused, K)
    _, kinds = P.lsgd_schedule(cfg, T_job)
    stream = torch.cuda.current_stream()
    ctx = P.lsgd_create(cfg, stream=stream.cuda_stream)
    P.lsgd_set_dataset(ctx, X, y)
    d = P.lsgd_num_params(ctx)

    def run_steps(n):
        while n > 0:
            m = min(n, T_job - P.lsgd_step_count(ctx))
            P.lsgd_run(ctx, m)
            n -= m
            if P.lsgd_step_count(ctx) == T_job:
                P.lsgd_set_step(ctx, 0)

    # ---- device-resident timing ----
    run_steps(W_)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    n0 = P.lsgd_kernel_launches(ctx)
    syncs0 = P.lsgd_sync_count(ctx)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    run_steps(S_)
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    t_ms = e0.elapsed_time(e1)
    launches = P.lsgd_kernel_launches(ctx) - n0
    n_syncs = P.lsgd_sync_count(ctx) - syncs0
    clk = clocks.stop()

    # ---- the same number of steps again with per-phase CUDA events (the split and roofline) ----
    n_chk = min(P.lsgd_step_count(ctx), 16)
    if n_chk and not np.isfinite(P.lsgd_losses(ctx, n_chk, K)).all():
        raise RuntimeError("non-finite loss in the timed steps")
    P.lsgd_profile_enable(ctx, True)
    run_steps(S_)
    torch.cuda.synchronize()
    prof = P.lsgd_profile_read(ctx)
    P.lsgd_profile_enable(ctx, False)
    samples_per_rank = S_ * K * B
    t_ms = max_over_ranks(t_ms, world)
    value = whole_job_throughput(samples_per_rank, t_ms / 1000.0, world)

    # ---- end to end through the C ABI with host buffers ----
    rng = np.random.default_rng(0)
    n_stage = 4
    xs, ys = [], []
    for i in range(n_stage):
        idx = P.lsgd_debug_indices(ctx, (P.lsgd_step_count(ctx) + i) % T_job, K, B).reshape(-1)
        xs.append(torch.from_numpy(X[idx].reshape(K, B, -1)).pin_memory())
        ys.append(torch.from_numpy(y[idx].reshape(K, B).copy()).pin_memory())
    del rng
    # every step's K losses come back to pinned host memory; the reads are asynchronous, like the
    # host-to-device copies (which run on the library's copy stream, one batch ahead), and all
    # of them have landed when the timed region ends
    loss_host = torch.empty((max(S_, e2e_warm), K), dtype=torch.float32).pin_memory()

    def e2e_step(i):
        s = P.lsgd_step_count(ctx)
        P.lsgd_local_step_batch(ctx, xs[i % n_stage], ys[i % n_stage])
        if kinds[s] == 2:  # the round ends with this step (the schedule of lsgd_run)
            P.lsgd_sync_average(ctx)
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

    # ---- roofline of the dominant kernel (the fused update) ----
    hbm, bf16_peak, peak_src = _peaks()
    upd_n, upd_ms = prof["update"]
    avg_n, avg_ms = prof["average"]
    widths = w["widths"]
    # The update phase is each step's fused update launches (the head's backward, then one
    # weight-gradient + update launch over both hidden layers); the roofline unit is one step's
    # worth of them (bytes summed over the layers).
    if fused:
        upd_bytes = sum(FUSED_UPDATE_BYTES_PER_PARAM * K * widths[l] * widths[l + 1]
                        + 2 * K * B * (widths[l] + widths[l + 1]) for l in range(len(widths) - 1))
    else:
        upd_bytes = UPDATE_BYTES_PER_PARAM * K * d
    upd_gbs = upd_bytes / (upd_ms / S_ / 1000.0) / 1e9
    avg_gbs = (AVERAGE_BYTES_PER_PARAM * K * d / (avg_ms / avg_n / 1000.0) / 1e9) if avg_n else None
    gemm_flops = 0
    for l in range(len(widths) - 1):
        mac = B * widths[l] * widths[l + 1]
        gemm_flops += 2 * mac * (3 if l > 0 else 2)
    gemm_flops *= K
    gemm_ms = (prof["forward"][1] + prof["backward"][1] + prof["update"][1]) / max(prof["forward"][0], 1)
    gemm_tflops = gemm_flops / (gemm_ms / 1000.0) / 1e12
    phase_ms = {k: v[1] for k, v in prof.items()}
    tot_phase = sum(phase_ms.values())

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        t_cpu, samples_cpu, steps_cpu = oracle_sample(X, y, 64, B, 15.0)
        cpu = {"value": samples_cpu / t_cpu, "unit": "samples/s", "cores": 1, "kind": "oracle",
               "sample": f"{steps_cpu} single-replica local steps of the workload (B = {B} rows "
                         f"each, forward, backward and update) timed on one host core"}

    line = {
        "metric": "samples/s over K simulated workers (1 GB300)",
        "value": value, "unit": "samples/s", "n_gpus": world, "steps": S_, "warmup": W_,
        "ms_per_step": t_ms / S_, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(workload_config(w, K, world, fused), syncs_in_timed_region=n_syncs),
        "e2e": {"value": e2e_value, "unit": "samples/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": launches,
        "roofline": {"kernel": ("wgrad_update_kernel (weight gradient + fused local update)"
                                if fused else "sgd_update_kernel"),
                     "bound": "hbm", "achieved": upd_gbs, "peak": hbm, "unit": "GB/s",
                     "frac": upd_gbs / hbm, "peak_source": f"{peak_src} hbm_gbs",
                     "traffic": UPDATE_TRAFFIC_PER_STEP if fused and K == w["K"] else None,
                     "unit_of_work": ("one step's fused weight-gradient + update launches "
                                      "(3 layers: the head's backward, one launch for the rest)"
                                      if fused else "one launch over the whole K x d buffer"),
                     "algorithmic_bytes": upd_bytes, "launches_per_unit": upd_n // S_},
        "sync_average": {"gbs": avg_gbs, "frac_of_hbm": (avg_gbs / hbm) if avg_gbs else None,
                         "ms_per_sync": (avg_ms / avg_n) if avg_n else None},
        "step_split": {"local_frac": 1.0 - phase_ms["average"] / tot_phase,
                       "sync_frac": phase_ms["average"] / tot_phase,
                       "phase_ms_per_step": {k: v / S_ for k, v in phase_ms.items()}},
        "gemm": {"tflops": gemm_tflops, "frac_of_bf16_peak": gemm_tflops / bf16_peak,
                 "peak_source": f"{peak_src} bf16_tflops_sustained"},
        "clocks": clk,
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    P.lsgd_destroy(ctx)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
