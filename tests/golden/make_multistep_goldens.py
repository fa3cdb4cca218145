#!/usr/bin/env python3
"""Write the oracle's results for the multi-step bf16 parity tests (tests/test_gpu_multistep.py).

For each case below the oracle (oracle/, fp64) runs local or post-local SGD (Eq. 2; Algorithms 1
and 2) for T steps on the configured synthetic dataset from its own initial model -- with the
GEMM operands rounded to bf16 as the accelerated path stores them, and (--fp32) without that
rounding -- and this script stores, in tests/golden/multistep_<case>.npz (multistep_<case>_fp32.npz):

  w_sub      the final averaged parameters at every `stride`-th canonical index (fp32)
  norm_full  the fp64 L2 norm of all final parameters
  losses     per-step mean mini-batch loss of every worker, [T][K]
  eval_loss  the mean loss of the final model over the first n_eval dataset rows
  syncs      the number of averages the schedule performed

The bf16 and fp32 results together measure how much the method's own trajectory moves when only
the rounding of the products changes: at the configured learning rates of the dense networks
(e.g. 0.1 with momentum 0.9) that is several per cent after 64 steps, the regime is chaotic, and
no implementation that rounds in another order can be held closer to the oracle than that.  The
"_lr002" cases run the same networks and schedules at learning rate 0.02, where the two differ
by about 1 % and the 2e-2 bar applies as stated.

The networks are those of the configurations (MLP 3072-1024-1024-10, MLP 3072-512-512-10,
MLP 3072-4096-4096-4096-100, ResNet-20 on 32x32x3 images) at fewer workers and, where the
oracle's cost requires it, smaller local batches.  Only the oracle and the input generator run
here.  Usage: python tests/golden/make_multistep_goldens.py [--fp32] [case ...]
"""
from __future__ import annotations

import json
import multiprocessing as mp
import os
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

N_DATA, DATA_SEED = 50000, 1234

_MLP1024 = dict(kind="mlp", widths=(3072, 1024, 1024, 10), C=10, K=2, B=128, H=16, T=64,
                t_switch=-1, base_lr=0.1, scale_by_K=True, warmup_epochs=5.0, milestones=(),
                momentum=0.9, nesterov=True, weight_decay=5e-4, seed=0, stride=64, n_eval=8192,
                bar="sensitivity")
_MLP512 = dict(kind="mlp", widths=(3072, 512, 512, 10), C=10, K=8, B=32, H=4, T=64, t_switch=-1,
               base_lr=0.1, scale_by_K=False, warmup_epochs=0.0, milestones=(), momentum=0.9,
               nesterov=False, weight_decay=0.0, seed=0, stride=32, n_eval=8192,
               bar="sensitivity")
_MLP4096 = dict(kind="mlp", widths=(3072, 4096, 4096, 4096, 100), C=100, K=2, B=32, H=16, T=64,
                t_switch=32, base_lr=0.02, scale_by_K=False, warmup_epochs=0.0,
                milestones=(0.5, 0.75), momentum=0.9, nesterov=True, weight_decay=5e-4, seed=0,
                stride=512, n_eval=2048, bar="strict")

CASES = {
    # MLP 3072-1024-1024-10 with its configured schedule (lr 0.1 scaled by K with a 5-epoch
    # warm-up, Nesterov 0.9, weight decay 5e-4, H = 16) at K = 2: four rounds, four averages
    "mlp1024_K2": _MLP1024,
    "mlp1024_K2_lr002": dict(_MLP1024, base_lr=0.02, bar="strict"),
    # the K x H sweep network (B = 32, heavy-ball 0.9, lr 0.1) at K = 8, H = 4
    "mlp512_K8": _MLP512,
    "mlp512_K8_lr002": dict(_MLP512, base_lr=0.02, bar="strict"),
    # post-local SGD on MLP 3072-4096-4096-4096-100 with its configured schedule shape (H = 1
    # before t' = T / 2, H = 16 after, decays 10x at 50 % and 75 %) at K = 2, B = 32.  Only at
    # learning rate 0.02: with the configured 0.1 the oracle itself reaches NaN at this local batch
    # (a quarter of the configured 128, which the oracle's cost rules out: ~1 h for 64 steps here)
    "mlp4096_K2_lr002": _MLP4096,
    # post-local ResNet-20 (16/32/64 channels, option-A shortcuts, per-worker BatchNorm) at K = 2,
    # B = 16, H = 4 after t' = 16, Nesterov 0.9, weight decay 1e-4, learning rate 0.02
    "resnet20_K2": dict(kind="resnet", C=10, K=2, B=16, H=4, T=64, t_switch=16, base_lr=0.02,
                        scale_by_K=False, warmup_epochs=0.0, milestones=(0.5, 0.75),
                        momentum=0.9, nesterov=True, weight_decay=1e-4, seed=0, stride=1,
                        n_eval=512, bar="strict"),
}


def oracle_cfg(oracle, c, bf16=True):
    common = dict(bf16=bf16, K=c["K"], B=c["B"], H=c["H"], t_switch=c["t_switch"], T=c["T"],
                  N=N_DATA, base_lr=c["base_lr"], scale_by_K=c["scale_by_K"],
                  warmup_epochs=c["warmup_epochs"], milestones=c["milestones"],
                  momentum=c["momentum"], nesterov=c["nesterov"], weight_decay=c["weight_decay"],
                  seed=c["seed"])
    if c["kind"] == "resnet":
        return oracle.make_cfg(kind=oracle.RESNET20, in_hwc=(32, 32, 3), n_classes=c["C"],
                               base_ch=16, res_blocks=3, **common)
    return oracle.make_cfg(widths=c["widths"], **common)


def path_of(name, fp32=False):
    return os.path.join(HERE, f"multistep_{name}{'_fp32' if fp32 else ''}.npz")


def make(job):
    import numpy as np

    import oracle
    import synthdata

    name, fp32 = job
    c = CASES[name]
    X, y = synthdata.gaussian_mixture_cached(N_DATA, 3072, c["C"], DATA_SEED)
    o = oracle_cfg(oracle, c, bf16=not fp32)
    w0 = oracle.init_params(o).astype(np.float32).astype(np.float64)
    t0 = time.time()
    W, _, losses, syncs = oracle.run(o, X, y=y, W=np.tile(w0, (c["K"], 1)))
    w = W[0]
    ev = oracle.eval_loss(o, w, X, y=y, n=c["n_eval"])
    np.savez(path_of(name, fp32), w_sub=w[::c["stride"]].astype(np.float32),
             norm_full=np.float64(np.linalg.norm(w)), losses=losses.astype(np.float32),
             eval_loss=np.float64(ev), syncs=np.int64(syncs), case=json.dumps(c))
    return (f"{name}{' fp32' if fp32 else ''}: {time.time() - t0:.0f} s, {syncs} averages, eval loss {ev:.4f}, mean loss "
            f"first/last {losses[0].mean():.4f} / {losses[-1].mean():.4f}, finite "
            f"{bool(np.isfinite(losses).all())}")


def main():
    args = sys.argv[1:]
    fp32 = "--fp32" in args
    names = [a for a in args if a != "--fp32"] or list(CASES)
    jobs = [(n, fp32) for n in names]
    ctx = mp.get_context("spawn")
    with ctx.Pool(min(len(jobs), os.cpu_count() or 1)) as pool:
        for line in pool.imap_unordered(make, jobs):
            print(line, flush=True)


if __name__ == "__main__":
    main()
