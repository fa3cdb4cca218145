"""Shared helpers of the GPU tests: build once, matching GPU / oracle configurations, comparisons."""
import numpy as np

import oracle


def built_package():
    from paper_1808_07217_gb300 import _build

    _build.build()
    oracle.build()
    import paper_1808_07217_gb300 as P

    P.lib()
    return P


def dense_cfgs(P, *, widths, K, B, H, T, N, precision, kind="mlp", t_switch=-1, base_lr=0.1,
               scale_by_K=False, warmup_epochs=0.0, milestones=(), momentum=0.0, nesterov=False,
               weight_decay=0.0, seed=0, init="he", fused_update=False, hier_block=0,
               hier_rounds=1, compress=0, global_momentum=0.0, h_warmup=0, h_warmup_epochs=0.0,
               sampling=0):
    """The same run described for the GPU library and for the oracle."""
    gk = {"mlp": P.MLP, "lsq": P.LSQ}[kind]
    ok = {"mlp": oracle.DENSE, "lsq": oracle.LSQ}[kind]
    g = P.make_config(K=K, B_loc=B, H=H, t_switch=t_switch, total_steps=T, N=N, kind=gk,
                      widths=widths, init=P.INIT_HE if init == "he" else P.INIT_ZERO,
                      base_lr=base_lr, scale_by_K=scale_by_K, warmup_epochs=warmup_epochs,
                      milestones=milestones, momentum=momentum, nesterov=nesterov,
                      weight_decay=weight_decay, seed=seed, precision=precision,
                      fused_update=fused_update, hier_block=hier_block, hier_rounds=hier_rounds,
                      compress=compress, global_momentum=global_momentum, h_warmup=h_warmup,
                      h_warmup_epochs=h_warmup_epochs, sampling=sampling)
    o = oracle.make_cfg(kind=ok, widths=widths, has_bias=(kind == "mlp"),
                        bf16=(precision == P.BF16), K=K, B=B, H=H, t_switch=t_switch, T=T, N=N,
                        base_lr=base_lr, scale_by_K=scale_by_K, warmup_epochs=warmup_epochs,
                        milestones=milestones, momentum=momentum, nesterov=nesterov,
                        weight_decay=weight_decay, seed=seed, hier_block=hier_block,
                        hier_rounds=hier_rounds, compress=compress,
                        global_momentum=global_momentum, h_warmup=h_warmup,
                        h_warmup_epochs=h_warmup_epochs, sampling=sampling)
    return g, o


def dense_segments(widths, bias=True):
    """(offset, length) of every tensor in the canonical parameter order."""
    segs, off = [], 0
    for i in range(len(widths) - 1):
        n = widths[i] * widths[i + 1]
        segs.append((off, n))
        off += n
        if bias:
            segs.append((off, widths[i + 1]))
            off += widths[i + 1]
    return segs


def max_rel_per_tensor(a, o, segs):
    """max over tensors of max_i |a_i - o_i| / max_i |o_i| (cancellation-free normalisation)."""
    worst = 0.0
    for off, n in segs:
        x, y = a[off:off + n].astype(np.float64), o[off:off + n]
        den = max(np.abs(y).max(), 1e-30)
        worst = max(worst, float(np.abs(x - y).max() / den))
    return worst


def rel_l2(a, o):
    return float(np.linalg.norm(np.asarray(a, np.float64) - o) / max(np.linalg.norm(o), 1e-30))
