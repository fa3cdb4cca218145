"""Pure-fp32 parity of whole local SGD steps against the oracle.

Each step starts from the oracle's own state (rounded to fp32 and imported into every GPU replica),
runs one GPU step (and the average when the schedule ends a round), and must match the oracle's
step from the same state within max relative error 1e-5 per tensor.  Workloads: the softmax
regression run (3072 -> 10, K = 4, B = 32, H = 4, plain SGD lr 0.1, 64 steps, N = 8192), a small
MLP with Nesterov momentum and weight decay on ragged tile sizes, post-local SGD, and least squares
reaching its closed-form optimum."""
import numpy as np
import pytest

import oracle
import synthdata
from _gpu_common import built_package, dense_cfgs, dense_segments, max_rel_per_tensor

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


def _stepwise_parity(P, g, o, X, y=None, t=None, widths=None, bias=True, tol=1e-5, steps=None,
                     check_every=1):
    ctx = P.lsgd_create(g)
    if t is not None:
        P.lsgd_set_targets(ctx, X, t)
    else:
        P.lsgd_set_dataset(ctx, X, y)
    d = P.lsgd_num_params(ctx)
    K = g.K
    init = oracle.INIT_HE if g.model.init == P.INIT_HE else oracle.INIT_ZERO
    Wo = np.tile(oracle.init_params(o, init), (K, 1))
    Uo = np.zeros_like(Wo)
    segs = dense_segments(widths, bias)
    worst = 0.0
    n = o.T if steps is None else steps
    syncs = 0
    for s in range(n):
        if s % check_every == 0:
            Wf, Uf = Wo.astype(np.float32), Uo.astype(np.float32)
            for k in range(K):
                P.lsgd_set_params(ctx, k, Wf[k])
                if g.momentum != 0.0:
                    P.lsgd_set_momentum(ctx, k, Uf[k])
            Wo, Uo = Wf.astype(np.float64), Uf.astype(np.float64)
        P.lsgd_run(ctx, 1)
        Wo, Uo, lo, ns = oracle.run(o, X, y=y, t=t, W=Wo, U=Uo, s0=s, n_steps=1)
        syncs += ns
        if (s + 1) % check_every == 0 or s == n - 1:
            for k in range(K):
                worst = max(worst, max_rel_per_tensor(P.lsgd_params(ctx, k), Wo[k], segs))
            lg = P.lsgd_losses(ctx, 1, K)[0]
            np.testing.assert_allclose(lg, lo[0], rtol=1e-4, atol=1e-5)
    assert P.lsgd_sync_count(ctx) == syncs
    P.lsgd_destroy(ctx)
    assert worst <= tol, worst
    return worst


def test_softmax_regression_config_stepwise(P):
    # 3072 -> 10 softmax regression, zero init, K = 4 workers over shards of 2048 points, B = 32,
    # H = 4, plain SGD with lr 0.1, 64 local steps, fp32 throughout.
    X, y = synthdata.gaussian_mixture_cached(8192, 3072, 10, 1234)
    g, o = dense_cfgs(P, widths=(3072, 10), K=4, B=32, H=4, T=64, N=8192, precision=P.FP32,
                      base_lr=0.1, seed=0, init="zero")
    _stepwise_parity(P, g, o, X, y=y, widths=(3072, 10))


@pytest.mark.parametrize("K,B,H,tp,hb", [(3, 7, 3, -1, 0), (5, 40, 2, 4, 0), (1, 9, 4, -1, 0),
                                         (4, 8, 1, 2, 2)])
def test_mlp_momentum_stepwise(P, K, B, H, tp, hb):
    widths = (50, 72, 36, 13)
    N = 400
    rng = np.random.default_rng(K * 10 + B)
    X = rng.standard_normal((N, widths[0])).astype(np.float32)
    y = rng.integers(0, widths[-1], N).astype(np.int32)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=H, T=10, N=N, precision=P.FP32, t_switch=tp,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=4,
                      scale_by_K=True, warmup_epochs=1.0, milestones=(0.5, 0.75),
                      hier_block=hb, hier_rounds=3 if hb else 1)
    _stepwise_parity(P, g, o, X, y=y, widths=widths)


def test_mlp_heavy_ball_multi_step_drift(P):
    # Several steps without re-import: fp32 drift stays far below bf16-level differences.
    widths = (64, 48, 10)
    N = 256
    rng = np.random.default_rng(1)
    X = rng.standard_normal((N, 64)).astype(np.float32)
    y = rng.integers(0, 10, N).astype(np.int32)
    g, o = dense_cfgs(P, widths=widths, K=4, B=16, H=4, T=16, N=N, precision=P.FP32,
                      base_lr=0.05, momentum=0.9, seed=9)
    _stepwise_parity(P, g, o, X, y=y, widths=widths, check_every=16, tol=1e-4)


def test_least_squares_parity_and_optimum(P):
    N, dd = 512, 20
    A, t, _ = synthdata.least_squares(N, dd, seed=7)
    g, o = dense_cfgs(P, widths=(dd, 1), K=4, B=16, H=8, T=1600, N=N, precision=P.FP32,
                      kind="lsq", base_lr=0.02, seed=5, init="zero")
    _stepwise_parity(P, g, o, A, t=t, widths=(dd, 1), bias=False, steps=24)
    ctx = P.lsgd_create(g)
    P.lsgd_set_targets(ctx, A, t)
    P.lsgd_run(ctx, 1600)
    w = P.lsgd_params(ctx, -1).astype(np.float64)
    w_opt = np.linalg.lstsq(A.astype(np.float64), t.astype(np.float64), rcond=None)[0]
    assert np.linalg.norm(w - w_opt) / np.linalg.norm(w_opt) <= 1e-5
    assert P.lsgd_sync_count(ctx) == 1600 // 8
    P.lsgd_destroy(ctx)
