"""Local-step warm-up and the reshuffling sampler on the GPU against the oracle: indices bit-exact
(the full-size 50,000-point, K = 16, B = 128 layout at epoch boundaries and a ragged layout over
whole epochs), whole runs per step at the fp32 bar (1e-5 per tensor) with the oracle's sync
counts, and a bf16 run at the bf16 bar."""
import numpy as np
import pytest

import oracle
import synthdata
from _gpu_common import built_package, dense_cfgs, dense_segments, max_rel_per_tensor, rel_l2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


def test_reshuffle_indices_full_size_epoch_boundaries(P):
    N, K, B = 50000, 16, 128
    g, o = dense_cfgs(P, widths=(16, 4), K=K, B=B, H=16, T=2000, N=N, precision=P.FP32,
                      seed=0x1234567890ABCDEF, sampling=P.SAMPLE_RESHUFFLE)
    ctx = P.lsgd_create(g)
    steps_per_epoch = N / (K * B)
    picks = set()
    for e in range(0, 80, 7):
        first = int(np.ceil(e * steps_per_epoch))
        picks.update({first - 1, first, first + 1, first + 23})
    for s in sorted(p for p in picks if p >= 0):
        got = P.lsgd_debug_indices(ctx, s, K, B)
        want = np.stack([oracle.sample_indices(o, k, s) for k in range(K)])
        assert np.array_equal(got, want), s
    P.lsgd_destroy(ctx)


def test_reshuffle_indices_ragged_whole_epochs(P):
    N, K, B = 1000, 3, 7
    g, o = dense_cfgs(P, widths=(16, 4), K=K, B=B, H=4, T=200, N=N, precision=P.FP32, seed=77,
                      sampling=P.SAMPLE_RESHUFFLE)
    ctx = P.lsgd_create(g)
    for s in range(150):  # epochs 0, 1, 2 and part of 3
        got = P.lsgd_debug_indices(ctx, s, K, B)
        want = np.stack([oracle.sample_indices(o, k, s) for k in range(K)])
        assert np.array_equal(got, want), s
    P.lsgd_destroy(ctx)


def _stepwise(P, g, o, X, y, widths, steps, tol=1e-5):
    K = g.K
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    segs = dense_segments(widths)
    Wo = np.tile(oracle.init_params(o), (K, 1))
    Uo = np.zeros_like(Wo)
    worst, syncs = 0.0, 0
    for s in range(steps):
        Wf, Uf = Wo.astype(np.float32), Uo.astype(np.float32)
        for k in range(K):
            P.lsgd_set_params(ctx, k, Wf[k])
            if g.momentum != 0.0:
                P.lsgd_set_momentum(ctx, k, Uf[k])
        P.lsgd_run(ctx, 1)
        Wo, Uo, lo, ns = oracle.run(o, X, y=y, W=Wf.astype(np.float64), U=Uf.astype(np.float64),
                                    s0=s, n_steps=1)
        syncs += ns
        for k in range(K):
            worst = max(worst, max_rel_per_tensor(P.lsgd_params(ctx, k), Wo[k], segs))
        np.testing.assert_allclose(P.lsgd_losses(ctx, 1, K)[0], lo[0], rtol=1e-4, atol=1e-5)
    assert P.lsgd_sync_count(ctx) == syncs
    P.lsgd_destroy(ctx)
    assert worst <= tol, worst
    return syncs


@pytest.mark.parametrize("kind,P_ep,H,sampling", [("linear", 2.0, 4, 1), ("exponential", 3.0, 8, 1),
                                                  ("constant", 1.5, 4, 0)])
def test_warmup_runs_stepwise_fp32(P, kind, P_ep, H, sampling):
    widths = (40, 24, 10)
    N, K, B = 320, 4, 8  # 10 steps per epoch
    rng = np.random.default_rng(H)
    X = rng.standard_normal((N, widths[0])).astype(np.float32)
    y = rng.integers(0, widths[-1], N).astype(np.int32)
    hw = {"linear": P.HWARM_LINEAR, "exponential": P.HWARM_EXPONENTIAL,
          "constant": P.HWARM_CONSTANT}[kind]
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=H, T=45, N=N, precision=P.FP32,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=8,
                      h_warmup=hw, h_warmup_epochs=P_ep, sampling=sampling)
    syncs = _stepwise(P, g, o, X, y, widths, 45)
    assert syncs == sum(oracle.is_round_end(o, s) for s in range(45))


def test_warmup_reshuffle_bf16_run(P):
    widths = (264, 136, 72, 10)
    N, K, B, H, T = 1280, 4, 32, 8, 40  # 10 steps per epoch
    X, y = synthdata.gaussian_mixture(N, widths[0], widths[-1], seed=21)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=H, T=T, N=N, precision=P.BF16,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=2,
                      h_warmup=P.HWARM_EXPONENTIAL, h_warmup_epochs=3.0,
                      sampling=P.SAMPLE_RESHUFFLE, fused_update=True)
    w0 = oracle.init_params(o).astype(np.float32)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_set_params(ctx, -1, w0)
    P.lsgd_run(ctx, T)
    W, _, losses, syncs = oracle.run(o, X, y=y, W=np.tile(w0.astype(np.float64), (K, 1)))
    # rounds: 10 of 1, 5 of 2, 3 of 4 (the third runs to step 31), then 8 to the end
    assert P.lsgd_sync_count(ctx) == syncs == 10 + 5 + 3 + 1
    assert rel_l2(P.lsgd_params(ctx, 0), W[0]) <= 2e-2
    assert np.abs(P.lsgd_losses(ctx, T, K) - losses).max() <= 2e-2
    P.lsgd_destroy(ctx)
