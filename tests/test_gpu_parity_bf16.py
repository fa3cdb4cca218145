"""bf16-GEMM parity (tcgen05 grouped GEMMs, fp32 accumulation, fp32 master weights).

Tolerances: after 64 steps the parameters within 2e-2 relative L2 of the oracle's and the loss of
the averaged model within 1e-2 absolute; indices bit-exact.  The full-size MLP 3072-1024-1024-10
run (K = 16, B = 128, N = 50,000) is checked on sampled replicas the oracle recomputes one by one.
The tcgen05 products are also compared against the SIMT products on the same bf16 operands."""
import os

import numpy as np
import pytest

import oracle
import synthdata
from _gpu_common import built_package, dense_cfgs, rel_l2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


def _run_both(P, g, o, X, y, steps):
    w0 = oracle.init_params(o)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_set_params(ctx, -1, w0.astype(np.float32))
    P.lsgd_run(ctx, steps)
    W, _, losses, syncs = oracle.run(o, X, y=y, W=np.tile(w0.astype(np.float32).astype(np.float64),
                                                          (o.K, 1)), n_steps=steps)
    return ctx, W, losses, syncs


@pytest.mark.parametrize("widths,K,B,H", [((264, 136, 72, 10), 3, 40, 4),
                                          ((128, 256, 100), 4, 128, 16)])
def test_small_mlp_64_steps(P, widths, K, B, H):
    N = 1200
    X, y = synthdata.gaussian_mixture(N, widths[0], widths[-1], seed=21)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=H, T=64, N=N, precision=P.BF16,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=2)
    ctx, W, losses, syncs = _run_both(P, g, o, X, y, 64)
    w_gpu = P.lsgd_params(ctx, -1)
    assert rel_l2(w_gpu, W[0]) <= 2e-2
    assert P.lsgd_sync_count(ctx) == syncs == 64 // H
    n_eval = min(N, 8192)
    l_gpu = P.lsgd_eval_loss(ctx, -1, n_eval)
    l_orc = oracle.eval_loss(o, W[0], X, y=y, n=n_eval)
    assert abs(l_gpu - l_orc) <= 1e-2, (l_gpu, l_orc)
    lg = P.lsgd_losses(ctx, 64, K)
    assert np.abs(lg - losses).max() <= 2e-2
    P.lsgd_destroy(ctx)


def test_post_local_switch_bf16(P):
    widths = (192, 64, 10)
    N = 960
    X, y = synthdata.gaussian_mixture(N, widths[0], 10, seed=3)
    g, o = dense_cfgs(P, widths=widths, K=4, B=32, H=4, T=20, N=N, precision=P.BF16, t_switch=10,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=6,
                      milestones=(0.5, 0.75))
    ctx, W, _, syncs = _run_both(P, g, o, X, y, 20)
    assert P.lsgd_sync_count(ctx) == syncs == 10 + 3
    assert rel_l2(P.lsgd_params(ctx, -1), W[0]) <= 2e-2
    P.lsgd_destroy(ctx)


def test_tcgen05_matches_simt_products(P):
    # Same bf16 operands, fp32 accumulation in both; only the accumulation differs.  The tensor
    # cores' accumulation behaves like ~3e-6 relative noise per output (the SIMT kernel's like
    # ~3e-7), and every bf16 re-rounding of a hidden activation or gradient amplifies it: injecting
    # 3e-6 relative noise into each product of an fp64 bf16-operand network moves one step's
    # gradients by 0.3-0.8 % (relative L2).  So the two engines agree to the bf16-mode bar, and the
    # products themselves are checked at fp32 level in test_gpu_gemm.py.
    widths = (3072, 1024, 1024, 10)
    N = 4096
    X, y = synthdata.gaussian_mixture(N, 3072, 10, seed=8)
    outs = {}
    for mode in ("tc", "simt"):
        os.environ["LSGD_FORCE_SIMT"] = "1" if mode == "simt" else "0"
        try:
            g, o = dense_cfgs(P, widths=widths, K=4, B=128, H=16, T=49, N=N, precision=P.BF16,
                              base_lr=0.1, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=1)
            ctx = P.lsgd_create(g)
        finally:
            os.environ.pop("LSGD_FORCE_SIMT", None)
        P.lsgd_set_dataset(ctx, X, y)
        w0 = P.lsgd_params(ctx, 0)
        P.lsgd_run(ctx, 1)
        outs[mode] = (w0, [P.lsgd_params(ctx, k) for k in range(4)], P.lsgd_losses(ctx, 1, 4))
        P.lsgd_destroy(ctx)
    w0 = outs["tc"][0]
    assert np.array_equal(w0, outs["simt"][0])
    np.testing.assert_allclose(outs["tc"][2], outs["simt"][2], rtol=1e-3, atol=1e-6)
    for k in range(4):
        d_tc = outs["tc"][1][k].astype(np.float64) - w0
        d_si = outs["simt"][1][k].astype(np.float64) - w0
        assert rel_l2(d_tc, d_si) <= 2e-2, k


def test_full_size_mlp_sampled_replicas(P):
    # MLP 3072-1024-1024-10 with K = 16, B = 128 on N = 50,000 points, the launch configuration
    # of the benchmark.  One step on all replicas; replicas 0 and 15 recomputed by the oracle.
    widths = (3072, 1024, 1024, 10)
    N, K, B = 50000, 16, 128
    X, y = synthdata.gaussian_mixture_cached(N, 3072, 10, 1234)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=16, T=49, N=N, precision=P.BF16,
                      base_lr=0.1, scale_by_K=True, warmup_epochs=5, momentum=0.9, nesterov=True,
                      weight_decay=5e-4, seed=0, fused_update=True)
    w0 = oracle.init_params(o)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_set_params(ctx, -1, w0.astype(np.float32))
    w0 = w0.astype(np.float32).astype(np.float64)
    P.lsgd_run(ctx, 1)
    lg = P.lsgd_losses(ctx, 1, K)[0]
    lr = oracle.lr(o, 0)
    assert abs(lr - P.lsgd_lr_at(ctx, 0)) < 1e-12
    for k in (0, K - 1):
        idx = oracle.sample_indices(o, k, 0)
        loss, grad = oracle.loss_grad(o, w0, X, y=y, idx=idx)
        w1, _ = oracle.sgd_update(o, lr, w0, np.zeros_like(w0), grad)
        got = P.lsgd_params(ctx, k).astype(np.float64)
        assert rel_l2(got - w0, w1 - w0) <= 2e-2, k
        assert abs(lg[k] - loss) <= 1e-2
    got_idx = P.lsgd_debug_indices(ctx, 0, K, B)
    assert np.array_equal(got_idx, np.stack([oracle.sample_indices(o, k, 0) for k in range(K)]))
    P.lsgd_destroy(ctx)


@pytest.mark.parametrize("mom,nest,wd", [(0.9, True, 5e-4), (0.9, False, 0.0), (0.0, False, 1e-4)])
@pytest.mark.parametrize("widths,K,B", [((264, 136, 72, 10), 3, 40), ((3072, 1024, 1024, 10), 4, 128),
                                        ((200, 136, 96, 72, 10), 2, 24), ((264, 136, 72, 40), 3, 40),
                                        ((200, 136, 96, 72, 40), 2, 24)])
def test_fused_update_is_bitwise_identical(P, mom, nest, wd, widths, K, B):
    # The update applied in the weight-gradient epilogue uses the same arithmetic as the
    # stand-alone update kernel, so parameters, momentum and losses agree bit for bit.  (The
    # first two layers' updates share one launch; with four layers the third has its own; with
    # 40 classes there is no classifier head and the top layer's update joins the last launch.)
    N = 2048
    X, y = synthdata.gaussian_mixture(N, widths[0], widths[-1], seed=4)
    res = []
    for fused in (False, True):
        g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=3, T=7, N=N, precision=P.BF16,
                          base_lr=0.05, momentum=mom, nesterov=nest, weight_decay=wd, seed=9,
                          fused_update=fused)
        ctx = P.lsgd_create(g)
        P.lsgd_set_dataset(ctx, X, y)
        P.lsgd_run(ctx, 7)
        res.append(([P.lsgd_params(ctx, k) for k in range(K)],
                    [P.lsgd_momentum(ctx, k) for k in range(K)], P.lsgd_losses(ctx, 7, K),
                    P.lsgd_kernel_launches(ctx)))
        P.lsgd_destroy(ctx)
    for k in range(K):
        assert np.array_equal(res[0][0][k], res[1][0][k])
        assert np.array_equal(res[0][1][k], res[1][1][k])
    assert np.array_equal(res[0][2], res[1][2])
    assert res[1][3] < res[0][3]  # no stand-alone update launches


def test_post_local_mlp4096_sampled_replica(P):
    # Post-local SGD on MLP 3072-4096-4096-4096-100 (K = 16, B = 128, N = 50,000, 100 classes):
    # the first step recomputed by the oracle for one sampled replica, then the whole 10-epoch
    # schedule (t' = first decay = floor(0.5 T)) run on the GPU with its sync count checked.
    widths = (3072, 4096, 4096, 4096, 100)
    N, K, B = 50000, 16, 128
    T = -(-10 * N // (K * B))  # ceil(10 epochs of N samples / (K B))
    tp = T // 2
    X, y = synthdata.gaussian_mixture_cached(N, 3072, 100, 1234)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=16, T=T, N=N, precision=P.BF16, t_switch=tp,
                      base_lr=0.1, milestones=(0.5, 0.75), momentum=0.9, nesterov=True,
                      weight_decay=5e-4, seed=3, fused_update=True)
    w0 = oracle.init_params(o)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_set_params(ctx, -1, w0.astype(np.float32))
    w0 = w0.astype(np.float32).astype(np.float64)
    P.lsgd_run(ctx, 1)
    k = K - 1
    idx = oracle.sample_indices(o, k, 0)
    loss, grad = oracle.loss_grad(o, w0, X, y=y, idx=idx)
    # Step 0 is in the mini-batch phase, so the parameters are averaged right after it; the
    # worker's momentum stays local and after the first step equals g' = g + lambda w0.
    got_k = P.lsgd_momentum(ctx, k).astype(np.float64)
    gp = grad + 5e-4 * w0
    assert rel_l2(got_k, gp) <= 2e-2
    assert abs(P.lsgd_losses(ctx, 1, K)[0][k] - loss) <= 1e-2
    P.lsgd_run(ctx, T - 1)
    assert P.lsgd_sync_count(ctx) == tp + -(-(T - tp) // 16)
    assert P.lsgd_check_finite(ctx)
    lg = P.lsgd_losses(ctx, T, K)
    # the configured job trains: every loss finite, the last round's mean well below the first's
    assert np.isfinite(lg).all() and lg[-16:].mean() < 0.7 * lg[:16].mean()
    print("post-local MLP4096 mean loss every 16 steps:", lg.mean(1)[::16].round(3).tolist())
    P.lsgd_destroy(ctx)


@pytest.mark.parametrize("K", [8, 64])
def test_sweep_shape_mlp512_sampled_replicas(P, K):
    # MLP 3072-512-512-10, B = 32, heavy-ball momentum 0.9, H = 4: two local steps on all
    # replicas; replicas 0 and K-1 recomputed step by step by the oracle.
    widths = (3072, 512, 512, 10)
    N, B = 50000, 32
    X, y = synthdata.gaussian_mixture_cached(N, 3072, 10, 1234)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=4, T=500, N=N, precision=P.BF16,
                      base_lr=0.1, momentum=0.9, seed=5, fused_update=True)
    w0 = oracle.init_params(o).astype(np.float32).astype(np.float64)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_set_params(ctx, -1, w0.astype(np.float32))
    P.lsgd_run(ctx, 2)
    lg = P.lsgd_losses(ctx, 2, K)
    for k in (0, K - 1):
        w, u = w0.copy(), np.zeros_like(w0)
        for s in range(2):
            loss, grad = oracle.loss_grad(o, w, X, y=y, idx=oracle.sample_indices(o, k, s))
            w, u = oracle.sgd_update(o, oracle.lr(o, s), w, u, grad)
            assert abs(lg[s][k] - loss) <= 1e-2
        got = P.lsgd_params(ctx, k).astype(np.float64)
        assert rel_l2(got - w0, w - w0) <= 2e-2, k
    P.lsgd_destroy(ctx)


def test_hierarchical_local_sgd(P):
    # Hierarchical local SGD (Sec. D): K = 8 workers in blocks of K' = 2, H = 2, H^b = 3.
    widths = (256, 128, 10)
    N, K, B, T = 2048, 8, 32, 24
    X, y = synthdata.gaussian_mixture(N, 256, 10, seed=6)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=2, T=T, N=N, precision=P.BF16, base_lr=0.05,
                      momentum=0.9, nesterov=True, weight_decay=5e-4, seed=8, fused_update=True,
                      hier_block=2, hier_rounds=3)
    w0 = oracle.init_params(o)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_set_params(ctx, -1, w0.astype(np.float32))
    P.lsgd_run(ctx, 2)  # first round: ends with a block average
    reps = [P.lsgd_params(ctx, k) for k in range(K)]
    for b in range(0, K, 2):
        assert np.array_equal(reps[b], reps[b + 1])
    assert not np.array_equal(reps[0], reps[2])
    P.lsgd_run(ctx, T - 2)
    W, _, lo, ng, nb = oracle.run_counted(o, X, y=y, W=np.tile(w0.astype(np.float32).astype(np.float64),
                                                                (K, 1)))
    assert (P.lsgd_sync_count(ctx), P.lsgd_block_sync_count(ctx)) == (ng, nb) == (4, 8)
    assert rel_l2(P.lsgd_params(ctx, -1), W[0]) <= 2e-2
    assert np.abs(P.lsgd_losses(ctx, T, K) - lo).max() <= 2e-2
    P.lsgd_destroy(ctx)


@pytest.mark.parametrize("mom,nest,wd", [(0.9, True, 5e-4), (0.9, False, 0.0), (0.0, False, 1e-4)])
@pytest.mark.parametrize("widths,K,B", [((264, 136, 72, 10), 3, 40),
                                        ((200, 136, 96, 72, 100), 4, 24),
                                        ((264, 136, 72, 40), 3, 40),
                                        ((3072, 1024, 1024, 10), 16, 128)])
def test_average_in_update_launches_is_bitwise_identical(P, mom, nest, wd, widths, K, B):
    # lsgd_run forms the K-way average of a round-ending step inside that step's weight-gradient
    # + update launches (Eq. 2: the mean of the updated replicas).  Post-local schedule: steps 0-4
    # average after every step (the replicas are identical at each step's start), then rounds of
    # three (the round's last step starts from different replicas).  The separate path -- local
    # steps, then lsgd_sync_average -- must give the same parameters, momentum and losses.
    N, T = 2048, 12
    X, y = synthdata.gaussian_mixture(N, widths[0], widths[-1], seed=12)
    res = []
    for fused_avg in (True, False):
        g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=3, T=T, N=N, precision=P.BF16,
                          t_switch=5, base_lr=0.05, momentum=mom, nesterov=nest, weight_decay=wd,
                          seed=7, fused_update=True, milestones=(0.5,))
        ctx = P.lsgd_create(g)
        P.lsgd_set_dataset(ctx, X, y)
        if fused_avg:
            P.lsgd_run(ctx, T)
        else:
            _, kinds = P.lsgd_schedule(g, T)
            for s in range(T):
                P.lsgd_local_step(ctx)
                if kinds[s] == 2:
                    P.lsgd_sync_average(ctx)
        res.append(([P.lsgd_params(ctx, k) for k in range(K)],
                    [P.lsgd_momentum(ctx, k) for k in range(K)] if mom else [],
                    P.lsgd_losses(ctx, T, K), P.lsgd_sync_count(ctx)))
        P.lsgd_destroy(ctx)
    assert res[0][3] == res[1][3] == 5 + 3  # t' syncs, then steps 7, 10 and the last (11)
    for k in range(K):
        assert np.array_equal(res[0][0][k], res[1][0][k]), k
        if mom:
            assert np.array_equal(res[0][1][k], res[1][1][k]), k
    assert np.array_equal(res[0][2], res[1][2])


def test_run_batch_matches_run(P):
    # lsgd_run_batch on the mini-batches lsgd_run samples (host buffers) is the same schedule
    widths, K, B, N, T = (264, 136, 72, 10), 4, 32, 2048, 9
    X, y = synthdata.gaussian_mixture(N, widths[0], 10, seed=13)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=2, T=T, N=N, precision=P.BF16, t_switch=3,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=5,
                      fused_update=True)
    a = P.lsgd_create(g)
    P.lsgd_set_dataset(a, X, y)
    P.lsgd_run(a, T)
    b = P.lsgd_create(g)
    P.lsgd_set_dataset(b, X, y)
    for s in range(T):
        idx = P.lsgd_debug_indices(b, s, K, B).reshape(-1)
        P.lsgd_run_batch(b, np.ascontiguousarray(X[idx].reshape(K, B, -1)),
                         np.ascontiguousarray(y[idx].reshape(K, B)))
    assert P.lsgd_sync_count(a) == P.lsgd_sync_count(b) == 3 + 3
    for k in range(K):
        assert np.array_equal(P.lsgd_params(a, k), P.lsgd_params(b, k)), k
    assert np.array_equal(P.lsgd_losses(a, T, K), P.lsgd_losses(b, T, K))
    P.lsgd_destroy(a)
    P.lsgd_destroy(b)


def test_distinct_replicas_use_their_own_weights(P):
    # After lsgd_set_params on single replicas the replicas differ: every replica's step must use
    # its own weights (a step that follows an average reads one shared copy instead), checked
    # against the oracle's step of each replica from its own parameters.
    widths, K, B, N = (512, 256, 256, 100), 4, 64, 4096
    X, y = synthdata.gaussian_mixture(N, widths[0], widths[-1], seed=17)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=4, T=8, N=N, precision=P.BF16,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=3,
                      fused_update=True)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    rng = np.random.default_rng(4)
    w0 = oracle.init_params(o)
    Ws = [(w0 * (1.0 + 0.5 * k) + 0.01 * rng.standard_normal(len(w0))).astype(np.float32)
          for k in range(K)]
    for k in range(K):
        P.lsgd_set_params(ctx, k, Ws[k])
    P.lsgd_run(ctx, 1)  # step 0 of an H = 4 round: no average
    for k in range(K):
        wk = Ws[k].astype(np.float64)
        loss, grad = oracle.loss_grad(o, wk, X, y=y, idx=oracle.sample_indices(o, k, 0))
        w1, _ = oracle.sgd_update(o, oracle.lr(o, 0), wk, np.zeros_like(wk), grad)
        got = P.lsgd_params(ctx, k).astype(np.float64)
        assert rel_l2(got - wk, w1 - wk) <= 2e-2, k
        assert abs(P.lsgd_losses(ctx, 1, K)[0][k] - loss) <= 1e-2
    P.lsgd_destroy(ctx)


def test_average_left_in_one_replica_is_materialized_for_readers(P):
    # After a step that ends with the average, the mean is written to replica 0 alone (every
    # kernel of the next step reads it there); reading or changing single replicas through the
    # API first gives every replica its copy.
    widths, K, B, N = (264, 136, 72, 10), 4, 32, 2048
    X, y = synthdata.gaussian_mixture(N, widths[0], 10, seed=19)
    g, o = dense_cfgs(P, widths=widths, K=K, B=B, H=4, T=8, N=N, precision=P.BF16, t_switch=4,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=2,
                      fused_update=True)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_run(ctx, 2)  # two H = 1 steps, each ending with the average
    reps = [P.lsgd_params(ctx, k) for k in range(K)]
    assert all(np.array_equal(reps[0], reps[k]) for k in range(K))
    P.lsgd_run(ctx, 1)  # again, then overwrite replica 2 only
    mean = P.lsgd_params(ctx, 0)
    new = (mean * 0.5).astype(np.float32)
    P.lsgd_set_params(ctx, 2, new)
    assert np.array_equal(P.lsgd_params(ctx, 1), mean)
    assert np.array_equal(P.lsgd_params(ctx, 3), mean)
    assert np.array_equal(P.lsgd_params(ctx, 2), new)
    # the next step starts from distinct replicas: the same as the separate-average path's
    ref = P.lsgd_create(g)
    P.lsgd_set_dataset(ref, X, y)
    for s in range(3):
        P.lsgd_local_step(ref)
        P.lsgd_sync_average(ref)
    P.lsgd_set_params(ref, 2, new)
    P.lsgd_run(ctx, 1)
    P.lsgd_local_step(ref)
    P.lsgd_sync_average(ref)  # step 3 ends the H = 1 phase (t' = 4) with an average
    for k in range(K):
        assert np.array_equal(P.lsgd_params(ctx, k), P.lsgd_params(ref, k)), k
    P.lsgd_destroy(ctx)
    P.lsgd_destroy(ref)
