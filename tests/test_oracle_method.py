"""Pin the oracle's local / post-local SGD driver, optimizer and schedules against what the paper
fixes: the mini-batch special cases of Eq. 2 (H = 1, K = 1) and of post-local SGD's first phase, the
momentum expansion of Sec. C.3.1, the sync count of the communication model (Sec. F), the
learning-rate schemes of Sec. A.3 / A.4, the ResNet-20 size of the scaling-ratio table, and
convergence to the closed-form least-squares optimum."""
import math

import numpy as np
import pytest

import oracle
import synthdata


def _mlp_cfg(**kw):
    args = dict(widths=(12, 7, 5), K=4, B=3, H=1, T=6, N=48, base_lr=0.05, seed=21)
    args.update(kw)
    return oracle.make_cfg(**args)


def _data(N, D, C, seed=0):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((N, D)).astype(np.float32), rng.integers(0, C, N).astype(np.int32)


def test_k1_local_sgd_is_minibatch_sgd_bitwise():
    # Eq. 2 with K = 1: the average of one model is the model; local SGD is plain mini-batch SGD.
    for H in (1, 3):
        c = _mlp_cfg(K=1, H=H, momentum=0.9, nesterov=True, weight_decay=5e-4)
        X, y = _data(48, 12, 5)
        W, U, l_local, _ = oracle.run(c, X, y=y)
        w, u, l_mb = oracle.run_minibatch(c, X, y=y)
        assert np.array_equal(W[0], w)
        assert np.array_equal(U[0], u)
        assert np.array_equal(l_local[:, 0], l_mb)


@pytest.mark.parametrize("mom,nest,wd", [(0.0, False, 0.0), (0.9, False, 0.0), (0.9, True, 5e-4)])
def test_h1_local_sgd_is_minibatch_sgd_with_union_batch(mom, nest, wd):
    # "Mini-batch SGD is a special case if H = 1" (Sec. 1, Eq. 1 vs Eq. 2): averaging after every
    # step equals one step on the average of the K local gradients.  With local momentum the
    # equality holds too because averaging is linear and all workers share w after each sync.
    c = _mlp_cfg(H=1, momentum=mom, nesterov=nest, weight_decay=wd)
    X, y = _data(48, 12, 5, 1)
    W, _, _, syncs = oracle.run(c, X, y=y)
    w, _, _ = oracle.run_minibatch(c, X, y=y)
    assert syncs == c.T
    for k in range(c.K):
        np.testing.assert_allclose(W[k], w, rtol=0, atol=1e-13 * np.abs(w).max())


def test_local_sgd_differs_from_minibatch_for_h_gt_1():
    c = _mlp_cfg(H=3, T=6)
    X, y = _data(48, 12, 5, 2)
    W, _, _, _ = oracle.run(c, X, y=y)
    w, _, _ = oracle.run_minibatch(c, X, y=y)
    assert np.abs(W[0] - w).max() > 1e-8


def test_post_local_first_phase_is_minibatch():
    # Post-local SGD with t' >= T never leaves its mini-batch phase (Sec. 3).
    c_pl = _mlp_cfg(H=4, t_switch=6, T=6, momentum=0.9, nesterov=True, weight_decay=1e-4)
    c_h1 = _mlp_cfg(H=1, T=6, momentum=0.9, nesterov=True, weight_decay=1e-4)
    X, y = _data(48, 12, 5, 3)
    W1, _, l1, s1 = oracle.run(c_pl, X, y=y)
    W2, _, l2, s2 = oracle.run(c_h1, X, y=y)
    assert np.array_equal(W1, W2) and np.array_equal(l1, l2) and s1 == s2 == 6
    w, _, _ = oracle.run_minibatch(c_h1, X, y=y)
    np.testing.assert_allclose(W1[0], w, rtol=0, atol=1e-13 * np.abs(w).max())


@pytest.mark.parametrize("T,H,tp", [(64, 4, -1), (49, 16, -1), (245, 16, 122), (25, 16, 12),
                                    (500, 32, -1), (10, 3, 0), (7, 1, -1), (30, 8, 30)])
def test_sync_count_matches_communication_model(T, H, tp):
    # Sec. F: a run of T local steps with H local steps per round has ceil(T/H) averaging rounds;
    # post-local adds one round per step of its first phase: t' + ceil((T - t') / H).
    c = oracle.make_cfg(K=2, B=1, H=H, T=T, t_switch=tp)
    n = sum(oracle.is_round_end(c, s) for s in range(T))
    tp_eff = max(tp, 0)
    expect = tp_eff + math.ceil((T - tp_eff) / H) if tp_eff < T else T
    assert n == expect


def test_run_counts_syncs_and_ends_synchronised():
    c = _mlp_cfg(H=4, T=10)
    X, y = _data(48, 12, 5, 4)
    W, _, _, syncs = oracle.run(c, X, y=y)
    assert syncs == math.ceil(10 / 4)
    for k in range(1, c.K):
        assert np.array_equal(W[0], W[k])


def test_split_run_equals_straight_run():
    c = _mlp_cfg(H=3, T=9, momentum=0.9, nesterov=True)
    X, y = _data(48, 12, 5, 5)
    W, U, l, s = oracle.run(c, X, y=y)
    Wa, Ua, la, sa = oracle.run(c, X, y=y, n_steps=4)
    Wb, Ub, lb, sb = oracle.run(c, X, y=y, W=Wa, U=Ua, s0=4, n_steps=5)
    assert np.array_equal(W, Wb) and np.array_equal(U, Ub)
    assert np.array_equal(l, np.concatenate([la, lb])) and s == sa + sb


def test_momentum_h_step_expansion():
    # Sec. C.3.1: with a fixed gradient g and momentum m, H local steps give
    # w_H = w_0 - gamma (sum_{tau=1..H} m^tau u_0 + sum_{h=1..H} sum_{tau=0..H-h} m^tau g).
    c = oracle.make_cfg(widths=(3, 2), momentum=0.9, nesterov=False)
    d = oracle.num_params(c)
    rng = np.random.default_rng(0)
    w0, u0, g = rng.standard_normal(d), rng.standard_normal(d), rng.standard_normal(d)
    gamma, m, H = 0.05, 0.9, 7
    w, u = w0.copy(), u0.copy()
    for _ in range(H):
        w, u = oracle.sgd_update(c, gamma, w, u, g)
    expect = w0 - gamma * (sum(m**tau for tau in range(1, H + 1)) * u0
                           + sum(sum(m**tau for tau in range(0, H - h + 1)) for h in range(1, H + 1)) * g)
    np.testing.assert_allclose(w, expect, rtol=1e-12, atol=1e-12)


def test_nesterov_and_weight_decay_step():
    # PyTorch-form Nesterov without dampening (Sec. A.4): u' = m u + g + lam w,
    # w' = w - gamma (g + lam w + m u').  Plain SGD when m = 0.
    c = oracle.make_cfg(widths=(3, 2), momentum=0.9, nesterov=True, weight_decay=0.01)
    d = oracle.num_params(c)
    rng = np.random.default_rng(1)
    w, u, g = rng.standard_normal(d), rng.standard_normal(d), rng.standard_normal(d)
    w1, u1 = oracle.sgd_update(c, 0.1, w, u, g)
    gp = g + 0.01 * w
    np.testing.assert_allclose(u1, 0.9 * u + gp, rtol=1e-15)
    np.testing.assert_allclose(w1, w - 0.1 * (gp + 0.9 * u1), rtol=1e-15)
    c0 = oracle.make_cfg(widths=(3, 2))
    w2, u2 = oracle.sgd_update(c0, 0.1, w, u, g)
    np.testing.assert_allclose(w2, w - 0.1 * g, rtol=1e-15)
    assert np.array_equal(u2, u)


def test_lr_warmup_and_decay_schedule():
    # Sec. A.3: start at eta, add (eta_hat - eta) / (5 N / (K B)) each step until eta_hat = K eta.
    c = oracle.make_cfg(K=16, B=128, N=50000, T=49, base_lr=0.1, scale_by_K=True, warmup_epochs=5)
    inc = (1.6 - 0.1) / (5 * 50000 / (16 * 128))
    assert abs(inc - 0.012288) < 1e-12
    for s in (0, 1, 10, 48):
        assert abs(oracle.lr(c, s) - (0.1 + s * inc)) < 1e-12
    c2 = oracle.make_cfg(K=16, B=128, N=50000, T=1000, base_lr=0.1, scale_by_K=True, warmup_epochs=5)
    assert abs(oracle.lr(c2, 200) - 1.6) < 1e-12
    # Sec. 4: divide by 10 once 50% and 75% of the samples have been accessed.
    c3 = oracle.make_cfg(K=16, B=128, N=50000, T=245, base_lr=0.1, scale_by_K=True, warmup_epochs=5,
                         milestones=(0.5, 0.75), decay=0.1)
    # warm-up spans 5 N / (K B) = 122.07 steps, so step 122 is still on the ramp when decayed
    assert abs(oracle.lr(c3, 121) - (0.1 + 121 * inc)) < 1e-12
    assert abs(oracle.lr(c3, 122) - 0.1 * (0.1 + 122 * inc)) < 1e-12
    assert abs(oracle.lr(c3, 183) - 0.016) < 1e-12
    c4 = oracle.make_cfg(K=4, B=32, N=8192, T=64, base_lr=0.1)
    assert all(oracle.lr(c4, s) == 0.1 for s in range(64))


def test_average_is_mean_and_identity_on_equal_replicas():
    rng = np.random.default_rng(3)
    W = rng.standard_normal((5, 17))
    A = oracle.average(W)
    np.testing.assert_allclose(A, np.tile(W.mean(0), (5, 1)), rtol=1e-15, atol=1e-15)
    e = rng.standard_normal(17)
    for K in (1, 2):  # x + x = 2x and 2x / 2 = x exactly
        E = np.tile(e, (K, 1))
        assert np.array_equal(oracle.average(E), E)
    E = np.tile(e, (7, 1))
    np.testing.assert_allclose(oracle.average(E), E, rtol=4e-16, atol=0)


def test_least_squares_converges_to_closed_form():
    # Local SGD on a consistent least-squares problem reaches the closed-form optimum
    # w* = (A^T A)^-1 A^T t (computed by LAPACK in fp64) for K in {1, 4}, H in {1, 8}.
    N, d = 512, 20
    A, t, _ = synthdata.least_squares(N, d, seed=7)
    w_opt = np.linalg.lstsq(A.astype(np.float64), t.astype(np.float64), rcond=None)[0]
    for K in (1, 4):
        for H in (1, 8):
            c = oracle.make_cfg(kind=oracle.LSQ, widths=(d, 1), has_bias=False, K=K, B=16, H=H,
                                T=1600, N=N, base_lr=0.02, seed=5)
            W, _, _, _ = oracle.run(c, A, t=t, W=np.zeros((K, d)))
            err = np.linalg.norm(W[0] - w_opt) / np.linalg.norm(w_opt)
            assert err <= 1e-6, (K, H, err)


def test_resnet20_size_matches_paper():
    # Scaling-ratio table (Sec. A.2): ResNet-20 has 0.27 M parameters; with option-A shortcuts the
    # count is 269,722.
    c = oracle.make_cfg(kind=oracle.RESNET20)
    assert oracle.num_params(c) == 269722
    mask = oracle.weight_decay_mask(c)
    n_bn = 2 * (16 + 6 * 16 + 6 * 32 + 6 * 64)
    assert int((mask == 0).sum()) == n_bn  # BN affine parameters carry no weight decay


def test_resnet_with_zeroed_residual_branches_reduces_to_shortcuts():
    # With gamma = beta = 0 in every block's second BN, each block outputs relu(shortcut(x)), so the
    # network is stem -> option-A subsampling -> global average pool -> classifier.
    c = oracle.make_cfg(kind=oracle.RESNET20, in_hwc=(8, 8, 3), base_ch=4, res_blocks=2, n_classes=5,
                        B=3, N=3, seed=4)
    d = oracle.num_params(c)
    w = oracle.init_params(c)
    # parameter layout: stem (w, g, b), then per conv (w, g, b), then fc W, fc b
    specs = []
    off = 0
    cin = 3
    chans = [4] + [4 * (1 << st) for st in range(3) for _ in range(2 * 2)]
    convs = [(3, 4)]
    ch = 4
    for st in range(3):
        co = 4 << st
        for b in range(2):
            convs.append((ch, co))
            convs.append((co, co))
            ch = co
    for ci, co in convs:
        specs.append((off, off + 9 * ci * co, off + 9 * ci * co + co, ci, co))
        off += 9 * ci * co + 2 * co
    fc_w, fc_b = off, off + 5 * 16
    assert fc_b + 5 == d
    for j, (wo, go, bo, ci, co) in enumerate(specs):
        if j >= 1 and j % 2 == 0:
            w[go:go + co] = 0.0
            w[bo:bo + co] = 0.0
    rng = np.random.default_rng(0)
    w[fc_w:fc_b + 5] = rng.standard_normal(5 * 16 + 5)
    X, y = _data(3, 8 * 8 * 3, 5, 6)
    loss, _ = oracle.loss_grad(c, w, X, y=y, idx=np.arange(3))
    # stem in numpy
    x = X.reshape(3, 8, 8, 3).astype(np.float64)
    wo, go, bo, ci, co = specs[0]
    Wst = w[wo:wo + 9 * ci * co].reshape(co, 3, 3, ci)
    xp = np.pad(x, ((0, 0), (1, 1), (1, 1), (0, 0)))
    ystem = np.zeros((3, 8, 8, co))
    for kh in range(3):
        for kw in range(3):
            ystem += np.einsum("bhwc,oc->bhwo", xp[:, kh:kh + 8, kw:kw + 8, :], Wst[:, kh, kw, :])
    mu = ystem.mean((0, 1, 2))
    var = ystem.var((0, 1, 2))
    a = np.maximum((ystem - mu) / np.sqrt(var + 1e-5) * w[go:go + co] + w[bo:bo + co], 0)
    # stage 2, 3 entries: subsample by 2 and append zero channels
    a = a[:, ::2, ::2, :]
    a = a[:, ::2, ::2, :]
    feat = np.zeros((3, 16))
    feat[:, :4] = a.mean((1, 2))
    Z = feat @ w[fc_w:fc_b].reshape(5, 16).T + w[fc_b:fc_b + 5]
    lse = np.log(np.exp(Z - Z.max(1, keepdims=True)).sum(1)) + Z.max(1)
    np.testing.assert_allclose(loss, np.mean(lse - Z[np.arange(3), y]), rtol=1e-12)


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(9)
    vals = np.concatenate([rng.standard_normal(2000) * 10.0 ** rng.integers(-30, 30, 2000),
                           [1.0, 1.0 + 2**-8, 1.0 + 3 * 2**-9, -2.5, 0.0, 65504.0, 1e-40]])
    for v in vals:
        ref = float(torch.tensor(np.float32(v)).to(torch.bfloat16).float())
        assert oracle.bf16_round(float(np.float32(v))) == ref


def test_bf16_mode_is_exact_when_operands_are_representable():
    # Least squares with small-integer data, weights and targets and B a power of two: every GEMM
    # operand is exactly representable in bf16, so bf16 mode equals fp32-operand mode.
    rng = np.random.default_rng(4)
    X = rng.integers(-3, 4, (16, 8)).astype(np.float32)
    t = rng.integers(-5, 6, 16).astype(np.float32)
    w = rng.integers(-2, 3, 8).astype(np.float64)
    c32 = oracle.make_cfg(kind=oracle.LSQ, widths=(8, 1), has_bias=False, B=4, N=16)
    c16 = oracle.make_cfg(kind=oracle.LSQ, widths=(8, 1), has_bias=False, B=4, N=16, bf16=True)
    idx = np.array([1, 3, 3, 9])
    l32, g32 = oracle.loss_grad(c32, w, X, t=t, idx=idx)
    l16, g16 = oracle.loss_grad(c16, w, X, t=t, idx=idx)
    assert l32 == l16 and np.array_equal(g32, g16)


def test_bf16_mode_rounds_operands():
    # With generic values the bf16 operands change the gradient by about bf16's precision.
    c32 = oracle.make_cfg(widths=(40, 30, 10), B=8, N=8)
    c16 = oracle.make_cfg(widths=(40, 30, 10), B=8, N=8, bf16=True)
    X, y = _data(8, 40, 10, 7)
    w = np.random.default_rng(8).standard_normal(oracle.num_params(c32)) * 0.2
    _, g32 = oracle.loss_grad(c32, w, X, y=y, idx=np.arange(8))
    _, g16 = oracle.loss_grad(c16, w, X, y=y, idx=np.arange(8))
    rel = np.linalg.norm(g16 - g32) / np.linalg.norm(g32)
    assert 1e-4 < rel < 3e-2


def test_init_statistics():
    # He-normal weights: mean 0, variance 2 / fan_in; zero biases.
    c = oracle.make_cfg(widths=(3072, 1024, 10), seed=3)
    w = oracle.init_params(c)
    W1 = w[:3072 * 1024]
    assert abs(W1.mean()) < 5 * math.sqrt(2 / 3072) / math.sqrt(W1.size)
    assert abs(W1.var() / (2 / 3072) - 1) < 0.01
    assert np.all(w[3072 * 1024:3072 * 1024 + 1024] == 0)
    assert np.all(oracle.init_params(c, oracle.INIT_ZERO) == 0)
    # fp32-representable (the accelerated path stores fp32 master weights)
    assert np.array_equal(w, w.astype(np.float32).astype(np.float64))


# ---- hierarchical local SGD (Sec. D) ----

def test_hierarchical_with_one_block_is_local_sgd():
    # K' = K: every block average is the global average, so the run equals plain local SGD.
    X, y = _data(48, 12, 5, 11)
    c_h = _mlp_cfg(H=2, T=12, hier_block=4, hier_rounds=3, momentum=0.9, nesterov=True)
    c_l = _mlp_cfg(H=2, T=12, momentum=0.9, nesterov=True)
    Wh, _, lh, ng, nb = oracle.run_counted(c_h, X, y=y)
    Wl, _, ll, _ = oracle.run(c_l, X, y=y)
    assert np.array_equal(Wh, Wl) and np.array_equal(lh, ll)
    assert (ng, nb) == (2, 4)


def test_hierarchical_with_singleton_blocks_is_local_sgd_with_longer_rounds():
    # K' = 1: a block average leaves every worker unchanged, so hierarchical (H, H^b) equals local
    # SGD with rounds of H H^b steps.
    X, y = _data(48, 12, 5, 12)
    c_h = _mlp_cfg(H=2, T=12, hier_block=1, hier_rounds=3)
    c_l = _mlp_cfg(H=6, T=12)
    Wh, _, _, ng, nb = oracle.run_counted(c_h, X, y=y)
    Wl, _, _, nl = oracle.run(c_l, X, y=y)
    assert np.array_equal(Wh, Wl) and ng == nl == 2 and nb == 4


def test_block_average_is_blockwise_mean():
    rng = np.random.default_rng(2)
    W = rng.standard_normal((6, 9))
    A = oracle.block_average(W, 3)
    np.testing.assert_allclose(A[:3], np.tile(W[:3].mean(0), (3, 1)), rtol=1e-15, atol=1e-15)
    np.testing.assert_allclose(A[3:], np.tile(W[3:].mean(0), (3, 1)), rtol=1e-15, atol=1e-15)


@pytest.mark.parametrize("T,H,Hb", [(64, 4, 4), (96, 2, 8), (48, 16, 3)])
def test_hierarchical_sync_counts_match_communication_model(T, H, Hb):
    # Sec. F: with T a multiple of H H^b there are T/(H H^b) global and T/H - T/(H H^b) block
    # averages (the two terms of the hierarchical communication cost).
    c = oracle.make_cfg(K=4, B=1, H=H, T=T, hier_block=2, hier_rounds=Hb)
    kinds = [oracle.sync_kind(c, s) for s in range(T)]
    assert kinds.count(2) == T // (H * Hb)
    assert kinds.count(1) == T // H - T // (H * Hb)


# ---- global momentum (Sec. C.3.1) and compressed averaging (Sec. B.3, Algorithms 4 and 5) ----

def _sr_cfg(**kw):
    # softmax regression: no ReLU, so no gradient component is exactly zero on random data
    args = dict(widths=(12, 5), K=3, B=4, H=1, T=8, N=48, base_lr=0.05, seed=31)
    args.update(kw)
    return oracle.make_cfg(**args)


def test_global_momentum_h1_is_heavy_ball_minibatch_sgd():
    # With H = 1 and plain local steps, the global momentum u = m u + (w_ref - mean w^k) / lr
    # = m u + mean_k grad^k, w_ref -= lr u: heavy-ball mini-batch SGD on the union batch.
    X, y = _data(48, 12, 5, 21)
    c_g = _sr_cfg(global_momentum=0.9)
    c_m = _sr_cfg(momentum=0.9)
    W, _, _, _, _, _, ng, _ = oracle.run_ext(c_g, X, y=y)
    w, _, _ = oracle.run_minibatch(c_m, X, y=y)
    assert ng == 8
    np.testing.assert_allclose(W[0], w, rtol=0, atol=1e-12 * np.abs(w).max())


def test_global_momentum_vanishing_factor_is_plain_averaging():
    X, y = _data(48, 12, 5, 22)
    W, _, _, _, _, _, _, _ = oracle.run_ext(_sr_cfg(H=2, global_momentum=1e-12), X, y=y)
    Wp, _, _, _ = oracle.run(_sr_cfg(H=2), X, y=y)
    np.testing.assert_allclose(W, Wp, rtol=0, atol=1e-12 * np.abs(Wp).max())


def test_sign_compression_is_lossless_for_one_worker_and_one_step():
    # Algorithm 4 with K = 1, H = 1: the sign local step moves every coordinate by exactly lr, so
    # ||Delta||_1 / d = lr and sign(Delta) lr = Delta: the run is plain signSGD, w -= lr sign(grad).
    X, y = _data(48, 12, 5, 23)
    c = _sr_cfg(K=1, compress=oracle.COMPRESS_SIGN)
    W, _, _, _, _, _, ng, _ = oracle.run_ext(c, X, y=y)
    w = oracle.init_params(c)
    for s in range(c.T):
        _, g = oracle.loss_grad(c, w, X, y=y, idx=oracle.sample_indices(c, 0, s))
        w = w - 0.05 * np.sign(g)
    assert ng == 8
    np.testing.assert_allclose(W[0], w, rtol=0, atol=1e-13)


def test_sign_compressed_average_of_a_round():
    # One round of K = 2 workers (H = 3): the model after the sync is w_ref - (1/K) sum_k s^k p^k
    # of the workers' models before it (taken from the same run with a longer round).
    X, y = _data(48, 12, 5, 24)
    c = _sr_cfg(K=2, H=3, T=100, compress=oracle.COMPRESS_SIGN)
    c_long = _sr_cfg(K=2, H=4, T=100, compress=oracle.COMPRESS_SIGN)
    w0 = oracle.init_params(c)
    Wpre, _, _, _, _, _, _, _ = oracle.run_ext(c_long, X, y=y, n_steps=3)
    Wpost, _, wref, _, _, _, ng, _ = oracle.run_ext(c, X, y=y, n_steps=3)
    assert ng == 1
    delta = w0[None, :] - Wpre
    p = np.abs(delta).sum(1) / delta.shape[1]
    expect = w0 - (np.sign(delta) * p[:, None]).mean(0)
    np.testing.assert_allclose(wref, expect, rtol=0, atol=1e-14)
    assert np.array_equal(Wpost[0], wref) and np.array_equal(Wpost[1], wref)


def test_error_feedback_bookkeeping():
    # Algorithm 5 with K = 1: the synchronised model equals the worker's own model after the round
    # corrected by the change of its error memory, w_ref(t+1) = w(t+H) - e(t) + e(t+1), and the memory
    # keeps exactly what the compression dropped.
    X, y = _data(48, 12, 5, 25)
    c = _sr_cfg(K=1, H=3, T=100, compress=oracle.COMPRESS_EF_SIGN)
    c_plain = _sr_cfg(K=1, H=3, T=100)
    rng = np.random.default_rng(5)
    d = oracle.num_params(c)
    e0 = 1e-3 * rng.standard_normal((1, d))
    W, _, wref, e1, _, _, _, _ = oracle.run_ext(c, X, y=y, E=e0, n_steps=3)
    Wl, _, _, _ = oracle.run(c_plain, X, y=y, n_steps=3)  # EF does not change the local steps
    np.testing.assert_allclose(wref, Wl[0] - e0[0] + e1[0], rtol=0, atol=1e-14)
    w0 = oracle.init_params(c)
    delta = w0 - Wl[0] + e0[0]
    sp = np.sign(delta) * np.abs(delta).mean()
    np.testing.assert_allclose(e1[0], delta - sp, rtol=0, atol=1e-14)


def test_split_run_with_sync_state_equals_straight_run():
    X, y = _data(48, 12, 5, 26)
    for kw in (dict(compress=oracle.COMPRESS_EF_SIGN), dict(global_momentum=0.8),
               dict(compress=oracle.COMPRESS_SIGN, momentum=0.9)):
        c = _sr_cfg(H=2, T=9, **kw)
        A = oracle.run_ext(c, X, y=y)
        B = oracle.run_ext(c, X, y=y, n_steps=4)
        C = oracle.run_ext(c, X, y=y, W=B[0], U=B[1], Wref=B[2], E=B[3], Ug=B[4], s0=4, n_steps=5)
        for a, b in zip(A[:5], C[:5]):
            assert np.array_equal(a, b)
