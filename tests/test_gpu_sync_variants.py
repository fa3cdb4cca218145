"""The averaging variants on the GPU against the oracle: global momentum (Sec. C.3.1) and the
sign / error-feedback sign compressed averages (Algorithms 4 and 5).

Stepwise cases import the oracle's whole state (w, u, w_ref, e^k, u_g rounded to fp32) before
every GPU step and compare the step's result at max relative error 1e-5 per tensor.  Global
momentum has no data-dependent decision, so every element must meet that bar.  The sign variants
quantise, and a sign whose argument is zero in exact arithmetic is decided by rounding on both
sides: sign local steps that cancel over a round (+gamma then -gamma) leave Delta_k = 0 exactly,
but w - gamma + gamma is not w in floating point.  Coordinates where the oracle's Delta_k lies
within a few fp32 ulps of zero are therefore ambiguous; there the GPU's average must be one of the
valid outcomes (within 2 p_k / K per ambiguous replica of the oracle's), and they are excluded
from the element bar.  Every other element meets the 1e-5 bar, except sign local steps whose direction
lies within rounding of zero, which must stay below 1e-4 of the run's sign decisions.

Multi-step bf16 runs (no re-import, 16 steps) are checked at the bf16 bar, 2e-2 relative L2 of
the parameters, and their displacement from the start must sit closer to the oracle's bf16 run
than the oracle's bf16 run sits to its own fp32-operand run: sign decisions turn the tensor cores'
accumulation noise into whole +-gamma steps, so longer runs drift apart at the rate bf16
rounding itself makes them drift."""
import ctypes
import os
import tempfile

import numpy as np
import pytest

import oracle
import synthdata
from _gpu_common import built_package, dense_cfgs, dense_segments, rel_l2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


WIDTHS = (50, 72, 36, 13)


def _data(N, widths, seed):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((N, widths[0])).astype(np.float32)
    y = rng.integers(0, widths[-1], N).astype(np.int32)
    return X, y


def _mismatch(a, o, segs, tol):
    """Elements of a that miss o by more than tol x max |o| of their tensor."""
    a = np.asarray(a, np.float64)
    bad = np.zeros(a.shape, dtype=bool)
    for off, n in segs:
        den = max(np.abs(o[off:off + n]).max(), 1e-30)
        bad[off:off + n] = np.abs(a[off:off + n] - o[off:off + n]) > tol * den
    return bad


def _local_only(o):
    """The oracle configuration with the same local steps and no synchronisation."""
    assert o.n_milestones == 0 and o.warmup_epochs == 0.0  # lr must not depend on T
    ol = type(o).from_buffer_copy(o)
    ol.H, ol.T, ol.t_switch = 1 << 30, 1 << 40, -1
    return ol


def _ambiguous(o, ol, X, y, Wf, Uf, Rf, Ef, s):
    """Coordinates whose Delta_k is zero up to fp32 rounding for some k, and the bound on how far
    the average may move there: sum over those k of 2 p_k / K (a sign taken the other way)."""
    W1, _, _, _ = oracle.run(ol, X, y=y, W=Wf.astype(np.float64), U=Uf.astype(np.float64), s0=s,
                             n_steps=1)
    R = Rf.astype(np.float64)
    D = R[None, :] - W1
    # Rounding happened at the size of every value the round passed through: w_ref, the replicas
    # before and after this step, and one step of the learning rate (a weight that started at 0).
    mag = np.abs(R)[None, :] + np.abs(Wf) + np.abs(W1) + oracle.lr(o, s)
    if o.compress == oracle.COMPRESS_EF_SIGN:
        D += Ef.astype(np.float64)
        mag += np.abs(Ef)
    ulp = np.spacing(mag.astype(np.float32)).astype(np.float64)
    amb_k = np.abs(D) <= 4.0 * ulp
    p = np.abs(D).sum(axis=1) / D.shape[1]
    slack = 2.0 * (amb_k * p[:, None]).sum(axis=0) / o.K
    return amb_k.any(axis=0), slack


def _stepwise(P, g, o, X, y, widths, steps, tol=1e-5):
    """Returns (elements off the bar, sign decisions taken, ambiguous coordinates) over the run."""
    K = g.K
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    d = P.lsgd_num_params(ctx)
    segs = dense_segments(widths)
    Wo = np.tile(oracle.init_params(o), (K, 1))
    Uo = np.zeros_like(Wo)
    Ro = Wo[0].copy()
    Eo = np.zeros_like(Wo)
    Go = np.zeros(d)
    ef = o.compress == oracle.COMPRESS_EF_SIGN
    gm = o.global_momentum > 0.0
    ol = _local_only(o) if o.compress != oracle.COMPRESS_NONE else None
    off_bar, decisions, n_amb, syncs = 0, 0, 0, 0
    for s in range(steps):
        f32 = lambda a: a.astype(np.float32)  # noqa: E731
        Wf, Uf, Rf, Ef, Gf = f32(Wo), f32(Uo), f32(Ro), f32(Eo), f32(Go)
        for k in range(K):
            P.lsgd_set_params(ctx, k, Wf[k])
            if g.momentum != 0.0:
                P.lsgd_set_momentum(ctx, k, Uf[k])
            if ef:
                P.lsgd_set_sync_state(ctx, P.STATE_ERROR, k, Ef[k])
        P.lsgd_set_sync_state(ctx, P.STATE_WREF, 0, Rf)
        if gm:
            P.lsgd_set_sync_state(ctx, P.STATE_GLOBAL_MOMENTUM, 0, Gf)
        P.lsgd_run(ctx, 1)
        Wo, Uo, Ro, Eo, Go, lo, ng, _ = oracle.run_ext(
            o, X, y=y, W=Wf.astype(np.float64), U=Uf.astype(np.float64), Wref=Rf.astype(np.float64),
            E=Ef.astype(np.float64), Ug=Gf.astype(np.float64), s0=s, n_steps=1)
        syncs += ng
        if o.compress == oracle.COMPRESS_SIGN:
            decisions += K * d                      # one sign per local-step element
        amb = np.zeros(d, dtype=bool)
        if o.compress != oracle.COMPRESS_NONE and ng:
            decisions += K * d                      # one sign per element of every Delta_k
            amb, slack = _ambiguous(o, ol, X, y, Wf, Uf, Rf, Ef, s)
            n_amb += int(amb.sum())
            got = P.lsgd_sync_state(ctx, P.STATE_WREF, 0).astype(np.float64)
            assert np.all(np.abs(got - Ro)[amb] <= 1.0001 * slack[amb] + 1e-6)
        bad = np.zeros(d, dtype=bool)
        for k in range(K):
            bad |= _mismatch(P.lsgd_params(ctx, k), Wo[k], segs, tol)
            if g.momentum != 0.0:
                bad |= _mismatch(P.lsgd_momentum(ctx, k), Uo[k], segs, tol)
            if ef:
                bad |= _mismatch(P.lsgd_sync_state(ctx, P.STATE_ERROR, k), Eo[k], segs, tol)
        bad |= _mismatch(P.lsgd_sync_state(ctx, P.STATE_WREF, 0), Ro, segs, tol)
        if gm:
            bad |= _mismatch(P.lsgd_sync_state(ctx, P.STATE_GLOBAL_MOMENTUM, 0), Go, segs, tol)
        off_bar += int((bad & ~amb).sum())
        np.testing.assert_allclose(P.lsgd_losses(ctx, 1, K)[0], lo[0], rtol=1e-4, atol=1e-5)
    assert P.lsgd_sync_count(ctx) == syncs
    P.lsgd_destroy(ctx)
    return off_bar, decisions, n_amb


@pytest.mark.parametrize("K,B,H,tp,mg", [(4, 8, 3, -1, 0.9), (3, 7, 2, 4, 0.5), (1, 9, 4, -1, 0.9)])
def test_global_momentum_stepwise(P, K, B, H, tp, mg):
    X, y = _data(400, WIDTHS, K * 7 + B)
    g, o = dense_cfgs(P, widths=WIDTHS, K=K, B=B, H=H, T=12, N=400, precision=P.FP32, t_switch=tp,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=4,
                      warmup_epochs=0.5, milestones=(0.5,), global_momentum=mg)
    off_bar, _, _ = _stepwise(P, g, o, X, y, WIDTHS, 12)
    assert off_bar == 0


@pytest.mark.parametrize("compress", ["sign", "ef_sign"])
@pytest.mark.parametrize("K,B,H,mom", [(4, 8, 3, 0.0), (3, 16, 2, 0.9), (5, 5, 4, 0.9)])
def test_sign_compressed_stepwise(P, compress, K, B, H, mom):
    X, y = _data(400, WIDTHS, K * 11 + B)
    cm = P.COMPRESS_SIGN if compress == "sign" else P.COMPRESS_EF_SIGN
    g, o = dense_cfgs(P, widths=WIDTHS, K=K, B=B, H=H, T=12, N=400, precision=P.FP32,
                      base_lr=0.01 if compress == "sign" else 0.05, momentum=mom,
                      nesterov=mom > 0, weight_decay=5e-4, seed=5, compress=cm)
    off_bar, decisions, n_amb = _stepwise(P, g, o, X, y, WIDTHS, 12)
    assert decisions > 0
    assert off_bar <= 1e-4 * decisions, (off_bar, decisions, n_amb)


def test_softmax_regression_ef_sign_stepwise(P):
    # 3072 -> 10 softmax regression (zero init), K = 4, B = 32, H = 4: Delta_k of d = 30,730
    # coordinates, the compressed average every 4 steps.
    X, y = synthdata.gaussian_mixture_cached(8192, 3072, 10, 1234)
    g, o = dense_cfgs(P, widths=(3072, 10), K=4, B=32, H=4, T=16, N=8192, precision=P.FP32,
                      base_lr=0.1, seed=0, init="zero", compress=P.COMPRESS_EF_SIGN)
    off_bar, decisions, n_amb = _stepwise(P, g, o, X, y, (3072, 10), 16)
    assert off_bar <= 1e-4 * decisions, (off_bar, decisions, n_amb)


@pytest.mark.parametrize("variant", ["gm", "sign", "ef_sign"])
def test_variants_bf16_multi_step(P, variant):
    widths = (264, 136, 72, 10)
    N, K, B, H, T = 1200, 4, 32, 4, 16
    X, y = synthdata.gaussian_mixture(N, widths[0], widths[-1], seed=21)
    kw = {"gm": dict(global_momentum=0.5, base_lr=0.05),
          "sign": dict(compress=P.COMPRESS_SIGN, base_lr=0.001),
          "ef_sign": dict(compress=P.COMPRESS_EF_SIGN, base_lr=0.025)}[variant]
    common = dict(widths=widths, K=K, B=B, H=H, T=T, N=N, momentum=0.9, nesterov=True,
                  weight_decay=5e-4, seed=2, **kw)
    g, o = dense_cfgs(P, precision=P.BF16, **common)
    _, o32 = dense_cfgs(P, precision=P.FP32, **common)
    w0 = oracle.init_params(o).astype(np.float32)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_set_params(ctx, -1, w0)
    P.lsgd_run(ctx, T)
    W0 = np.tile(w0.astype(np.float64), (K, 1))
    W, _, Wref, _, _, losses, ng, _ = oracle.run_ext(o, X, y=y, W=W0, n_steps=T)
    W32 = oracle.run_ext(o32, X, y=y, W=W0, n_steps=T)[0]
    assert P.lsgd_sync_count(ctx) == ng == T // H
    wg = P.lsgd_params(ctx, 0).astype(np.float64)
    assert rel_l2(wg, W[0]) <= 2e-2
    assert rel_l2(P.lsgd_sync_state(ctx, P.STATE_WREF, 0), Wref) <= 2e-2
    assert rel_l2(wg - w0, W[0] - w0) <= rel_l2(W[0] - w0, W32[0] - w0)
    assert np.abs(P.lsgd_losses(ctx, T, K) - losses).max() <= 2e-2
    # training makes progress under every variant
    assert losses[-1].mean() < losses[0].mean()
    P.lsgd_destroy(ctx)


@pytest.mark.parametrize("mom,nest", [(0.9, True), (0.0, False)])
def test_fused_sign_update_is_bitwise_identical(P, mom, nest):
    widths = (264, 136, 72, 10)
    N, K = 2048, 3
    X, y = synthdata.gaussian_mixture(N, widths[0], widths[-1], seed=4)
    res = []
    for fused in (False, True):
        g, _ = dense_cfgs(P, widths=widths, K=K, B=40, H=3, T=7, N=N, precision=P.BF16,
                          base_lr=0.005, momentum=mom, nesterov=nest, weight_decay=5e-4, seed=9,
                          fused_update=fused, compress=P.COMPRESS_SIGN)
        ctx = P.lsgd_create(g)
        P.lsgd_set_dataset(ctx, X, y)
        P.lsgd_run(ctx, 7)
        res.append(([P.lsgd_params(ctx, k) for k in range(K)], P.lsgd_losses(ctx, 7, K)))
        P.lsgd_destroy(ctx)
    for k in range(K):
        assert np.array_equal(res[0][0][k], res[1][0][k])
    assert np.array_equal(res[0][1], res[1][1])


@pytest.mark.parametrize("variant", ["gm", "ef_sign"])
def test_checkpoint_resume_keeps_sync_state(P, variant):
    widths = (128, 64, 10)
    kw = dict(global_momentum=0.7) if variant == "gm" else dict(compress=P.COMPRESS_EF_SIGN)
    g, _ = dense_cfgs(P, widths=widths, K=4, B=16, H=3, T=12, N=512, precision=P.FP32,
                      base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=3, **kw)
    X, y = synthdata.gaussian_mixture(512, widths[0], widths[-1], seed=1)
    a = P.lsgd_create(g)
    P.lsgd_set_dataset(a, X, y)
    P.lsgd_run(a, 12)
    want = [P.lsgd_params(a, k) for k in range(4)]
    b = P.lsgd_create(g)
    P.lsgd_set_dataset(b, X, y)
    P.lsgd_run(b, 7)
    with tempfile.TemporaryDirectory() as d:
        path = os.path.join(d, "ck.bin")
        P.lsgd_save(b, path)
        c = P.lsgd_create(g)
        P.lsgd_set_dataset(c, X, y)
        P.lsgd_load(c, path)
        # a checkpoint of another variant does not load
        g2, _ = dense_cfgs(P, widths=widths, K=4, B=16, H=3, T=12, N=512, precision=P.FP32,
                           base_lr=0.05, momentum=0.9, nesterov=True, weight_decay=5e-4, seed=3)
        e = P.lsgd_create(g2)
        with pytest.raises(RuntimeError):
            P.lsgd_load(e, path)
        P.lsgd_destroy(e)
    P.lsgd_run(c, 5)
    for k in range(4):
        assert np.array_equal(P.lsgd_params(c, k), want[k])
    for h in (a, b, c):
        P.lsgd_destroy(h)


def test_sync_state_errors(P):
    widths = (32, 16, 4)
    X, y = _data(64, widths, 0)
    g, _ = dense_cfgs(P, widths=widths, K=2, B=4, H=2, T=4, N=64, precision=P.FP32)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    with pytest.raises(RuntimeError):
        P.lsgd_sync_state(ctx, P.STATE_WREF, 0)
    P.lsgd_destroy(ctx)
    g, _ = dense_cfgs(P, widths=widths, K=2, B=4, H=2, T=4, N=64, precision=P.FP32,
                      compress=P.COMPRESS_SIGN)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    # w_ref starts as the broadcast initial model; sign compression keeps no e^k or u_g
    assert np.array_equal(P.lsgd_sync_state(ctx, P.STATE_WREF, 0), P.lsgd_params(ctx, 0))
    for which, k in ((P.STATE_ERROR, 0), (P.STATE_GLOBAL_MOMENTUM, 0), (P.STATE_WREF, 1)):
        with pytest.raises(RuntimeError):
            P.lsgd_sync_state(ctx, which, k)
    P.lsgd_destroy(ctx)
    for bad in (dict(compress=P.COMPRESS_SIGN, global_momentum=0.5),
                dict(compress=P.COMPRESS_EF_SIGN, hier_block=1, hier_rounds=2),
                dict(global_momentum=0.5, hier_block=1, hier_rounds=2),
                dict(compress=3), dict(global_momentum=-0.1)):
        g = P.make_config(K=2, B_loc=4, H=2, total_steps=4, N=64, kind=P.MLP, widths=widths,
                          precision=P.FP32, **bad)
        with pytest.raises(RuntimeError):
            P.lsgd_create(g)
    # the L1-norm kernel keeps one value per warp and replica in shared memory: K <= 1024
    g = P.make_config(K=1025, B_loc=4, H=2, total_steps=4, N=8200, kind=P.MLP, widths=widths,
                      precision=P.FP32, compress=P.COMPRESS_SIGN)
    with pytest.raises(RuntimeError):
        P.lsgd_create(g)
