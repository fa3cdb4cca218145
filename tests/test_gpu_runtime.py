"""Runtime behaviour on the GPU: checkpoint / resume, caller-supplied mini-batches, schedule sync
counts, error handling (bad arguments, call order, failed allocation, non-finite parameters)."""
import ctypes
import os
import tempfile

import numpy as np
import pytest

import oracle
import synthdata
from _gpu_common import built_package, dense_cfgs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


def _small(P, precision, **kw):
    widths = kw.pop("widths", (128, 64, 10))
    args = dict(widths=widths, K=4, B=16, H=3, T=12, N=512, precision=precision, base_lr=0.05,
                momentum=0.9, nesterov=True, weight_decay=5e-4, seed=3)
    args.update(kw)
    g, o = dense_cfgs(P, **args)
    X, y = synthdata.gaussian_mixture(args["N"], widths[0], widths[-1], seed=1)
    return g, o, X, y


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_checkpoint_resume_is_bitwise(P, prec):
    pr = P.FP32 if prec == "fp32" else P.BF16
    g, o, X, y = _small(P, pr)
    a = P.lsgd_create(g)
    P.lsgd_set_dataset(a, X, y)
    P.lsgd_run(a, 12)
    want = [P.lsgd_params(a, k) for k in range(4)]
    b = P.lsgd_create(g)
    P.lsgd_set_dataset(b, X, y)
    P.lsgd_run(b, 5)
    with tempfile.TemporaryDirectory() as d:
        path = os.path.join(d, "ck.bin")
        P.lsgd_save(b, path)
        c = P.lsgd_create(g)
        P.lsgd_set_dataset(c, X, y)
        P.lsgd_load(c, path)
    assert P.lsgd_step_count(c) == 5 and P.lsgd_sync_count(c) == P.lsgd_sync_count(b)
    P.lsgd_run(c, 7)
    for k in range(4):
        assert np.array_equal(P.lsgd_params(c, k), want[k])
    assert P.lsgd_sync_count(c) == P.lsgd_sync_count(a) == 4
    for h in (a, b, c):
        P.lsgd_destroy(h)


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_caller_batches_equal_sampled_steps(P, prec):
    import torch

    pr = P.FP32 if prec == "fp32" else P.BF16
    g, o, X, y = _small(P, pr)
    a = P.lsgd_create(g)
    P.lsgd_set_dataset(a, X, y)
    b = P.lsgd_create(g)
    P.lsgd_set_dataset(b, X, y)
    for s in range(3):
        P.lsgd_local_step(a)
        idx = P.lsgd_debug_indices(b, s, 4, 16)
        xb = torch.from_numpy(X[idx.reshape(-1)].reshape(4, 16, -1).copy()).pin_memory()
        yb = torch.from_numpy(y[idx.reshape(-1)].reshape(4, 16).copy()).pin_memory()
        if s == 1:
            xb, yb = xb.cuda(), yb.cuda()
        P.lsgd_local_step_batch(b, xb, yb)
    torch.cuda.synchronize()
    for k in range(4):
        assert np.array_equal(P.lsgd_params(a, k), P.lsgd_params(b, k))
    assert np.array_equal(P.lsgd_losses(a, 3, 4), P.lsgd_losses(b, 3, 4))
    P.lsgd_destroy(a)
    P.lsgd_destroy(b)


def test_pipelined_host_batches_equal_sampled_steps(P):
    # Seven host batches enqueued back to back with asynchronous loss reads: the copies run ahead
    # on the library's copy stream through its two staging buffers, and every step must still
    # see its own batch (a buffer overwritten before its gather ran would change the result).
    import torch

    g, o, X, y = _small(P, P.BF16, T=8, H=3)
    a = P.lsgd_create(g)
    P.lsgd_set_dataset(a, X, y)
    b = P.lsgd_create(g)
    P.lsgd_set_dataset(b, X, y)
    n = 7
    batches = []
    for s in range(n):
        idx = P.lsgd_debug_indices(b, s, 4, 16).reshape(-1)
        xb = torch.from_numpy(X[idx].reshape(4, 16, -1).copy())
        yb = torch.from_numpy(y[idx].reshape(4, 16).copy())
        if s != 4:  # one pageable batch among the pinned ones
            xb, yb = xb.pin_memory(), yb.pin_memory()
        batches.append((xb, yb))
    losses = torch.zeros((n, 4), dtype=torch.float32).pin_memory()
    for s in range(n):
        P.lsgd_local_step(a)
        P.lsgd_local_step_batch(b, *batches[s])
        if (s + 1) % 3 == 0:
            P.lsgd_sync_average(a)
            P.lsgd_sync_average(b)
        P.lsgd_losses_async(b, losses[s], 1)
    P.lsgd_synchronize(b)
    for k in range(4):
        assert np.array_equal(P.lsgd_params(a, k), P.lsgd_params(b, k))
    assert np.array_equal(P.lsgd_losses(a, n, 4), losses.numpy())
    P.lsgd_destroy(a)
    P.lsgd_destroy(b)


def test_least_squares_host_batches_equal_sampled_steps(P):
    # Targets (fp32) instead of labels travel through the same staging buffers.
    import torch

    N, dd, K, B = 256, 20, 4, 16
    A, t, _ = synthdata.least_squares(N, dd, seed=3)
    g, o = dense_cfgs(P, widths=(dd, 1), K=K, B=B, H=3, T=6, N=N, precision=P.FP32, kind="lsq",
                      base_lr=0.02, seed=5, init="zero")
    a = P.lsgd_create(g)
    P.lsgd_set_targets(a, A, t)
    b = P.lsgd_create(g)
    P.lsgd_set_targets(b, A, t)
    batches = []
    for s in range(6):
        idx = P.lsgd_debug_indices(b, s, K, B).reshape(-1)
        batches.append((torch.from_numpy(A[idx].reshape(K, B, -1).copy()).pin_memory(),
                        torch.from_numpy(t[idx].reshape(K, B).copy()).pin_memory()))
    for s in range(6):
        P.lsgd_local_step(a)
        P.lsgd_local_step_batch(b, *batches[s])
        if (s + 1) % 3 == 0:
            P.lsgd_sync_average(a)
            P.lsgd_sync_average(b)
    P.lsgd_synchronize(b)
    for k in range(K):
        assert np.array_equal(P.lsgd_params(a, k), P.lsgd_params(b, k))
    assert np.array_equal(P.lsgd_losses(a, 6, K), P.lsgd_losses(b, 6, K))
    P.lsgd_destroy(a)
    P.lsgd_destroy(b)


def test_set_step_restarts_the_schedule(P):
    # A job run to its end, then lsgd_set_step(0) and three more steps, equals a fresh context
    # given the end state (parameters and momentum) and run three steps from step 0: the step
    # counter alone decides learning rate, sampled mini-batches and round ends.
    g, o, X, y = _small(P, P.BF16, T=7, H=3)
    a = P.lsgd_create(g)
    P.lsgd_set_dataset(a, X, y)
    P.lsgd_run(a, 7)
    assert P.lsgd_step_count(a) == 7 and P.lsgd_sync_count(a) == 3
    W = [P.lsgd_params(a, k) for k in range(4)]
    U = [P.lsgd_momentum(a, k) for k in range(4)]
    P.lsgd_set_step(a, 0)
    assert P.lsgd_step_count(a) == 0
    P.lsgd_run(a, 3)
    c = P.lsgd_create(g)
    P.lsgd_set_dataset(c, X, y)
    for k in range(4):
        P.lsgd_set_params(c, k, W[k])
        P.lsgd_set_momentum(c, k, U[k])
    P.lsgd_run(c, 3)
    for k in range(4):
        assert np.array_equal(P.lsgd_params(a, k), P.lsgd_params(c, k))
        assert np.array_equal(P.lsgd_momentum(a, k), P.lsgd_momentum(c, k))
    assert np.array_equal(P.lsgd_losses(a, 3, 4), P.lsgd_losses(c, 3, 4))
    assert P.lsgd_sync_count(a) == 3 + P.lsgd_sync_count(c) == 4
    for bad in (-1, 8):
        with pytest.raises(P.LsgdError):
            P.lsgd_set_step(a, bad)
    P.lsgd_destroy(a)
    P.lsgd_destroy(c)


def test_sync_counts_follow_schedule(P):
    for T, H, tp in [(49, 16, -1), (25, 16, 12), (10, 3, 0), (9, 4, 20)]:
        g, o, X, y = _small(P, P.BF16, T=T, H=H, t_switch=tp)
        ctx = P.lsgd_create(g)
        P.lsgd_set_dataset(ctx, X, y)
        P.lsgd_run(ctx, T)
        assert P.lsgd_sync_count(ctx) == sum(oracle.is_round_end(o, s) for s in range(T))
        # the run ends synchronised: every replica holds the average
        w0 = P.lsgd_params(ctx, 0)
        assert all(np.array_equal(w0, P.lsgd_params(ctx, k)) for k in range(1, 4))
        for s in (0, T // 2, T - 1):
            assert abs(P.lsgd_lr_at(ctx, s) - oracle.lr(o, s)) < 1e-12
        P.lsgd_destroy(ctx)


def test_errors(P):
    g, o, X, y = _small(P, P.BF16)
    ctx = P.lsgd_create(g)
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_local_step(ctx)
    assert e.value.status == P.ESTATE
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_set_dataset(ctx, X[:100], y[:100])
    assert e.value.status == P.EINVAL
    bad = y.copy()
    bad[3] = 10
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_set_dataset(ctx, X, bad)
    assert e.value.status == P.EINVAL
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_params(ctx, 4)
    assert e.value.status == P.EINVAL
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_run(ctx, 2)
    assert P.lsgd_check_finite(ctx)
    w = P.lsgd_params(ctx, 1)
    w[17] = np.nan
    P.lsgd_set_params(ctx, 1, w)
    assert not P.lsgd_check_finite(ctx)
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_load(ctx, "/nonexistent/ck.bin")
    assert e.value.status == P.EIO
    P.lsgd_destroy(ctx)


def test_failed_allocation_reports_enomem(P):
    import torch

    calls = {"n": 0}

    def _alloc(user, nbytes, stream):
        calls["n"] += 1
        if calls["n"] >= 3:
            return None  # injected allocation failure
        return torch.cuda.caching_allocator_alloc(int(nbytes), 0, stream)

    def _free(user, p, stream):
        torch.cuda.caching_allocator_delete(p)

    cb = (P.ALLOC_FN(_alloc), P.FREE_FN(_free))
    a = P.Allocator(cb[0], cb[1], None)
    g, o, X, y = _small(P, P.FP32)
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_create(g, allocator=a)
    assert e.value.status == P.ENOMEM
    # a fresh context still works afterwards
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_run(ctx, 1)
    P.lsgd_destroy(ctx)


def test_default_allocator_and_launch_count(P):
    g, o, X, y = _small(P, P.BF16)
    ctx = P.lsgd_create(g, allocator=None)
    P.lsgd_set_dataset(ctx, X, y)
    before = P.lsgd_kernel_launches(ctx)
    P.lsgd_local_step(ctx)
    per_step = P.lsgd_kernel_launches(ctx) - before
    # sample, gather, the first layer's forward GEMM, the classifier head's two kernels (last
    # layer forward, loss and the data gradient below; the head's gradients and the first layer's
    # bias gradient), the first layer's weight-gradient GEMM, the update
    assert per_step == 7
    P.lsgd_destroy(ctx)
