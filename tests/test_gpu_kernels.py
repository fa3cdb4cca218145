"""GPU parity of the stand-alone kernels against the oracle: mini-batch indices (bit-exact), He
initialisation, the fused momentum-SGD update and the K-way average (Eq. 2 right, 1e-6 relative)."""
import numpy as np
import pytest

import oracle
from _gpu_common import built_package, dense_cfgs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    return built_package()


@pytest.fixture(scope="module")
def torch():
    import torch

    assert torch.cuda.is_available()
    return torch


@pytest.mark.parametrize("K,B,N,seed", [(4, 32, 8192, 0), (16, 128, 50000, 1), (64, 32, 50000, 2),
                                        (3, 5, 31, 7), (1, 1, 1, 0), (8, 33, 50000, 2**40 + 5)])
def test_indices_bit_exact(P, torch, K, B, N, seed):
    dst = torch.empty((K, B), dtype=torch.int32, device="cuda")
    oc = oracle.make_cfg(K=K, B=B, N=N, seed=seed)
    for step in (0, 1, 7, 123456):
        P.lsgd_sample_indices(dst, seed, step, K, B, N)
        torch.cuda.synchronize()
        got = dst.cpu().numpy()
        want = np.stack([oracle.sample_indices(oc, k, step) for k in range(K)])
        assert np.array_equal(got, want), (step,)


def test_context_indices_and_init_match_oracle(P, torch):
    g, o = dense_cfgs(P, widths=(3072, 1024, 1024, 10), K=16, B=128, H=16, T=49, N=50000,
                      precision=P.BF16, seed=11)
    ctx = P.lsgd_create(g)
    w0 = P.lsgd_params(ctx, 3)
    want = oracle.init_params(o)
    assert np.abs(w0 - want).max() <= 1e-6 * np.abs(want).max()
    # every replica starts from the same model (Algorithm 1 synchronises the initial models)
    assert np.array_equal(P.lsgd_params(ctx, 0), P.lsgd_params(ctx, 15))
    for step in (0, 48):
        got = P.lsgd_debug_indices(ctx, step, 16, 128)
        assert np.array_equal(got, np.stack([oracle.sample_indices(o, k, step) for k in range(16)]))
    P.lsgd_destroy(ctx)


def _assert_average_bar(got, W0, ref):
    """The averaging bar: max_i |a_i - o_i| / ((1/K) sum_k |w_k,i|) <= 1e-6 (relative in fp32,
    normalised so that cancellation between replicas is not penalised)."""
    scale = np.abs(W0).mean(0)
    rel = np.abs(got.astype(np.float64) - ref) / np.maximum(scale, 1e-30)
    assert rel.max() <= 1e-6, float(rel.max())
    return rel


@pytest.mark.parametrize("K,d", [(1, 4), (2, 4096), (3, 1028), (4, 4096 + 36), (5, 8192),
                                 (16, 67 * 1024 + 12), (33, 96), (64, 2052), (64, 65536),
                                 (100, 4096), (1024, 512)])
def test_kway_average(P, torch, K, d):
    gen = torch.Generator(device="cuda").manual_seed(K * 1000 + d)
    W = torch.randn((K, d), device="cuda", generator=gen, dtype=torch.float32) * 3
    Wb = torch.zeros((K, d), device="cuda", dtype=torch.bfloat16)
    W0 = W.cpu().numpy().astype(np.float64)
    ref = oracle.average(W0)[0]
    P.lsgd_kway_average(W, Wb, K, d)
    torch.cuda.synchronize()
    got = W.cpu().numpy()
    # every replica holds exactly the same mean afterwards
    assert all(np.array_equal(got[0], got[k]) for k in range(K))
    _assert_average_bar(got[0], W0, ref)
    # the compensated sum makes the mean the correctly rounded fp32 value of the exact mean
    # except in rare midpoint cases
    assert np.mean(got[0] == ref.astype(np.float32)) >= 0.999
    assert torch.equal(Wb.float(), W.to(torch.bfloat16).float())


@pytest.mark.parametrize("K", [3, 16, 64])
def test_kway_average_of_close_replicas_meets_1e6(P, torch, K):
    # Replicas a local-SGD round apart (relative spread 1e-3), the case every sync of a run sees.
    d = 4 * 2053
    gen = torch.Generator(device="cuda").manual_seed(K)
    w = torch.randn(d, device="cuda", generator=gen)
    W = (w[None, :] * (1 + 1e-3 * torch.randn((K, d), device="cuda", generator=gen))).contiguous()
    W0 = W.cpu().numpy().astype(np.float64)
    ref = W0.mean(0)
    P.lsgd_kway_average(W, None, K, d)
    torch.cuda.synchronize()
    got = W[0].cpu().numpy()
    rel = _assert_average_bar(got, W0, ref)
    # within one rounding of the exact mean
    assert rel.max() <= 2.0 ** -23, float(rel.max())


@pytest.mark.parametrize("K", [3, 8, 33])
def test_kway_average_of_identical_replicas_is_identity(P, torch, K):
    w = torch.randn(4096, device="cuda") * 3
    W = w.repeat(K, 1).contiguous()
    P.lsgd_kway_average(W, None, K, 4096)
    torch.cuda.synchronize()
    assert torch.equal(W[K - 1], w)


def test_block_average_meets_1e6(P, torch):
    # hierarchical local SGD's block average (Sec. D) runs the same kernel once per block
    K, block, widths = 16, 4, (64, 40, 10)
    cfg = P.make_config(K=K, B_loc=4, H=2, total_steps=8, N=64, widths=widths, seed=1,
                        precision=P.FP32, hier_block=block, hier_rounds=2)
    ctx = P.lsgd_create(cfg)
    d = P.lsgd_num_params(ctx)
    rng = np.random.default_rng(9)
    W0 = (rng.standard_normal((K, d)) * 2).astype(np.float32)
    for k in range(K):
        P.lsgd_set_params(ctx, k, W0[k])
    P.lsgd_block_average(ctx)
    got = np.stack([P.lsgd_params(ctx, k) for k in range(K)])
    ref = oracle.block_average(W0.astype(np.float64), block)
    for g in range(K // block):
        rows = slice(g * block, (g + 1) * block)
        _assert_average_bar(got[g * block], W0[rows].astype(np.float64), ref[g * block])
        assert all(np.array_equal(got[g * block], got[k]) for k in range(g * block, (g + 1) * block))
    P.lsgd_destroy(ctx)


@pytest.mark.parametrize("mom,nest,wd", [(0.0, False, 0.0), (0.9, False, 0.0), (0.9, True, 5e-4),
                                         (0.0, False, 1e-4)])
def test_sgd_update(P, torch, mom, nest, wd):
    n = 4 * 10007
    gen = torch.Generator(device="cuda").manual_seed(3)
    w = torch.randn(n, device="cuda", generator=gen)
    u = torch.randn(n, device="cuda", generator=gen)
    g = torch.randn(n, device="cuda", generator=gen)
    wb = torch.zeros(n, device="cuda", dtype=torch.bfloat16)
    oc = oracle.make_cfg(widths=(n, 1), has_bias=False, momentum=mom, nesterov=nest, weight_decay=wd)
    w_ref, u_ref = oracle.sgd_update(oc, 0.05, w.cpu().numpy(), u.cpu().numpy(), g.cpu().numpy())
    P.lsgd_sgd_update(w, u, g, wb, n, 0.05, mom, nest, wd)
    torch.cuda.synchronize()
    np.testing.assert_allclose(w.cpu().numpy(), w_ref, rtol=1e-6, atol=1e-6)
    if mom != 0.0:
        np.testing.assert_allclose(u.cpu().numpy(), u_ref, rtol=1e-6, atol=1e-6)
    assert torch.equal(wb.float(), w.to(torch.bfloat16).float())


def test_sgd_update_decay_region(P, torch):
    # weight decay only where (i mod period) < decay_end (BatchNorm gamma / beta are exempt, Sec. A.4)
    period, end, K = 64, 40, 3
    n = period * K
    w = torch.ones(n, device="cuda")
    g = torch.zeros(n, device="cuda")
    P.lsgd_sgd_update(w, None, g, None, n, 1.0, 0.0, False, 0.5, period, end)
    torch.cuda.synchronize()
    got = w.cpu().numpy().reshape(K, period)
    assert np.all(got[:, :end] == 0.5) and np.all(got[:, end:] == 1.0)


def test_bad_arguments_are_rejected(P, torch):
    W = torch.zeros(10, device="cuda")
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_kway_average(W, None, 2, 5)  # d not a multiple of 4
    assert e.value.status == P.EINVAL
    with pytest.raises(P.LsgdError):
        P.lsgd_sgd_update(W, None, W, None, 6, 0.1, 0.9)  # momentum without a buffer


@pytest.mark.parametrize("G,n,C", [(16, 131072, 16), (3, 1000, 64), (2, 2049, 3), (1, 1, 8)])
def test_batchnorm_stats(P, torch, G, n, C):
    # mean and biased variance over the positions of each replica (numpy fp64 as the definition);
    # an offset mean tests the two-pass / pairwise-combination variance
    gen = torch.Generator(device="cuda").manual_seed(G * 7 + C)
    y = torch.randn((G, n, C), device="cuda", generator=gen) * 2.0 + 5.0
    mean = torch.empty((G, C), device="cuda")
    rstd = torch.empty((G, C), device="cuda")
    P.lsgd_batchnorm_stats(y, n, C, G, mean, rstd)
    torch.cuda.synchronize()
    yn = y.double().cpu().numpy()
    m = yn.mean(axis=1)
    r = 1.0 / np.sqrt(yn.var(axis=1) + 1e-5)
    np.testing.assert_allclose(mean.cpu().numpy(), m, rtol=1e-5, atol=1e-5)
    np.testing.assert_allclose(rstd.cpu().numpy(), r, rtol=1e-4)
    with pytest.raises(P.LsgdError):
        P.lsgd_batchnorm_stats(y, n, 300, G, mean, rstd)
