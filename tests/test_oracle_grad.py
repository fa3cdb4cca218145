"""Pin the oracle's gradients (the (1/B) sum of per-sample gradients of Eq. 2) against central finite
differences of its own loss, in fp64, on tiny models: softmax regression, an MLP, least squares and
a reduced ResNet-20 (same topology: stem, 3 stages with option-A shortcuts, batch-stat BN, pooling,
classifier)."""
import numpy as np
import pytest

import oracle


def _fd_check(c, w, X, y=None, t=None, idx=None, h=1e-5, tol=1e-6, n_check=None, seed=0):
    loss, g = oracle.loss_grad(c, w, X, y=y, t=t, idx=idx)
    d = len(w)
    coords = np.arange(d)
    if n_check is not None and n_check < d:
        coords = np.random.default_rng(seed).choice(d, n_check, replace=False)
    fd = np.zeros(len(coords))
    for n, i in enumerate(coords):
        wp = w.copy()
        wp[i] += h
        wm = w.copy()
        wm[i] -= h
        fd[n] = (oracle.loss_grad(c, wp, X, y=y, t=t, idx=idx)[0]
                 - oracle.loss_grad(c, wm, X, y=y, t=t, idx=idx)[0]) / (2 * h)
    err = np.max(np.abs(fd - g[coords])) / max(np.max(np.abs(fd)), 1e-30)
    assert err <= tol, err
    return loss, g


def _data(N, D, C, seed):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((N, D)).astype(np.float32)
    y = rng.integers(0, C, N).astype(np.int32)
    return X, y


def test_fd_softmax_regression():
    c = oracle.make_cfg(widths=(7, 4), B=5, N=20)
    X, y = _data(20, 7, 4, 1)
    w = np.random.default_rng(2).standard_normal(oracle.num_params(c))
    _fd_check(c, w, X, y=y, idx=np.array([3, 9, 9, 0, 17]))


def test_fd_mlp():
    c = oracle.make_cfg(widths=(6, 5, 4, 3), B=3, N=10)
    X, y = _data(10, 6, 3, 3)
    w = np.random.default_rng(4).standard_normal(oracle.num_params(c))
    _fd_check(c, w, X, y=y, idx=np.array([1, 4, 8]))


def test_fd_mlp_without_bias():
    c = oracle.make_cfg(widths=(6, 5, 3), has_bias=False, B=4, N=10)
    X, y = _data(10, 6, 3, 5)
    w = np.random.default_rng(6).standard_normal(oracle.num_params(c))
    _fd_check(c, w, X, y=y, idx=np.array([0, 1, 2, 3]))


def test_fd_least_squares():
    c = oracle.make_cfg(kind=oracle.LSQ, widths=(5, 1), has_bias=False, B=4, N=12)
    rng = np.random.default_rng(7)
    X = rng.standard_normal((12, 5)).astype(np.float32)
    t = rng.standard_normal(12).astype(np.float32)
    w = rng.standard_normal(5)
    loss, g = _fd_check(c, w, X, t=t, idx=np.array([2, 5, 5, 11]))
    # closed form: (1/B) A^T (A w - t) on the batch rows
    A = X[[2, 5, 5, 11]].astype(np.float64)
    r = A @ w - t[[2, 5, 5, 11]]
    np.testing.assert_allclose(g, A.T @ r / 4, rtol=1e-13, atol=1e-15)
    assert abs(loss - 0.5 * np.mean(r * r)) < 1e-14


def _tiny_resnet(**kw):
    args = dict(kind=oracle.RESNET20, in_hwc=(8, 8, 3), base_ch=2, res_blocks=1, n_classes=3, B=3,
                N=6)
    args.update(kw)
    return oracle.make_cfg(**args)


def test_fd_tiny_resnet():
    c = _tiny_resnet()
    X, y = _data(6, 8 * 8 * 3, 3, 8)
    rng = np.random.default_rng(9)
    w = oracle.init_params(c) + 0.1 * rng.standard_normal(oracle.num_params(c))
    _fd_check(c, w, X, y=y, idx=np.array([0, 2, 5]), tol=2e-6, n_check=400)


def test_fd_tiny_resnet_two_blocks_odd_size():
    c = _tiny_resnet(in_hwc=(6, 6, 3), res_blocks=2, B=2)
    X, y = _data(6, 6 * 6 * 3, 3, 10)
    rng = np.random.default_rng(11)
    w = oracle.init_params(c) + 0.1 * rng.standard_normal(oracle.num_params(c))
    _fd_check(c, w, X, y=y, idx=np.array([1, 4]), tol=2e-6, n_check=300)


def test_softmax_regression_matches_closed_form_gradient():
    # For one linear layer, dL/dW = (1/B) (softmax(XW^T+b) - onehot)^T X exactly.
    c = oracle.make_cfg(widths=(9, 5), B=6, N=6)
    X, y = _data(6, 9, 5, 12)
    w = np.random.default_rng(13).standard_normal(oracle.num_params(c))
    loss, g = oracle.loss_grad(c, w, X, y=y, idx=np.arange(6))
    W = w[:45].reshape(5, 9)
    b = w[45:]
    Z = X.astype(np.float64) @ W.T + b
    P = np.exp(Z - Z.max(1, keepdims=True))
    P /= P.sum(1, keepdims=True)
    E = P.copy()
    E[np.arange(6), y] -= 1
    np.testing.assert_allclose(g[:45].reshape(5, 9), E.T @ X.astype(np.float64) / 6, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(g[45:], E.sum(0) / 6, rtol=1e-12, atol=1e-14)
    assert abs(loss - np.mean(-np.log(P[np.arange(6), y]))) < 1e-12
