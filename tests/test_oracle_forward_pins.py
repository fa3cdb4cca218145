"""Pin the oracle's forward passes (and with them Eq. 2's per-sample gradients) against independent
definitions written with PyTorch CPU operators in fp64: a dense network with ReLU on every hidden
layer and softmax cross-entropy on the logits, and a reduced ResNet-20 (Sec. 4 / A.2: stem,
three stages with stride-2 option-A shortcut blocks, batch-statistics BatchNorm, residual
branches, average pooling, classifier) with non-zero residual branches.

Finite differences only show that the oracle's gradient follows its own loss; these tests check
the loss itself and every gradient entry against autograd of a separately written network, so a
ReLU left off a hidden layer or put on the logits, a wrong stride-2 window, a shortcut added in
the wrong place or a BatchNorm with the wrong variance fails here.  In bf16 mode the independent
network rounds exactly the operands the accelerated path stores in bf16 (input, weights, stored
activations on the forward pass; the output gradient of every product on the backward pass).
"""
import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")
F = torch.nn.functional


def _bf16(t):
    """fp64 -> fp32 -> bf16 (round to nearest even) -> fp64, as the oracle stores bf16 operands."""
    return t.to(torch.float32).to(torch.bfloat16).to(torch.float64)


class _RoundValue(torch.autograd.Function):
    """Forward: the stored bf16 value; backward: the gradient passes unchanged."""

    @staticmethod
    def forward(ctx, x):
        return _bf16(x)

    @staticmethod
    def backward(ctx, g):
        return g


class _RoundGrad(torch.autograd.Function):
    """Forward: identity; backward: the gradient is stored as bf16 before the products use it."""

    @staticmethod
    def forward(ctx, x):
        return x.clone()

    @staticmethod
    def backward(ctx, g):
        return _bf16(g)


def _maybe(fn, on):
    return fn.apply if on else (lambda t: t)


# ------------------------------------------------------------------------------------------------
# dense networks


def _torch_dense(widths, has_bias, w, X, y, bf16):
    """Mean softmax cross-entropy of z_L, z_l = a_{l-1} W_l^T + b_l, a_l = relu(z_l) (l < L)."""
    rv, rg = _maybe(_RoundValue, bf16), _maybe(_RoundGrad, bf16)
    wt = torch.tensor(w, dtype=torch.float64, requires_grad=True)
    a = rv(torch.tensor(X, dtype=torch.float64))
    off, L = 0, len(widths) - 1
    for l in range(L):
        fin, fout = widths[l], widths[l + 1]
        W = wt[off:off + fin * fout].view(fout, fin)
        off += fin * fout
        z = a @ rv(W).T
        if has_bias:
            z = z + wt[off:off + fout]
            off += fout
        z = rg(z)
        a = rv(torch.relu(z)) if l + 1 < L else z
    loss = F.cross_entropy(a, torch.tensor(y, dtype=torch.int64))
    loss.backward()
    return float(loss.detach()), wt.grad.numpy()


@pytest.mark.parametrize("widths,has_bias,bf16", [
    ((12, 9, 7, 5), True, False),
    ((12, 9, 7, 5), True, True),
    ((10, 16, 8, 8, 4), True, False),
    ((10, 16, 8, 8, 4), False, True),
    ((24, 32, 3), True, True),
])
def test_dense_forward_and_gradient_match_independent_network(widths, has_bias, bf16):
    B, N = 7, 30
    rng = np.random.default_rng(sum(widths) + 3 * bf16)
    X = (rng.standard_normal((N, widths[0])) * 2.0).astype(np.float32)
    y = rng.integers(0, widths[-1], N).astype(np.int32)
    idx = rng.integers(0, N, B).astype(np.int32)
    c = oracle.make_cfg(widths=widths, has_bias=has_bias, bf16=bf16, B=B, N=N)
    # weights and biases large enough that many hidden units are active and many are not
    w = rng.standard_normal(oracle.num_params(c)) * 0.6
    loss, g = oracle.loss_grad(c, w, X, y=y, idx=idx)
    want_loss, want_g = _torch_dense(widths, has_bias, w, X[idx], y[idx], bf16)
    assert abs(loss - want_loss) <= 1e-12 * max(1.0, abs(want_loss)), (loss, want_loss)
    np.testing.assert_allclose(g, want_g, rtol=1e-9, atol=1e-12 * np.abs(want_g).max())


def test_dense_pin_detects_a_relu_on_the_logits():
    # the independent network with a ReLU on the logits gives a clearly different loss: the pin
    # above would reject an oracle that did this
    widths, B, N = (12, 9, 5), 6, 20
    rng = np.random.default_rng(1)
    X = rng.standard_normal((N, 12)).astype(np.float32)
    y = rng.integers(0, 5, N).astype(np.int32)
    idx = np.arange(B, dtype=np.int32)
    c = oracle.make_cfg(widths=widths, B=B, N=N)
    w = rng.standard_normal(oracle.num_params(c))
    loss, _ = oracle.loss_grad(c, w, X, y=y, idx=idx)
    wt = torch.tensor(w)
    W1, b1 = wt[:108].view(9, 12), wt[108:117]
    W2, b2 = wt[117:162].view(5, 9), wt[162:]
    xt = torch.tensor(X[idx], dtype=torch.float64)
    logits = torch.relu(xt @ W1.T + b1) @ W2.T + b2
    wrong = float(F.cross_entropy(torch.relu(logits), torch.tensor(y[idx], dtype=torch.int64)))
    right = float(F.cross_entropy(logits, torch.tensor(y[idx], dtype=torch.int64)))
    assert abs(loss - right) < 1e-12 and abs(loss - wrong) > 1e-3


# ------------------------------------------------------------------------------------------------
# ResNet-20 (reduced widths and image size, same topology)


def _resnet_layout(in_c, base, blocks, classes):
    """Canonical parameter order: per convolution (stem first, then two per block) its weight
    [Cout][3][3][Cin], BN gamma, BN beta; then the classifier W [classes][4 base] and b."""
    convs, off = [], 0

    def add(cin, cout, stride):
        nonlocal off
        spec = dict(cin=cin, cout=cout, stride=stride, w=off)
        off += cout * 9 * cin
        spec["g"] = off
        off += cout
        spec["b"] = off
        off += cout
        convs.append(spec)

    add(in_c, base, 1)
    ch = base
    for st in range(3):
        cout = base << st
        for b in range(blocks):
            add(ch, cout, 2 if (st > 0 and b == 0) else 1)
            add(cout, cout, 1)
            ch = cout
    fc_w = off
    off += classes * ch
    fc_b = off
    off += classes
    return convs, fc_w, fc_b, off


def _torch_resnet(geom, w, X, y, bf16):
    H, W_, C0, base, blocks, classes = geom
    rv, rg = _maybe(_RoundValue, bf16), _maybe(_RoundGrad, bf16)
    convs, fc_w, fc_b, total = _resnet_layout(C0, base, blocks, classes)
    assert total == len(w)
    wt = torch.tensor(w, dtype=torch.float64, requires_grad=True)
    B = X.shape[0]
    x = torch.tensor(X, dtype=torch.float64).view(B, H, W_, C0).permute(0, 3, 1, 2)  # HWC -> NCHW
    x = rv(x)

    def conv_bn(inp, s):
        k = wt[s["w"]:s["w"] + s["cout"] * 9 * s["cin"]].view(s["cout"], 3, 3, s["cin"])
        k = rv(k.permute(0, 3, 1, 2))  # [Cout][3][3][Cin] -> OIHW
        yconv = rg(F.conv2d(inp, k, stride=s["stride"], padding=1))
        gamma = wt[s["g"]:s["g"] + s["cout"]]
        beta = wt[s["b"]:s["b"] + s["cout"]]
        # batch statistics of this worker's mini-batch, biased variance, eps 1e-5
        return F.batch_norm(yconv, None, None, gamma, beta, training=True, eps=1e-5)

    cur = rv(torch.relu(conv_bn(x, convs[0])))
    for blk in range(3 * blocks):
        sa, sb = convs[1 + 2 * blk], convs[2 + 2 * blk]
        h = rv(torch.relu(conv_bn(cur, sa)))
        z = conv_bn(h, sb)
        # option A: spatial subsampling, zero channels appended after the input's channels
        shortcut = cur[:, :, ::sa["stride"], ::sa["stride"]]
        shortcut = F.pad(shortcut, (0, 0, 0, 0, 0, sa["cout"] - sa["cin"]))
        cur = rv(torch.relu(z + shortcut))
    feat = cur.mean(dim=(2, 3))
    Wfc = wt[fc_w:fc_w + classes * 4 * base].view(classes, 4 * base)
    logits = feat @ Wfc.T + wt[fc_b:fc_b + classes]
    loss = F.cross_entropy(logits, torch.tensor(y, dtype=torch.int64))
    loss.backward()
    return float(loss.detach()), wt.grad.numpy()


@pytest.mark.parametrize("geom,B,bf16", [
    ((8, 8, 3, 4, 1, 5), 3, False),
    ((8, 8, 3, 4, 2, 5), 2, False),
    ((6, 6, 3, 2, 2, 3), 3, False),   # odd sizes: 6 -> 3 -> 2 under the stride-2 convolutions
    ((8, 8, 3, 4, 1, 5), 3, True),
    ((6, 6, 3, 2, 2, 3), 2, True),
])
def test_resnet_forward_and_gradient_match_independent_network(geom, B, bf16):
    H, W_, C0, base, blocks, classes = geom
    N = 8
    rng = np.random.default_rng(H * 100 + base * 10 + blocks + 7 * bf16)
    X = (rng.standard_normal((N, H * W_ * C0)) * 1.5).astype(np.float32)
    y = rng.integers(0, classes, N).astype(np.int32)
    idx = rng.choice(N, B, replace=False).astype(np.int32)
    c = oracle.make_cfg(kind=oracle.RESNET20, in_hwc=(H, W_, C0), base_ch=base,
                        res_blocks=blocks, n_classes=classes, bf16=bf16, B=B, N=N)
    convs, fc_w, fc_b, total = _resnet_layout(C0, base, blocks, classes)
    assert oracle.num_params(c) == total
    # non-zero residual branches: perturbed He weights, BN gamma around 1, beta around 0, a
    # classifier large enough that the logits differ
    w = oracle.init_params(c) + 0.2 * rng.standard_normal(total)
    for s in convs:
        w[s["g"]:s["g"] + s["cout"]] = 1.0 + 0.3 * rng.standard_normal(s["cout"])
        w[s["b"]:s["b"] + s["cout"]] = 0.3 * rng.standard_normal(s["cout"])
    w[fc_w:fc_b] = 0.5 * rng.standard_normal(fc_b - fc_w)
    loss, g = oracle.loss_grad(c, w, X, y=y, idx=idx)
    want_loss, want_g = _torch_resnet(geom, w, X[idx], y[idx], bf16)
    assert abs(loss - want_loss) <= 1e-11 * max(1.0, abs(want_loss)), (loss, want_loss)
    np.testing.assert_allclose(g, want_g, rtol=1e-8, atol=1e-10 * np.abs(want_g).max())


def test_resnet_pin_needs_the_residual_branch():
    # the same network without its residual branches (the shortcut alone) gives another loss, so
    # the pin above constrains the branch's forward, not only the shortcut path
    geom, B, N = (8, 8, 3, 4, 1, 5), 3, 8
    H, W_, C0, base, blocks, classes = geom
    rng = np.random.default_rng(5)
    X = rng.standard_normal((N, H * W_ * C0)).astype(np.float32)
    y = rng.integers(0, classes, N).astype(np.int32)
    idx = np.arange(B, dtype=np.int32)
    c = oracle.make_cfg(kind=oracle.RESNET20, in_hwc=(H, W_, C0), base_ch=base, res_blocks=blocks,
                        n_classes=classes, B=B, N=N)
    convs, fc_w, fc_b, total = _resnet_layout(C0, base, blocks, classes)
    w = oracle.init_params(c) + 0.2 * rng.standard_normal(total)
    w[fc_w:fc_b] = 0.5 * rng.standard_normal(fc_b - fc_w)
    loss, _ = oracle.loss_grad(c, w, X, y=y, idx=idx)
    w_cut = w.copy()
    for s in convs[2::2]:  # second BN of every block: gamma = beta = 0 removes the branch
        w_cut[s["g"]:s["g"] + s["cout"]] = 0.0
        w_cut[s["b"]:s["b"] + s["cout"]] = 0.0
    loss_cut, _ = oracle.loss_grad(c, w_cut, X, y=y, idx=idx)
    want, _ = _torch_resnet(geom, w, X[idx], y[idx], False)
    assert abs(loss - want) < 1e-11 and abs(loss_cut - want) > 1e-4
