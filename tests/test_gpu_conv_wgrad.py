"""The convolution weight-gradient kernel (column matrix built in shared memory, tcgen05) against
an fp64 evaluation of its definition on the same bf16 operands:
    dW[g][co][kh][kw][ci] = sum over b, oy, ox of dy[g][b][oy][ox][co] x[g][b][s oy + kh - 1][s ox + kw - 1][ci]
(3x3 kernel, zero padding 1, stride s).  Every ResNet-20 shape (16 / 32 / 64 channels, both
strides, 32 / 16 / 8 wide outputs), several groups and several CTAs per group.  Error measure:
|dW - dW64| / (sum |dy| |x|) elementwise, the fp32 accumulation bound's scale; a wrong tap,
channel or halo row moves an element by ~1 / sqrt(terms) of that scale, far above the bar."""
import numpy as np
import pytest

from _gpu_common import built_package

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


def _reference(x, dy, stride):
    """fp64 weight gradient from the definition: pad the input, slice each tap's shifted view."""
    G, B, Hin, Win, Cin = x.shape
    Hout, Wout = dy.shape[2], dy.shape[3]
    xp = np.zeros((G, B, Hin + 2, Win + 2, Cin))
    xp[:, :, 1:Hin + 1, 1:Win + 1, :] = x
    dW = np.zeros((G, dy.shape[4], 3, 3, Cin))
    scale = np.zeros_like(dW)
    for kh in range(3):
        for kw in range(3):
            # input pixel (s oy + kh - 1, s ox + kw - 1) = padded pixel (s oy + kh, s ox + kw)
            v = xp[:, :, kh:kh + stride * Hout:stride, kw:kw + stride * Wout:stride, :]
            dW[:, :, kh, kw, :] = np.einsum("gbhwo,gbhwi->goi", dy, v)
            scale[:, :, kh, kw, :] = np.einsum("gbhwo,gbhwi->goi", np.abs(dy), np.abs(v))
    return dW, scale


SHAPES = [  # (G, B, Hout, Wout, Cin, Cout, stride)
    (2, 6, 32, 32, 16, 16, 1),
    (3, 4, 16, 16, 16, 32, 2),
    (2, 5, 16, 16, 32, 32, 1),
    (2, 6, 8, 8, 32, 64, 2),
    (3, 7, 8, 8, 64, 64, 1),
    (1, 3, 8, 16, 64, 48, 1),
    (4, 1, 8, 8, 16, 16, 1),
]


@pytest.mark.parametrize("shape", SHAPES)
def test_conv_wgrad_matches_fp64(P, shape):
    import torch

    G, B, Hout, Wout, Cin, Cout, s = shape
    gen = torch.Generator(device="cuda").manual_seed(sum(shape))
    x = torch.randn((G, B, s * Hout, s * Wout, Cin), device="cuda", generator=gen).to(torch.bfloat16)
    dy = torch.randn((G, B, Hout, Wout, Cout), device="cuda", generator=gen).to(torch.bfloat16)
    dW = torch.full((G, Cout, 3, 3, Cin), float("nan"), device="cuda")
    P.lsgd_conv_wgrad_bf16(x, dy, dW, G, B, Hout, Wout, Cin, Cout, s)
    torch.cuda.synchronize()
    want, scale = _reference(x.float().cpu().numpy().astype(np.float64),
                             dy.float().cpu().numpy().astype(np.float64), s)
    got = dW.cpu().numpy().astype(np.float64)
    err = np.abs(got - want) / scale
    assert np.isfinite(got).all()
    assert err.max() <= 1e-5, err.max()


def test_conv_wgrad_is_deterministic(P):
    import torch

    G, B, Hout, Wout, Cin, Cout, s = 2, 8, 32, 32, 16, 32, 1
    gen = torch.Generator(device="cuda").manual_seed(5)
    x = torch.randn((G, B, Hout, Wout, Cin), device="cuda", generator=gen).to(torch.bfloat16)
    dy = torch.randn((G, B, Hout, Wout, Cout), device="cuda", generator=gen).to(torch.bfloat16)
    outs = []
    for _ in range(2):
        dW = torch.empty((G, Cout, 3, 3, Cin), device="cuda")
        P.lsgd_conv_wgrad_bf16(x, dy, dW, G, B, Hout, Wout, Cin, Cout, s)
        outs.append(dW.cpu())
    assert torch.equal(outs[0], outs[1])


def test_conv_wgrad_rejects_unsupported_shapes(P):
    import torch

    x = torch.zeros((1, 1, 8, 8, 16), device="cuda", dtype=torch.bfloat16)
    dy = torch.zeros((1, 1, 8, 8, 16), device="cuda", dtype=torch.bfloat16)
    dW = torch.zeros((1, 16, 3, 3, 16), device="cuda")
    for bad in [dict(Cin=8), dict(Cout=8), dict(Cout=80), dict(stride=3), dict(Hout=4, Wout=4),
                dict(Wout=12)]:
        kw = dict(G=1, B=1, Hout=8, Wout=8, Cin=16, Cout=16, stride=1)
        kw.update(bad)
        with pytest.raises(P.LsgdError):
            P.lsgd_conv_wgrad_bf16(x, dy, dW, **kw)
