"""The persistent implicit-GEMM convolution kernel (tcgen05, TMA-shifted input tiles) in every mode
the ResNet-20 step runs it, element by element against an fp64 evaluation of the definition on
the same bf16 operands (3x3 kernel, zero padding 1; Sec. A.2's ResNet-20):

  forward        y[g][b][oy][ox][co] = sum_{kh,kw,ci} x[g][b][s oy + kh - 1][s ox + kw - 1][ci] w[g][co][kh][kw][ci]
  data gradient  dx[g][b][iy][ix][ci] = sum over (oy, ox, kh, kw) with iy = s oy + kh - 1,
                 ix = s ox + kw - 1 and co of dy[g][b][oy][ox][co] w[g][co][kh][kw][ci]

covering the stride-1 and stride-2 forwards, the 3-channel stem (padded to 16 channels), the
stride-1 data gradient (flipped, transposed weights) and the stride-2 data gradient (four parity
phases), at every ResNet-20 channel count and image size, with ragged batch sizes, several groups
and several 128-pixel tiles per CTA.  The call goes through lsgd_conv3x3_bf16, which runs the same
launch code as the training step.  Error measure: |out - out64| / sum |a| |b| per element, the
scale of the fp32 accumulation bound; a wrong tap, halo pixel or phase moves an element by about
1 / sqrt(terms) of that scale, far above the bar."""
import numpy as np
import pytest

from _gpu_common import built_package

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


def _taps(stride, Hout, Wout):
    """(kh, kw, padded-row slice, padded-column slice) of every tap: output pixel (oy, ox) reads
    padded input pixel (s oy + kh, s ox + kw)."""
    for kh in range(3):
        for kw in range(3):
            yield kh, kw, slice(kh, kh + stride * Hout, stride), slice(kw, kw + stride * Wout, stride)


def _forward64(x, w, stride):
    G, B, Hin, Win, Cin = x.shape
    Cout = w.shape[1]
    Hout, Wout = (Hin - 1) // stride + 1, (Win - 1) // stride + 1
    xp = np.zeros((G, B, Hin + 2, Win + 2, Cin))
    xp[:, :, 1:Hin + 1, 1:Win + 1, :] = x
    y = np.zeros((G, B * Hout * Wout, Cout))
    scale = np.zeros_like(y)
    for kh, kw, rs, cs in _taps(stride, Hout, Wout):
        v = xp[:, :, rs, cs, :].reshape(G, -1, Cin)
        wt = np.transpose(w[:, :, kh, kw, :], (0, 2, 1))  # [G][Cin][Cout]
        y += np.matmul(v, wt)
        scale += np.matmul(np.abs(v), np.abs(wt))
    return y.reshape(G, B, Hout, Wout, Cout), scale.reshape(G, B, Hout, Wout, Cout)


def _dgrad64(dy, w, stride, Hin, Win):
    G, B, Hout, Wout, Cout = dy.shape
    Cin = w.shape[4]
    dxp = np.zeros((G, B, Hin + 2, Win + 2, Cin))
    scp = np.zeros_like(dxp)
    d = dy.reshape(G, -1, Cout)
    for kh, kw, rs, cs in _taps(stride, Hout, Wout):
        wk = w[:, :, kh, kw, :]  # [G][Cout][Cin]
        dxp[:, :, rs, cs, :] += np.matmul(d, wk).reshape(G, B, Hout, Wout, Cin)
        scp[:, :, rs, cs, :] += np.matmul(np.abs(d), np.abs(wk)).reshape(G, B, Hout, Wout, Cin)
    return dxp[:, :, 1:Hin + 1, 1:Win + 1, :], scp[:, :, 1:Hin + 1, 1:Win + 1, :]


def _bf16_randn(torch, shape, gen):
    return torch.randn(shape, device="cuda", generator=gen).to(torch.bfloat16)


def _check(got, want, scale):
    got = got.cpu().numpy().astype(np.float64)
    assert np.isfinite(got).all(), "elements left unwritten"
    err = np.abs(got - want) / np.maximum(scale, 1e-30)
    assert err.max() <= 1e-5, (float(err.max()), np.unravel_index(err.argmax(), err.shape))


FORWARD = [  # (G, B, Hin, Win, Cin, Cout, stride): ResNet-20's forward convolutions
    (2, 3, 32, 32, 3, 16, 1),      # stem (3 channels, padded to 16)
    (3, 3, 32, 32, 16, 16, 1),     # stage 1
    (2, 5, 32, 32, 16, 32, 2),     # stage-2 entry, stride 2
    (2, 5, 16, 16, 32, 32, 1),     # stage 2
    (3, 6, 16, 16, 32, 64, 2),     # stage-3 entry, stride 2
    (2, 6, 8, 8, 64, 64, 1),       # stage 3
    (16, 16, 32, 32, 16, 16, 1),   # many groups, several tiles per CTA
    (16, 4, 32, 32, 3, 16, 1),     # stem with many groups
]


@pytest.mark.parametrize("shape", FORWARD)
def test_conv_forward_matches_fp64(P, shape):
    import torch

    G, B, Hin, Win, Cin, Cout, s = shape
    Hout, Wout = (Hin - 1) // s + 1, (Win - 1) // s + 1
    gen = torch.Generator(device="cuda").manual_seed(sum(shape))
    x = _bf16_randn(torch, (G, B, Hin, Win, Cin), gen)
    w = _bf16_randn(torch, (G, Cout, 3, 3, Cin), gen)
    y = torch.full((G, B, Hout, Wout, Cout), float("nan"), device="cuda")
    P.lsgd_conv3x3_bf16(P.CONV_FORWARD, x, w, y, G, B, Hin, Win, Cin, Cout, s)
    torch.cuda.synchronize()
    want, scale = _forward64(x.double().cpu().numpy(), w.double().cpu().numpy(), s)
    _check(y, want, scale)


DGRAD = [  # (G, B, Hin, Win, Cin, Cout, stride): ResNet-20's input gradients
    (3, 3, 32, 32, 16, 16, 1),     # stage 1
    (2, 5, 32, 32, 16, 32, 2),     # stage-2 entry: four parity phases
    (2, 5, 16, 16, 32, 32, 1),     # stage 2
    (3, 6, 16, 16, 32, 64, 2),     # stage-3 entry: four parity phases
    (2, 6, 8, 8, 64, 64, 1),       # stage 3
    (16, 16, 32, 32, 16, 16, 1),   # many groups, several tiles per CTA
    (16, 8, 32, 32, 16, 32, 2),    # parity phases with many groups
]


@pytest.mark.parametrize("shape", DGRAD)
def test_conv_data_gradient_matches_fp64(P, shape):
    import torch

    G, B, Hin, Win, Cin, Cout, s = shape
    Hout, Wout = (Hin - 1) // s + 1, (Win - 1) // s + 1
    gen = torch.Generator(device="cuda").manual_seed(7 * sum(shape))
    dy = _bf16_randn(torch, (G, B, Hout, Wout, Cout), gen)
    w = _bf16_randn(torch, (G, Cout, 3, 3, Cin), gen)
    dx = torch.full((G, B, Hin, Win, Cin), float("nan"), device="cuda")
    P.lsgd_conv3x3_bf16(P.CONV_DGRAD, dy, w, dx, G, B, Hin, Win, Cin, Cout, s)
    torch.cuda.synchronize()
    want, scale = _dgrad64(dy.double().cpu().numpy(), w.double().cpu().numpy(), s, Hin, Win)
    _check(dx, want, scale)


def test_conv_forward_at_the_full_stage1_size(P):
    # K = 16 replicas x B_loc = 128 images of 32 x 32 x 16 (the configured ResNet-20 step's
    # largest convolution), checked on a sample of images of every replica
    import torch

    G, B, H, C = 16, 128, 32, 16
    gen = torch.Generator(device="cuda").manual_seed(123)
    x = _bf16_randn(torch, (G, B, H, H, C), gen)
    w = _bf16_randn(torch, (G, C, 3, 3, C), gen)
    y = torch.full((G, B, H, H, C), float("nan"), device="cuda")
    P.lsgd_conv3x3_bf16(P.CONV_FORWARD, x, w, y, G, B, H, H, C, C, 1)
    torch.cuda.synchronize()
    pick = [0, 1, 63, 127]
    want, scale = _forward64(x[:, pick].double().cpu().numpy(), w.double().cpu().numpy(), 1)
    _check(y[:, pick], want, scale)


def test_conv_results_are_deterministic(P):
    import torch

    G, B, H, Cin, Cout = 4, 8, 16, 32, 64
    gen = torch.Generator(device="cuda").manual_seed(3)
    dy = _bf16_randn(torch, (G, B, H // 2, H // 2, Cout), gen)
    w = _bf16_randn(torch, (G, Cout, 3, 3, Cin), gen)
    outs = []
    for _ in range(2):
        dx = torch.empty((G, B, H, H, Cin), device="cuda")
        P.lsgd_conv3x3_bf16(P.CONV_DGRAD, dy, w, dx, G, B, H, H, Cin, Cout, 2)
        outs.append(dx.cpu())
    assert torch.equal(outs[0], outs[1])


def test_conv_rejects_shapes_the_kernel_does_not_take(P):
    import torch

    buf = torch.zeros(1 << 20, device="cuda", dtype=torch.bfloat16)
    out = torch.zeros(1 << 20, device="cuda")
    base = dict(G=1, B=2, Hin=8, Win=8, Cin=16, Cout=16, stride=1)
    cases = [(P.CONV_FORWARD, dict(Cin=48), P.EUNSUPPORTED),   # 48 channels per tap
             (P.CONV_FORWARD, dict(Cout=8), P.EUNSUPPORTED),
             (P.CONV_FORWARD, dict(B=1), P.EUNSUPPORTED),      # 64 output pixels: no 128 tile
             (P.CONV_FORWARD, dict(Cin=3, stride=2), P.EUNSUPPORTED),
             (P.CONV_DGRAD, dict(Cin=3), P.EUNSUPPORTED),
             (P.CONV_DGRAD, dict(Hin=9, Win=9, stride=2), P.EUNSUPPORTED),
             (P.CONV_FORWARD, dict(stride=3), P.EINVAL),
             (2, {}, P.EINVAL)]
    for mode, bad, status in cases:
        kw = dict(base)
        kw.update(bad)
        with pytest.raises(P.LsgdError) as e:
            P.lsgd_conv3x3_bf16(mode, buf, buf, out, **kw)
        assert e.value.status == status, (mode, bad, e.value.status)


BN_SHAPES = [  # (G, B, Hin, Win, Cin, Cout, stride): forward convolutions of ResNet-20
    (2, 3, 32, 32, 3, 16, 1),      # stem (padded to 16 channels)
    (3, 3, 32, 32, 16, 16, 1),     # stage 1, one CTA holds several tiles
    (2, 5, 32, 32, 16, 32, 2),     # stage-2 entry
    (3, 6, 16, 16, 32, 64, 2),     # stage-3 entry: 64 channels, four 16-channel chunks
    (2, 6, 8, 8, 64, 64, 1),       # stage 3
    (16, 16, 32, 32, 16, 16, 1),   # many groups
]


@pytest.mark.parametrize("shape", BN_SHAPES)
def test_conv_epilogue_batchnorm_statistics(P, shape):
    # Sec. A.4's per-worker batch statistics of the convolution output, formed by the epilogue
    # (two-pass moments of each warp's 32 rows per tile, combined by Chan et al.'s formula),
    # against fp64 moments of the same fp32 output; the output itself must be the plain
    # forward's, bit for bit
    import torch

    G, B, Hin, Win, Cin, Cout, s = shape
    Hout, Wout = (Hin - 1) // s + 1, (Win - 1) // s + 1
    gen = torch.Generator(device="cuda").manual_seed(11 * sum(shape))
    x = _bf16_randn(torch, (G, B, Hin, Win, Cin), gen)
    # a mean offset per output channel, so that the variance is not the raw second moment
    w = (torch.randn((G, Cout, 3, 3, Cin), device="cuda", generator=gen) +
         0.5 * torch.arange(Cout, device="cuda").view(1, Cout, 1, 1, 1) / Cout).to(torch.bfloat16)
    y = torch.full((G, B, Hout, Wout, Cout), float("nan"), device="cuda")
    y_plain = torch.empty_like(y)
    mean = torch.full((G, Cout), float("nan"), device="cuda")
    rstd = torch.full((G, Cout), float("nan"), device="cuda")
    P.lsgd_conv3x3_bn_bf16(x, w, y, mean, rstd, G, B, Hin, Win, Cin, Cout, s)
    P.lsgd_conv3x3_bf16(P.CONV_FORWARD, x, w, y_plain, G, B, Hin, Win, Cin, Cout, s)
    torch.cuda.synchronize()
    assert torch.equal(y, y_plain)
    y64 = y.double().cpu().numpy().reshape(G, -1, Cout)
    m64 = y64.mean(axis=1)
    v64 = y64.var(axis=1)  # biased, as BatchNorm normalises
    got_m = mean.cpu().numpy().astype(np.float64)
    got_r = rstd.cpu().numpy().astype(np.float64)
    scale = np.sqrt(v64)
    assert np.abs(got_m - m64).max() <= 1e-5 * (np.abs(m64) + scale).max()
    np.testing.assert_allclose(got_r, 1.0 / np.sqrt(v64 + 1e-5), rtol=2e-5)


def test_conv_epilogue_statistics_are_deterministic(P):
    import torch

    G, B, H, C = 4, 16, 32, 16
    gen = torch.Generator(device="cuda").manual_seed(5)
    x = _bf16_randn(torch, (G, B, H, H, C), gen)
    w = _bf16_randn(torch, (G, C, 3, 3, C), gen)
    outs = []
    for _ in range(2):
        y = torch.empty((G, B, H, H, C), device="cuda")
        mean = torch.empty((G, C), device="cuda")
        rstd = torch.empty((G, C), device="cuda")
        P.lsgd_conv3x3_bn_bf16(x, w, y, mean, rstd, G, B, H, H, C, C, 1)
        outs.append((mean.cpu(), rstd.cpu()))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_conv_output_alignment_does_not_change_results(P):
    # an output 16 but not 32 bytes aligned takes the 128-bit store path; same values
    import torch

    G, B, H, Cin, Cout = 2, 4, 32, 16, 32
    gen = torch.Generator(device="cuda").manual_seed(17)
    x = _bf16_randn(torch, (G, B, H, H, Cin), gen)
    w = _bf16_randn(torch, (G, Cout, 3, 3, Cin), gen)
    n = G * B * H * H * Cout
    y = torch.empty((G, B, H, H, Cout), device="cuda")
    buf = torch.full((n + 4,), float("nan"), device="cuda")
    y16 = buf[4:].view(G, B, H, H, Cout)
    assert y16.data_ptr() % 32 == 16
    P.lsgd_conv3x3_bf16(P.CONV_FORWARD, x, w, y, G, B, H, H, Cin, Cout, 1)
    P.lsgd_conv3x3_bf16(P.CONV_FORWARD, x, w, y16, G, B, H, H, Cin, Cout, 1)
    torch.cuda.synchronize()
    assert torch.equal(y, y16)
