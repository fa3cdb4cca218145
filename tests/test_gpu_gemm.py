"""The grouped bf16 GEMM kernels (tcgen05 / TMEM / TMA and SIMT) against an fp64 product of the same
bf16 operands, for every operand layout the dense layers use, on ragged shapes spanning several
tiles.  Error measure: |C - C64| / (|A| |B|^T) elementwise (the fp32 accumulation error bound
scale), which must stay at fp32 level (~1e-6)."""
import numpy as np
import pytest

from _gpu_common import built_package

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


SHAPES = [(128, 128, 64, 1), (128, 1024, 3072, 2), (1024, 3072, 128, 2), (40, 136, 264, 3),
          (128, 10, 1024, 2), (128, 1024, 16, 2), (10, 1024, 128, 2), (100, 256, 128, 1),
          (128, 64, 72, 2), (200, 136, 2104, 2)]


def _operands(torch, M, N, Kd, G, a_mn, b_mn, seed):
    gen = torch.Generator(device="cuda").manual_seed(seed)
    A = torch.randn((G, M, Kd), device="cuda", generator=gen).to(torch.bfloat16)
    B = torch.randn((G, N, Kd), device="cuda", generator=gen).to(torch.bfloat16)
    A_st = A.transpose(1, 2).contiguous() if a_mn else A.contiguous()
    B_st = B.transpose(1, 2).contiguous() if b_mn else B.contiguous()
    return A, B, A_st, B_st


@pytest.mark.parametrize("a_mn,b_mn", [(False, False), (False, True), (True, True), (True, False)])
@pytest.mark.parametrize("shape", SHAPES)
def test_grouped_gemm_matches_fp64(P, shape, a_mn, b_mn):
    import torch

    M, N, Kd, G = shape
    if (a_mn and M % 8) or (b_mn and N % 8) or (not a_mn and Kd % 8) or (not b_mn and Kd % 8):
        pytest.skip("contiguous extent must be a multiple of 8")
    A, B, A_st, B_st = _operands(torch, M, N, Kd, G, a_mn, b_mn, M * 7 + N * 3 + Kd)
    ref = torch.matmul(A.double(), B.double().transpose(1, 2))
    scale = torch.matmul(A.double().abs(), B.double().abs().transpose(1, 2))
    for engine in (0, 1):
        C = torch.full((G, M, N), float("nan"), device="cuda", dtype=torch.float32)
        P.lsgd_grouped_gemm_bf16(A_st, a_mn, B_st, b_mn, C, M, N, Kd, G, engine=engine)
        torch.cuda.synchronize()
        assert not torch.isnan(C).any(), engine
        err = ((C.double() - ref).abs() / scale.clamp_min(1e-30)).max().item()
        print(f"engine {engine} {shape} a_mn={a_mn} b_mn={b_mn}: max err / (|A||B|) = {err:.2e}")
        assert err <= 4e-6, (engine, err)


def test_persistent_and_one_tile_kernels_agree_bitwise():
    # Wide products (K-major or MN-major B, at least 2048 columns) run on the persistent
    # 128 x 256-tile kernel; the one-tile kernel
    # (LSGD_GEMM_ONE_TILE=1 at library load) accumulates every output in the same k order, so
    # both give the same bits.  Run in subprocesses: the switch is read once.
    import os
    import subprocess
    import sys
    prog = r"""
import numpy as np, torch, sys
sys.path.insert(0, %r)
from _gpu_common import built_package
P = built_package()
gen = torch.Generator(device="cuda").manual_seed(5)
out = []
for (M, N, Kd, G, a_mn, b_mn) in [(128, 4096, 4096, 3, 0, 0), (128, 1024, 3072, 2, 0, 1),
                                  (200, 520, 1000, 2, 0, 0), (128, 264, 136, 4, 0, 1),
                                  (128, 4096, 4096, 2, 0, 1), (96, 2048, 520, 3, 0, 1),
                                  (128, 2600, 1000, 2, 0, 1)]:
    A = torch.randn((G, Kd, M) if a_mn else (G, M, Kd), device="cuda", generator=gen).to(torch.bfloat16)
    B = torch.randn((G, Kd, N) if b_mn else (G, N, Kd), device="cuda", generator=gen).to(torch.bfloat16)
    C = torch.empty((G, M, N), device="cuda")
    P.lsgd_grouped_gemm_bf16(A, a_mn, B, b_mn, C, M, N, Kd, G, 0)
    torch.cuda.synchronize()
    out.append(C.cpu().numpy())
np.save(sys.argv[1], np.concatenate([o.ravel() for o in out]))
""" % os.path.dirname(os.path.abspath(__file__))
    import tempfile
    res = []
    with tempfile.TemporaryDirectory() as d:
        for one in ("0", "1"):
            path = os.path.join(d, f"c{one}.npy")
            env = dict(os.environ, LSGD_GEMM_ONE_TILE=one)
            r = subprocess.run([sys.executable, "-c", prog, path], env=env, capture_output=True,
                               text=True, timeout=600)
            assert r.returncode == 0, r.stderr[-2000:]
            res.append(np.load(path))
    assert np.array_equal(res[0], res[1])
