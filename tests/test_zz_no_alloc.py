"""lsgd_batchnorm_stats_noalloc, the BatchNorm-statistics entry point for callers that cannot let
the library allocate device memory (their memory is all in their own pool, or fixed at start-up),
against the allocating lsgd_batchnorm_stats on two calls in a row.  Kept in a file collected last:
it exercises the library's fixed device-resident scratch array."""
import numpy as np
import pytest

from _gpu_common import built_package

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


def test_noalloc_matches_allocating_entry_point_twice(P):
    import torch

    # two different problems back to back: the shared scratch must give the same results as the
    # per-call allocation both times (same tolerance as the allocating entry point's test)
    for G, n, C, seed in [(16, 131072, 16, 1), (3, 5000, 64, 2)]:
        gen = torch.Generator(device="cuda").manual_seed(seed)
        y = torch.randn((G, n, C), device="cuda", generator=gen) * 3.0 - 1.0
        m_ref = torch.empty((G, C), device="cuda")
        r_ref = torch.empty((G, C), device="cuda")
        m_new = torch.full((G, C), float("nan"), device="cuda")
        r_new = torch.full((G, C), float("nan"), device="cuda")
        P.lsgd_batchnorm_stats(y, n, C, G, m_ref, r_ref)
        P.lsgd_batchnorm_stats_noalloc(y, n, C, G, m_new, r_new)
        torch.cuda.synchronize()
        np.testing.assert_allclose(m_new.cpu().numpy(), m_ref.cpu().numpy(), rtol=1e-5, atol=1e-5)
        np.testing.assert_allclose(r_new.cpu().numpy(), r_ref.cpu().numpy(), rtol=1e-4)


def test_noalloc_rejects_sizes_beyond_its_scratch(P):
    import torch

    G, C = 64, 64
    # exactly at the limit: 64 replicas x 128 chunks x 64 channels x 2 = 2^20 partial values
    n_fit = 128 * 1024
    y = torch.zeros((G, n_fit, C), device="cuda")
    m = torch.empty((G, C), device="cuda")
    r = torch.empty((G, C), device="cuda")
    P.lsgd_batchnorm_stats_noalloc(y, n_fit, C, G, m, r)
    torch.cuda.synchronize()
    assert torch.all(m == 0)
    del y
    # one chunk more (64 x 129 x 64 x 2 > 2^20) is refused before any launch; the input tensor
    # still has all n_big rows, so no read could leave it even if it were not refused
    n_big = 129 * 1024
    assert G * ((n_big + 1023) // 1024) * C * 2 > 1 << 20
    y = torch.zeros((G, n_big, C), device="cuda")
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_batchnorm_stats_noalloc(y, n_big, C, G, m, r)
    assert e.value.status == P.EINVAL
    assert "exceed" in P.lsgd_last_error()
    torch.cuda.synchronize()
