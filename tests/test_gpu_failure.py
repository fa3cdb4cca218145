"""Failure detection of the device-side waits, exercised without faulting the GPU: a bounded
mbarrier wait that nothing completes runs out after its limit, the host reads LSGD_ETIMEOUT, the
device flag is consumed, and the same context keeps training afterwards."""
import time

import numpy as np
import pytest

import synthdata
from _gpu_common import built_package, dense_cfgs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


def test_bounded_wait_completes_when_the_phase_arrives(P):
    t0 = time.perf_counter()
    assert P.lsgd_bounded_wait_selftest(True, 200.0) == P.OK
    assert time.perf_counter() - t0 < 0.5
    assert P.lsgd_device_status(None) == P.OK


def test_bounded_wait_runs_out_and_the_context_stays_usable(P):
    import torch

    widths = (128, 64, 10)
    g, _ = dense_cfgs(P, widths=widths, K=4, B=16, H=3, T=12, N=512, precision=P.BF16,
                      base_lr=0.05, momentum=0.9, seed=3, fused_update=True)
    X, y = synthdata.gaussian_mixture(512, widths[0], widths[-1], seed=1)
    ctx = P.lsgd_create(g)
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_run(ctx, 5)
    assert P.lsgd_device_status(ctx) == P.OK
    t0 = time.perf_counter()
    assert P.lsgd_bounded_wait_selftest(False, 50.0) == P.ETIMEOUT
    dt = time.perf_counter() - t0
    assert 0.04 <= dt < 1.5, dt
    assert P.lsgd_device_status(ctx) == P.OK  # the self-test consumed the flag
    P.lsgd_run(ctx, 7)
    P.lsgd_check_finite(ctx)
    assert P.lsgd_sync_count(ctx) == 4
    assert np.isfinite(P.lsgd_params(ctx, 0)).all()
    assert float(torch.ones(8, device="cuda").sum()) == 8.0
    P.lsgd_destroy(ctx)


def test_bounded_wait_limits_are_checked(P):
    assert P.lsgd_bounded_wait_selftest(False, 5000.0) == P.EINVAL
    assert P.lsgd_bounded_wait_selftest(False, -1.0) == P.EINVAL
