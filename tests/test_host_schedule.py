"""The library's host-side schedule logic (no GPU): lsgd_schedule's learning rate and sync kind
for every step against the oracle's, over post-local, hierarchical and local-step warm-up
configurations with ragged epochs, plus the configuration checks lsgd_create applies."""
import numpy as np
import pytest

import oracle
from _gpu_common import dense_cfgs


@pytest.fixture(scope="module")
def P():
    from paper_1808_07217_gb300 import _build

    _build.build()
    import paper_1808_07217_gb300 as P

    P.lib()
    return P


CASES = [
    dict(K=16, B=128, H=16, T=49, N=50000, base_lr=0.1, scale_by_K=True, warmup_epochs=5.0),
    dict(K=16, B=128, H=16, T=245, N=50000, t_switch=122, base_lr=0.1, scale_by_K=True,
         warmup_epochs=5.0, milestones=(0.5, 0.75)),
    dict(K=8, B=32, H=4, T=500, N=50000, base_lr=0.1),
    dict(K=6, B=10, H=3, T=200, N=1000, hier_block=2, hier_rounds=4, milestones=(0.3,)),
    dict(K=6, B=10, H=3, T=200, N=1000, t_switch=37, hier_block=3, hier_rounds=2),
    dict(K=4, B=8, H=8, T=300, N=1000, h_warmup=1, h_warmup_epochs=3.5),
    dict(K=4, B=8, H=16, T=300, N=1000, h_warmup=2, h_warmup_epochs=4.0),
    dict(K=4, B=8, H=12, T=300, N=999, h_warmup=2, h_warmup_epochs=2.3),
    dict(K=3, B=7, H=5, T=250, N=1000, h_warmup=3, h_warmup_epochs=1.5, scale_by_K=True,
         warmup_epochs=2.0, milestones=(0.5, 0.75)),
]


@pytest.mark.parametrize("case", CASES)
def test_schedule_matches_oracle(P, case):
    g, o = dense_cfgs(P, widths=(16, 4), precision=P.FP32, **case)
    T = case["T"]
    lr, kinds = P.lsgd_schedule(g, T)
    want_lr = np.array([oracle.lr(o, s) for s in range(T)])
    want_kind = np.array([oracle.sync_kind(o, s) for s in range(T)])
    np.testing.assert_allclose(lr, want_lr, rtol=1e-15, atol=0)
    assert np.array_equal(kinds, want_kind)
    assert kinds[-1] == 2


def test_schedule_rejects_bad_configs(P):
    bad = [dict(h_warmup=1, h_warmup_epochs=2.0, t_switch=5),
           dict(h_warmup=1, h_warmup_epochs=2.0, hier_block=2, hier_rounds=2),
           dict(h_warmup=4), dict(h_warmup=1, h_warmup_epochs=-1.0), dict(sampling=2),
           dict(compress=1, global_momentum=0.5), dict(hier_block=3)]
    for kw in bad:
        g = P.make_config(K=4, B_loc=8, H=4, total_steps=10, N=100, widths=(16, 4), **kw)
        with pytest.raises(RuntimeError):
            P.lsgd_schedule(g, 10)
