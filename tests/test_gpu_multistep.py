"""Multi-step bf16 parity of the production path (tcgen05 GEMMs and convolutions, fused update,
K-way average) against the oracle on the configured networks: MLP 3072-1024-1024-10 with its
schedule, the sweep network MLP 3072-512-512-10 at K = 8, post-local MLP 3072-4096-4096-4096-100
and post-local ResNet-20, 64 local steps each (Eq. 2; Algorithms 1 and 2).

The oracle's results are stored in tests/golden/multistep_<case>.npz by
tests/golden/make_multistep_goldens.py (the oracle alone; see there for the cases), with and
without the bf16 rounding of the products.  Bar (bf16 mode): relative L2 of the final averaged
parameters <= 2e-2 and the final model's mean loss on the first n_eval rows within 1e-2, the
number of averages equal.  Where the oracle's own bf16 and fp32 runs end further apart than that
(the configured learning rates of the dense networks put them in a chaotic regime: a change of
rounding alone moves the 64-step result by several per cent), the GPU is held to twice that
distance instead (one pair of runs samples the spread a rounding change causes); the "_lr002" cases (learning rate 0.02, the oracle's two runs 0.1-1.3 % apart) must meet
the bar as stated.  The relative L2 is taken over the stored every-`stride`-th parameters (a uniform
subsample of all layers) and the norms over the whole vector."""
import importlib.util
import json
import os

import numpy as np
import pytest

import oracle
import synthdata
from _gpu_common import built_package

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
_spec = importlib.util.spec_from_file_location(
    "make_multistep_goldens", os.path.join(HERE, "golden", "make_multistep_goldens.py"))
goldens = importlib.util.module_from_spec(_spec)
_spec.loader.exec_module(goldens)


@pytest.fixture(scope="module")
def P():
    import torch

    assert torch.cuda.is_available()
    return built_package()


def _gpu_cfg(P, c):
    common = dict(K=c["K"], B_loc=c["B"], H=c["H"], t_switch=c["t_switch"], total_steps=c["T"],
                  N=goldens.N_DATA, base_lr=c["base_lr"], scale_by_K=c["scale_by_K"],
                  warmup_epochs=c["warmup_epochs"], milestones=c["milestones"],
                  momentum=c["momentum"], nesterov=c["nesterov"], weight_decay=c["weight_decay"],
                  seed=c["seed"], precision=P.BF16)
    if c["kind"] == "resnet":
        return P.make_config(kind=P.RESNET20, in_hwc=(32, 32, 3), n_classes=c["C"], base_ch=16,
                             res_blocks=3, **common)
    return P.make_config(widths=c["widths"], fused_update=True, **common)


def _rel(a, b):
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


@pytest.mark.parametrize("name", sorted(goldens.CASES))
def test_multistep_parity_against_oracle(P, name):
    c = goldens.CASES[name]
    gold = {}
    for fp32 in (False, True):
        path = goldens.path_of(name, fp32)
        if not os.path.exists(path):
            pytest.fail(f"{path} missing: run tests/golden/make_multistep_goldens.py")
        gold[fp32] = np.load(path)
        stored = json.loads(str(gold[fp32]["case"]))
        want = json.loads(json.dumps(c))
        stored.pop("bar", None)
        want.pop("bar", None)
        assert stored == want, "golden file is stale"
    g, g32 = gold[False], gold[True]
    X, y = synthdata.gaussian_mixture_cached(goldens.N_DATA, 3072, c["C"], goldens.DATA_SEED)
    o = goldens.oracle_cfg(oracle, c)
    w0 = oracle.init_params(o).astype(np.float32)
    ctx = P.lsgd_create(_gpu_cfg(P, c))
    P.lsgd_set_dataset(ctx, X, y)
    P.lsgd_set_params(ctx, -1, w0)
    P.lsgd_run(ctx, c["T"])
    w = P.lsgd_params(ctx, -1).astype(np.float64)
    ev = P.lsgd_eval_loss(ctx, -1, c["n_eval"])
    lg = P.lsgd_losses(ctx, c["T"], c["K"])
    # the run ends with an average: every replica holds the returned model
    assert np.array_equal(P.lsgd_params(ctx, 0), P.lsgd_params(ctx, c["K"] - 1))
    syncs = P.lsgd_sync_count(ctx)
    P.lsgd_destroy(ctx)

    ref = g["w_sub"].astype(np.float64)
    rel = _rel(w[::c["stride"]], ref)
    sens = _rel(ref, g32["w_sub"].astype(np.float64))  # the oracle's own rounding sensitivity
    ev_sens = abs(float(g["eval_loss"]) - float(g32["eval_loss"]))
    d_ev = abs(ev - float(g["eval_loss"]))
    print(f"{name}: rel L2 {rel:.2e} (oracle bf16 vs fp32 {sens:.2e}), eval loss {ev:.4f} vs "
          f"{float(g['eval_loss']):.4f} (oracle fp32 {float(g32['eval_loss']):.4f})")
    assert syncs == int(g["syncs"]) == int(g32["syncs"])
    assert np.isfinite(lg).all()
    if c["bar"] == "strict":
        # the regime is not chaotic: a change of rounding alone moves the oracle by less than
        # the bar
        assert sens < 2e-2, sens
        assert rel <= 2e-2, rel
        assert d_ev <= 1e-2, d_ev
        # every step's mini-batch losses, against the oracle's own spread between roundings
        # (100-class losses reach ~12 early on, where the two oracle runs differ by up to 0.14)
        loss_sens = float(np.abs(g["losses"] - g32["losses"]).max())
        d_loss = float(np.abs(lg - g["losses"]).max())
        assert d_loss <= max(2e-2, 2 * loss_sens), (d_loss, loss_sens)
    else:
        # one pair of trajectories (oracle bf16 vs fp32) samples how far a change of rounding
        # carries the run; another pair (GPU vs oracle bf16) may land up to about twice as far
        assert rel <= max(2e-2, 2 * sens), (rel, sens)
        assert d_ev <= max(1e-2, 2 * ev_sens), (d_ev, ev_sens)
        # the first steps, before rounding differences have grown
        assert np.abs(lg[:8] - g["losses"][:8]).max() <= 2e-2
    # over the whole vector, the norm of the GPU model matches the oracle's
    assert abs(np.linalg.norm(w) / float(g["norm_full"]) - 1.0) <= max(2e-2, 2 * sens)
