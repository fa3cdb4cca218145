"""Pin the oracle's local-step warm-up schedules and its reshuffling sampler.

Local-step warm-up (the "warm-up of the number of local SGD steps" study of Sec. C, and Sec. 4's
ImageNet runs, where the number of local steps doubles each epoch: 1, 2, 4, then H = 8): round-end
steps against hand-derived lists, the constant strategy against post-local SGD with the switch at
the end of the warm-up, a zero-length warm-up against plain local SGD, and sync counts against the
number of rounds.  Reshuffling sampler (Sec. 4 / A.4: the data is disjointly partitioned and
reshuffled globally every epoch): the epoch permutation is a bijection of [0, N) for every N,
position marginals are uniform over many epochs, one epoch whose steps cover the data visits every
point exactly once, and within an epoch the workers' partitions are disjoint."""
import numpy as np
import pytest

import oracle


def _cfg(**kw):
    args = dict(widths=(12, 5), K=4, B=8, H=8, T=60, N=320, base_lr=0.05, seed=41)
    args.update(kw)
    return oracle.make_cfg(**args)


def _round_ends(c):
    return [s for s in range(c.T) if oracle.is_round_end(c, s)]


def _data(N, D, C, seed=0):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((N, D)).astype(np.float32), rng.integers(0, C, N).astype(np.int32)


# ---- local-step warm-up ----

def test_epoch_of_step():
    c = _cfg(K=3, B=7, N=100)  # 21 samples per step: epochs start at steps 0, 5, 10, 15, 20
    assert [oracle.epoch(c, s) for s in range(12)] == [0] * 5 + [1] * 5 + [2] * 2


def test_exponential_warmup_doubles_each_epoch():
    # N / (K B) = 10 steps per epoch; H = 8 over 3 epochs: rounds of 1 in epoch 0, 2 in epoch 1,
    # 4 in epoch 2 (the round starting at step 28 runs to 31), then 8; the last step ends a round.
    c = _cfg(h_warmup=oracle.HWARM_EXPONENTIAL, h_warmup_epochs=3.0)
    want = list(range(10)) + [11, 13, 15, 17, 19] + [23, 27, 31] + [39, 47, 55] + [59]
    assert _round_ends(c) == want
    assert [oracle.round_length(c, s) for s in (0, 10, 20, 28, 32)] == [1, 2, 4, 4, 8]


def test_linear_warmup():
    # H = 4 over P = 4 epochs: lengths 1 + floor(3 e / 4) = 1, 1, 2, 3 in epochs 0..3, then 4.
    c = _cfg(H=4, h_warmup=oracle.HWARM_LINEAR, h_warmup_epochs=4.0)
    want = list(range(20)) + [21, 23, 25, 27, 29] + [32, 35, 38, 41] + [45, 49, 53, 57, 59]
    assert _round_ends(c) == want


def test_constant_warmup_is_post_local_sgd_with_switch_after_warmup():
    # Constant strategy: rounds of 1 while the round starts before epoch P, then rounds of H -- the
    # two phases of post-local SGD with t' = the first step of epoch P (P N / (K B) = 20).
    X, y = _data(320, 12, 5, 3)
    c_w = _cfg(H=4, h_warmup=oracle.HWARM_CONSTANT, h_warmup_epochs=2.0, momentum=0.9,
               nesterov=True)
    c_p = _cfg(H=4, t_switch=20, momentum=0.9, nesterov=True)
    assert _round_ends(c_w) == _round_ends(c_p)
    Ww, Uw, lw, nw = oracle.run(c_w, X, y=y)
    Wp, Up, lp, n_p = oracle.run(c_p, X, y=y)
    assert np.array_equal(Ww, Wp) and np.array_equal(Uw, Up) and np.array_equal(lw, lp)
    assert nw == n_p == 20 + 10


def test_zero_length_warmup_is_local_sgd():
    X, y = _data(320, 12, 5, 4)
    for kind in (oracle.HWARM_LINEAR, oracle.HWARM_EXPONENTIAL, oracle.HWARM_CONSTANT):
        Ww, _, _, nw = oracle.run(_cfg(H=4, h_warmup=kind, h_warmup_epochs=0.0), X, y=y)
        Wl, _, _, nl = oracle.run(_cfg(H=4), X, y=y)
        assert np.array_equal(Ww, Wl) and nw == nl == 15


@pytest.mark.parametrize("kind,P", [(oracle.HWARM_LINEAR, 2.5), (oracle.HWARM_EXPONENTIAL, 1.7),
                                    (oracle.HWARM_CONSTANT, 3.0)])
def test_sync_count_equals_rounds(kind, P):
    X, y = _data(320, 12, 5, 5)
    c = _cfg(H=6, h_warmup=kind, h_warmup_epochs=P, T=47)
    _, _, _, n = oracle.run(c, X, y=y)
    ends = _round_ends(c)
    assert n == len(ends) and ends[-1] == c.T - 1
    # round lengths never exceed H and never decrease while warming up
    lengths = np.diff([-1] + ends[:-1])
    assert lengths.max() <= 6 and np.all(np.diff(lengths) >= 0)


def test_warmup_rejects_switch_and_hierarchy():
    with pytest.raises(ValueError):
        _cfg(h_warmup=oracle.HWARM_LINEAR, h_warmup_epochs=2.0, t_switch=10)
    with pytest.raises(ValueError):
        _cfg(h_warmup=oracle.HWARM_LINEAR, h_warmup_epochs=2.0, hier_block=2, hier_rounds=2)


# ---- reshuffling sampler ----

@pytest.mark.parametrize("N", [1, 2, 3, 5, 16, 17, 64, 1000, 4097])
def test_epoch_permutation_is_a_bijection(N):
    c = _cfg(N=N)
    for e in (0, 7):
        p = [oracle.permute(c, e, i) for i in range(N)]
        assert sorted(p) == list(range(N))


def test_epoch_permutation_marginals_are_uniform():
    # Where element i lands, over 3000 epochs, for each of the first 8 elements of N = 64:
    # chi-square against uniform (63 degrees of freedom; 110 is beyond the 0.9998 quantile).
    c = _cfg(N=64, seed=9)
    E = 3000
    for i in range(8):
        counts = np.bincount([oracle.permute(c, e, i) for e in range(E)], minlength=64)
        exp = E / 64
        chi2 = float(((counts - exp) ** 2 / exp).sum())
        assert chi2 < 110.0, (i, chi2)
    # successive epochs use different permutations
    assert [oracle.permute(c, 0, i) for i in range(64)] != [oracle.permute(c, 1, i) for i in range(64)]


def test_reshuffle_epoch_visits_every_point_once():
    # N = K B m: every epoch is m = 10 whole steps and S = m B, so one epoch's mini-batches of all
    # workers are the dataset, each point once, and worker k's are its partition pi_e[kS, (k+1)S).
    c = _cfg(N=320, sampling=oracle.SAMPLE_RESHUFFLE)
    K, B, S = 4, 8, 80
    for e in range(3):
        seen = []
        for k in range(K):
            mine = np.concatenate([oracle.sample_indices(c, k, s) for s in range(10 * e, 10 * e + 10)])
            part = sorted(oracle.permute(c, e, k * S + q) for q in range(S))
            assert sorted(mine.tolist()) == part
            seen.extend(mine.tolist())
        assert sorted(seen) == list(range(320))


def test_reshuffle_partial_epochs_keep_partitions_disjoint():
    # N = 1000, K = 3, B = 7: 47.6 steps per epoch, S = 333 (one point per epoch unused).  Before a
    # worker wraps around its partition its mini-batches are distinct points of its partition.
    c = _cfg(N=1000, K=3, B=7, sampling=oracle.SAMPLE_RESHUFFLE)
    K, B, S = 3, 7, 333
    for e in (0, 1, 2):
        first = -(-e * 1000 // 21)
        parts = [set(oracle.permute(c, e, k * S + q) for q in range(S)) for k in range(K)]
        assert not (parts[0] & parts[1]) and not (parts[1] & parts[2]) and not (parts[0] & parts[2])
        steps = S // B  # 47 steps without wrapping
        for k in range(K):
            got = np.concatenate([oracle.sample_indices(c, k, first + t) for t in range(steps)])
            assert len(set(got.tolist())) == len(got)
            assert set(got.tolist()) <= parts[k]
    # the epoch's last step (t = 47) wraps around: positions 329..335 mod 333
    e, t = 0, 47
    got = oracle.sample_indices(c, 1, t)
    want = [oracle.permute(c, 0, S + (t * B + j) % S) for j in range(B)]
    assert got.tolist() == want


def test_reshuffle_run_trains():
    X, y = _data(320, 12, 5, 6)
    c = _cfg(H=4, T=40, sampling=oracle.SAMPLE_RESHUFFLE, momentum=0.9)
    _, _, losses, n = oracle.run(c, X, y=y)
    assert n == 10
    assert np.isfinite(losses).all()
