"""Pins for the oracle's Philox4x32-10 and its mini-batch index sampler.

* the published known-answer vectors of the Philox definition (SC'11 / Random123);
* an independent third-party implementation (Triton's `philox`, run by its CPU interpreter);
* the sampler's range (each worker draws only from its own shard, Eq. 1's "locally available
  datapoints") and its uniformity (chi-square over 10^6 draws).
"""
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        v = [int(x, 16) for x in line.split()]
        rows.append((v[0:4], v[4:6], v[6:10]))
    return rows


def test_known_answer_vectors():
    rows = _kat()
    assert len(rows) == 3
    for ctr, key, expect in rows:
        assert oracle.philox4x32_10(ctr, key).tolist() == expect


_TRITON_SCRIPT = textwrap.dedent(
    """
    import os, sys, json
    os.environ["TRITON_INTERPRET"] = "1"
    import torch, triton, triton.language as tl
    from triton.language.random import philox

    @triton.jit
    def k(out_ptr, c_ptr, seed):
        c0 = tl.load(c_ptr + 0); c1 = tl.load(c_ptr + 1); c2 = tl.load(c_ptr + 2); c3 = tl.load(c_ptr + 3)
        r0, r1, r2, r3 = philox(seed, c0, c1, c2, c3)
        tl.store(out_ptr + 0, r0); tl.store(out_ptr + 1, r1); tl.store(out_ptr + 2, r2); tl.store(out_ptr + 3, r3)

    cases = json.loads(sys.stdin.read())
    res = []
    for ctr, key in cases:
        c = torch.tensor([x - (1 << 32) if x >= (1 << 31) else x for x in ctr], dtype=torch.int32)
        out = torch.zeros(4, dtype=torch.int32)
        k[(1,)](out, c, key[0] | (key[1] << 32))
        res.append([x & 0xFFFFFFFF for x in out.tolist()])
    print(json.dumps(res))
    """
)


def test_matches_triton_interpreter():
    pytest.importorskip("triton")
    import json

    rng = np.random.default_rng(5)
    cases = [[[int(v) for v in rng.integers(0, 2**32, 4)], [int(v) for v in rng.integers(0, 2**32, 2)]]
             for _ in range(24)]
    cases += [[[j, s, k, 0], [1234, 0]] for j, s, k in [(0, 0, 0), (7, 3, 2), (31, 1000, 15)]]
    env = dict(os.environ, TRITON_INTERPRET="1", CUDA_VISIBLE_DEVICES="")
    try:
        out = subprocess.run([sys.executable, "-c", _TRITON_SCRIPT], input=json.dumps(cases),
                             capture_output=True, text=True, timeout=600, env=env)
    except subprocess.TimeoutExpired:
        pytest.skip("triton interpreter too slow here")
    if out.returncode != 0:
        pytest.skip("triton interpreter unavailable: " + out.stderr.strip().splitlines()[-1][:200])
    got = json.loads(out.stdout.strip().splitlines()[-1])
    for (ctr, key), ref in zip(cases, got):
        assert oracle.philox4x32_10(ctr, key).tolist() == ref


@pytest.mark.parametrize("N,K,B", [(8192, 4, 32), (50000, 16, 128), (50000, 64, 32), (1000, 3, 5)])
def test_indices_stay_in_own_shard(N, K, B):
    c = oracle.make_cfg(K=K, B=B, N=N, seed=11)
    S = N // K
    for k in [0, K // 2, K - 1]:
        for s in [0, 1, 77]:
            idx = oracle.sample_indices(c, k, s)
            assert idx.shape == (B,)
            assert idx.min() >= k * S and idx.max() < (k + 1) * S


def test_indices_uniform_chi_square():
    # 10^6 draws over a shard of 50 points: chi-square with 49 dof; mean 49, sd ~9.9.
    N, K, B = 200, 4, 1000
    c = oracle.make_cfg(K=K, B=B, N=N, seed=3)
    counts = np.zeros(N // K)
    for s in range(250):
        for k in range(K):
            idx = oracle.sample_indices(c, k, s) - k * (N // K)
            counts += np.bincount(idx, minlength=N // K)
    n = counts.sum()
    assert n == 10**6
    e = n / len(counts)
    chi2 = float(((counts - e) ** 2 / e).sum())
    assert chi2 < 49 + 6 * 9.9


def test_indices_depend_on_worker_step_seed():
    c = oracle.make_cfg(K=2, B=64, N=1 << 20, seed=1)
    a = oracle.sample_indices(c, 0, 0)
    assert not np.array_equal(a - 0, oracle.sample_indices(c, 1, 0) - (1 << 19))
    assert not np.array_equal(a, oracle.sample_indices(c, 0, 1))
    c2 = oracle.make_cfg(K=2, B=64, N=1 << 20, seed=2)
    assert not np.array_equal(a, oracle.sample_indices(c2, 0, 0))
    assert np.array_equal(a, oracle.sample_indices(c, 0, 0))
