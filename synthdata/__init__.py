"""Seeded synthetic inputs shared by the CUDA path's tests/benchmark and the oracle's tests.

This module only draws input data.  It holds none of the method's arithmetic and imports neither
the oracle nor the CUDA package.  The generators are counter-based (SplitMix64 of Steele, Lea and
Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014, applied to a stream key plus
the element index) with Box-Muller normals in fp64, so every platform produces the same bits.

Workload shapes stand in for the paper's CIFAR-10/100 (Sec. A.1: 50 K training images of
32 x 32 x 3, 10 or 100 classes): a Gaussian mixture with class means 4 * N(0, I/d), isotropic unit
noise and uniform labels.  Rows are stored HWC (channel fastest), fp32.  Data depend only on
(seed, N, D, C) for a given NumPy bit-generator stream, never on the code under test.
"""
from __future__ import annotations

import functools

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)

STREAM_LABELS, STREAM_MEANS, STREAM_NOISE, STREAM_LSQ_A, STREAM_LSQ_W = 1, 2, 3, 4, 5


def _splitmix64(x: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = x + _GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        return z ^ (z >> np.uint64(31))


def _key(seed: int, stream: int) -> np.uint64:
    with np.errstate(over="ignore"):
        k = _splitmix64(np.array([seed & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64))[0]
        return _splitmix64(np.array([k ^ np.uint64(stream * 0x1000003)], dtype=np.uint64))[0]


def uniform(seed: int, stream: int, start: int, count: int) -> np.ndarray:
    """Uniform doubles in (0, 1) for elements start .. start+count-1 of a stream."""
    i = np.arange(start, start + count, dtype=np.uint64)
    with np.errstate(over="ignore"):
        h = _splitmix64(i * _GOLDEN + _key(seed, stream))
    return ((h >> np.uint64(11)).astype(np.float64) + 0.5) * (1.0 / 9007199254740992.0)


def normal(seed: int, stream: int, start: int, count: int) -> np.ndarray:
    """Standard normals for elements start .. start+count-1 (Box-Muller on element pairs)."""
    p0 = start // 2
    p1 = (start + count + 1) // 2
    u1 = uniform(seed, stream, 2 * p0, 2 * (p1 - p0))
    a, b = u1[0::2], u1[1::2]
    r = np.sqrt(-2.0 * np.log(a))
    z = np.empty(2 * (p1 - p0), dtype=np.float64)
    z[0::2] = r * np.cos(2.0 * np.pi * b)
    z[1::2] = r * np.sin(2.0 * np.pi * b)
    off = start - 2 * p0
    return z[off:off + count]


def gaussian_mixture(N: int, D: int = 3072, C: int = 10, seed: int = 1234, mean_scale: float = 4.0,
                     sigma: float = 1.0):
    """X [N, D] fp32 and y [N] int32: y uniform over C classes, x = mean_scale * z_y + sigma * eps
    with z_c ~ N(0, I / D) and eps ~ N(0, I)."""
    y = np.minimum((uniform(seed, STREAM_LABELS, 0, N) * C).astype(np.int64), C - 1).astype(np.int32)
    means = normal(seed, STREAM_MEANS, 0, C * D).reshape(C, D) * (mean_scale / np.sqrt(D))
    # The bulk noise uses NumPy's SFC64 bit generator (a stable bit stream) for speed.
    gen = np.random.Generator(np.random.SFC64(int(_key(seed, STREAM_NOISE))))
    X = np.empty((N, D), dtype=np.float32)
    rows = max(1, (1 << 22) // D)
    means32 = means.astype(np.float32)
    for r0 in range(0, N, rows):
        r1 = min(N, r0 + rows)
        eps = gen.standard_normal((r1 - r0, D), dtype=np.float32)
        if sigma != 1.0:
            eps *= np.float32(sigma)
        eps += means32[y[r0:r1]]
        X[r0:r1] = eps
    return X, y


@functools.lru_cache(maxsize=4)
def gaussian_mixture_cached(N: int, D: int = 3072, C: int = 10, seed: int = 1234):
    X, y = gaussian_mixture(N, D, C, seed)
    X.setflags(write=False)
    y.setflags(write=False)
    return X, y


def least_squares(N: int, d: int, seed: int = 7):
    """A [N, d] fp32 with N(0, 1) entries, w_star [d] fp64 and consistent targets t = A w_star
    (computed in fp64 from the fp32 A, then stored fp32)."""
    A = normal(seed, STREAM_LSQ_A, 0, N * d).reshape(N, d).astype(np.float32)
    w_star = normal(seed, STREAM_LSQ_W, 0, d)
    t = (A.astype(np.float64) @ w_star).astype(np.float32)
    return A, t, w_star
