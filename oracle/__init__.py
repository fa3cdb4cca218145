"""Oracle for the local / post-local SGD hot path -- TEST INFRASTRUCTURE ONLY.

A plain, slow, single-threaded C++ restatement (fp64) of the method of "Don't Use Large
Mini-Batches, Use Local SGD": mini-batch SGD (Eq. 1), local SGD (Eq. 2, Algorithm 1), post-local
SGD (Sec. 3, Algorithm 2), local Nesterov momentum and weight decay (Sec. C.3.1, A.4) and the
learning-rate schemes (Sec. A.3, A.4).  This module only marshals numpy arrays into the C library
built from ``oracle/*.cpp``.

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg may import this
package.  It shares no code with the CUDA path and imports nothing from it.

Parity pins: every function here is checked by ``tests/test_oracle_*.py`` against closed forms,
special cases and published values (Philox known-answer vectors, finite differences, the paper's
mini-batch special cases, the least-squares optimum, the momentum expansion of Sec. C.3.1).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_SOURCES = ["oracle.cpp", "resnet.cpp"]
_lock = threading.Lock()
_lib = None

DENSE, LSQ, RESNET20 = 0, 1, 2
COMPRESS_NONE, COMPRESS_SIGN, COMPRESS_EF_SIGN = 0, 1, 2
HWARM_NONE, HWARM_LINEAR, HWARM_EXPONENTIAL, HWARM_CONSTANT = 0, 1, 2, 3
SAMPLE_SHARDS, SAMPLE_RESHUFFLE = 0, 1
INIT_ZERO, INIT_HE = 0, 1
MAX_LAYERS = 8


class Cfg(ctypes.Structure):
    _fields_ = [
        ("kind", ctypes.c_int),
        ("n_layers", ctypes.c_int),
        ("widths", ctypes.c_int * (MAX_LAYERS + 1)),
        ("has_bias", ctypes.c_int),
        ("bf16", ctypes.c_int),
        ("K", ctypes.c_int),
        ("B", ctypes.c_int),
        ("H", ctypes.c_int),
        ("t_switch", ctypes.c_int64),
        ("T", ctypes.c_int64),
        ("N", ctypes.c_int64),
        ("base_lr", ctypes.c_double),
        ("scale_by_K", ctypes.c_int),
        ("warmup_epochs", ctypes.c_double),
        ("n_milestones", ctypes.c_int),
        ("milestones", ctypes.c_double * 4),
        ("decay", ctypes.c_double),
        ("momentum", ctypes.c_double),
        ("nesterov", ctypes.c_int),
        ("weight_decay", ctypes.c_double),
        ("seed", ctypes.c_uint64),
        ("in_h", ctypes.c_int),
        ("in_w", ctypes.c_int),
        ("in_c", ctypes.c_int),
        ("n_classes", ctypes.c_int),
        ("base_ch", ctypes.c_int),
        ("res_blocks", ctypes.c_int),
        ("hier_block", ctypes.c_int),
        ("hier_rounds", ctypes.c_int),
        ("compress", ctypes.c_int),
        ("global_momentum", ctypes.c_double),
        ("h_warmup", ctypes.c_int),
        ("h_warmup_epochs", ctypes.c_double),
        ("sampling", ctypes.c_int),
    ]


def make_cfg(kind=DENSE, widths=(3072, 10), has_bias=True, bf16=False, K=1, B=1, H=1,
             t_switch=-1, T=1, N=1, base_lr=0.1, scale_by_K=False, warmup_epochs=0.0,
             milestones=(), decay=0.1, momentum=0.0, nesterov=False, weight_decay=0.0, seed=0,
             in_hwc=(32, 32, 3), n_classes=10, base_ch=16, res_blocks=3, hier_block=0,
             hier_rounds=1, compress=0, global_momentum=0.0, h_warmup=HWARM_NONE,
             h_warmup_epochs=0.0, sampling=SAMPLE_SHARDS) -> Cfg:
    if h_warmup != HWARM_NONE and (hier_block > 0 or t_switch >= 0):
        raise ValueError("local-step warm-up replaces the post-local switch and is not combined "
                         "with hierarchical averaging")
    c = Cfg()
    c.kind = kind
    if kind != RESNET20:
        c.n_layers = len(widths) - 1
        for i, w in enumerate(widths):
            c.widths[i] = int(w)
    c.has_bias = int(bool(has_bias))
    c.bf16 = int(bool(bf16))
    c.K, c.B, c.H = int(K), int(B), int(H)
    c.t_switch, c.T, c.N = int(t_switch), int(T), int(N)
    c.base_lr = float(base_lr)
    c.scale_by_K = int(bool(scale_by_K))
    c.warmup_epochs = float(warmup_epochs)
    c.n_milestones = len(milestones)
    for i, m in enumerate(milestones):
        c.milestones[i] = float(m)
    c.decay = float(decay)
    c.momentum = float(momentum)
    c.nesterov = int(bool(nesterov))
    c.weight_decay = float(weight_decay)
    c.seed = int(seed)
    c.in_h, c.in_w, c.in_c = (int(v) for v in in_hwc)
    c.n_classes = int(n_classes)
    c.base_ch = int(base_ch)
    c.res_blocks = int(res_blocks)
    c.hier_block = int(hier_block)
    c.hier_rounds = int(hier_rounds)
    c.compress = int(compress)
    c.global_momentum = float(global_momentum)
    c.h_warmup = int(h_warmup)
    c.h_warmup_epochs = float(h_warmup_epochs)
    c.sampling = int(sampling)
    return c


def build(force: bool = False) -> str:
    """Compile liboracle.so with g++ (-O2, single-threaded, no SIMD intrinsics)."""
    srcs = [os.path.join(_HERE, s) for s in _SOURCES]
    hdrs = [os.path.join(_HERE, h) for h in ("oracle.h", "philox.h")]
    newest = max(os.path.getmtime(p) for p in srcs + hdrs)
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= newest:
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-o", tmp] + srcs
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB_PATH)
            P = ctypes.POINTER
            cfgp = P(Cfg)
            dp = P(ctypes.c_double)
            fp = P(ctypes.c_float)
            ip = P(ctypes.c_int32)
            L.oracle_num_params.argtypes = [cfgp]
            L.oracle_num_params.restype = ctypes.c_int64
            L.oracle_weight_decay_mask.argtypes = [cfgp, P(ctypes.c_uint8)]
            L.oracle_philox4x32_10.argtypes = [P(ctypes.c_uint32), P(ctypes.c_uint32), P(ctypes.c_uint32)]
            L.oracle_sample_indices.argtypes = [cfgp, ctypes.c_int, ctypes.c_int64, ip]
            L.oracle_init_params.argtypes = [cfgp, ctypes.c_int, dp]
            L.oracle_loss_grad.argtypes = [cfgp, dp, fp, ip, fp, ip, ctypes.c_int, dp]
            L.oracle_loss_grad.restype = ctypes.c_double
            L.oracle_sgd_update.argtypes = [cfgp, ctypes.c_double, dp, dp, dp]
            L.oracle_lr.argtypes = [cfgp, ctypes.c_int64]
            L.oracle_lr.restype = ctypes.c_double
            L.oracle_is_round_end.argtypes = [cfgp, ctypes.c_int64]
            L.oracle_is_round_end.restype = ctypes.c_int
            L.oracle_average.argtypes = [ctypes.c_int, ctypes.c_int64, dp]
            L.oracle_block_average.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int64, dp]
            L.oracle_sync_kind.argtypes = [cfgp, ctypes.c_int64]
            L.oracle_sync_kind.restype = ctypes.c_int
            L.oracle_epoch.argtypes = [cfgp, ctypes.c_int64]
            L.oracle_epoch.restype = ctypes.c_int64
            L.oracle_round_length.argtypes = [cfgp, ctypes.c_int64]
            L.oracle_round_length.restype = ctypes.c_int64
            L.oracle_permute.argtypes = [cfgp, ctypes.c_int64, ctypes.c_int64]
            L.oracle_permute.restype = ctypes.c_int64
            L.oracle_run_counted.argtypes = [cfgp, fp, ip, fp, dp, dp, ctypes.c_int64,
                                             ctypes.c_int64, dp, P(ctypes.c_int64),
                                             P(ctypes.c_int64)]
            L.oracle_run.argtypes = [cfgp, fp, ip, fp, dp, dp, ctypes.c_int64, ctypes.c_int64, dp,
                                     P(ctypes.c_int64)]
            L.oracle_run_ext.argtypes = [cfgp, fp, ip, fp, dp, dp, dp, dp, dp, ctypes.c_int64,
                                         ctypes.c_int64, dp, P(ctypes.c_int64), P(ctypes.c_int64)]
            L.oracle_run_minibatch.argtypes = [cfgp, fp, ip, fp, dp, dp, ctypes.c_int64,
                                               ctypes.c_int64, dp]
            L.oracle_eval_loss.argtypes = [cfgp, dp, fp, ip, fp, ctypes.c_int64]
            L.oracle_eval_loss.restype = ctypes.c_double
            L.oracle_bf16_round.argtypes = [ctypes.c_double]
            L.oracle_bf16_round.restype = ctypes.c_double
            _lib = L
    return _lib


def _p(a, ct):
    if a is None:
        return None
    return a.ctypes.data_as(ctypes.POINTER(ct))


def _f32(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.float32)


def _i32(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.int32)


def num_params(c: Cfg) -> int:
    return int(lib().oracle_num_params(ctypes.byref(c)))


def weight_decay_mask(c: Cfg) -> np.ndarray:
    m = np.zeros(num_params(c), dtype=np.uint8)
    lib().oracle_weight_decay_mask(ctypes.byref(c), _p(m, ctypes.c_uint8))
    return m


def philox4x32_10(ctr, key) -> np.ndarray:
    c = np.asarray(ctr, dtype=np.uint32)
    k = np.asarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().oracle_philox4x32_10(_p(c, ctypes.c_uint32), _p(k, ctypes.c_uint32), _p(out, ctypes.c_uint32))
    return out


def sample_indices(c: Cfg, k: int, s: int) -> np.ndarray:
    out = np.zeros(c.B, dtype=np.int32)
    lib().oracle_sample_indices(ctypes.byref(c), int(k), int(s), _p(out, ctypes.c_int32))
    return out


def init_params(c: Cfg, init_kind: int = INIT_HE) -> np.ndarray:
    w = np.zeros(num_params(c), dtype=np.float64)
    lib().oracle_init_params(ctypes.byref(c), int(init_kind), _p(w, ctypes.c_double))
    return w


def loss_grad(c: Cfg, w, X, y=None, t=None, idx=None):
    w = np.ascontiguousarray(w, dtype=np.float64)
    X, y, t, idx = _f32(X), _i32(y), _f32(t), _i32(idx)
    g = np.zeros_like(w)
    loss = lib().oracle_loss_grad(ctypes.byref(c), _p(w, ctypes.c_double), _p(X, ctypes.c_float),
                                  _p(y, ctypes.c_int32), _p(t, ctypes.c_float),
                                  _p(idx, ctypes.c_int32), int(len(idx)), _p(g, ctypes.c_double))
    return float(loss), g


def sgd_update(c: Cfg, lr: float, w, u, g):
    w = np.array(w, dtype=np.float64)
    u = np.array(u, dtype=np.float64)
    g = np.ascontiguousarray(g, dtype=np.float64)
    lib().oracle_sgd_update(ctypes.byref(c), float(lr), _p(w, ctypes.c_double),
                            _p(u, ctypes.c_double), _p(g, ctypes.c_double))
    return w, u


def lr(c: Cfg, s: int) -> float:
    return float(lib().oracle_lr(ctypes.byref(c), int(s)))


def epoch(c: Cfg, s: int) -> int:
    return int(lib().oracle_epoch(ctypes.byref(c), int(s)))


def round_length(c: Cfg, s0: int) -> int:
    return int(lib().oracle_round_length(ctypes.byref(c), int(s0)))


def permute(c: Cfg, e: int, i: int) -> int:
    return int(lib().oracle_permute(ctypes.byref(c), int(e), int(i)))


def is_round_end(c: Cfg, s: int) -> bool:
    return bool(lib().oracle_is_round_end(ctypes.byref(c), int(s)))


def average(W) -> np.ndarray:
    W = np.array(W, dtype=np.float64)
    K, d = W.shape
    lib().oracle_average(int(K), int(d), _p(W, ctypes.c_double))
    return W


def sync_kind(c: Cfg, s: int) -> int:
    """0 = no average after step s, 1 = block average, 2 = global average."""
    return int(lib().oracle_sync_kind(ctypes.byref(c), int(s)))


def block_average(W, block: int) -> np.ndarray:
    W = np.array(W, dtype=np.float64)
    K, d = W.shape
    lib().oracle_block_average(int(K), int(block), int(d), _p(W, ctypes.c_double))
    return W


def run_counted(c: Cfg, X, y=None, t=None, W=None, U=None, s0=0, n_steps=None):
    """run() that also returns the number of block averages: W, U, losses, n_global, n_block."""
    d = num_params(c)
    if W is None:
        W = np.tile(init_params(c), (c.K, 1))
    W = np.array(W, dtype=np.float64).reshape(c.K, d)
    U = np.zeros_like(W) if U is None else np.array(U, dtype=np.float64).reshape(c.K, d)
    n = int(c.T - s0 if n_steps is None else n_steps)
    losses = np.zeros((n, c.K), dtype=np.float64)
    ng, nb = ctypes.c_int64(0), ctypes.c_int64(0)
    X, y, t = _f32(X), _i32(y), _f32(t)
    lib().oracle_run_counted(ctypes.byref(c), _p(X, ctypes.c_float), _p(y, ctypes.c_int32),
                             _p(t, ctypes.c_float), _p(W, ctypes.c_double), _p(U, ctypes.c_double),
                             int(s0), n, _p(losses, ctypes.c_double), ctypes.byref(ng),
                             ctypes.byref(nb))
    return W, U, losses, int(ng.value), int(nb.value)


def run_ext(c: Cfg, X, y=None, t=None, W=None, U=None, Wref=None, E=None, Ug=None, s0=0,
            n_steps=None):
    """Run with the synchronisation state of the compressed / global-momentum variants.
    Returns W, U, Wref, E, Ug, losses, n_global, n_block."""
    d = num_params(c)
    if W is None:
        W = np.tile(init_params(c), (c.K, 1))
    W = np.array(W, dtype=np.float64).reshape(c.K, d)
    U = np.zeros_like(W) if U is None else np.array(U, dtype=np.float64).reshape(c.K, d)
    Wref = W[0].copy() if Wref is None else np.array(Wref, dtype=np.float64).reshape(d)
    E = np.zeros_like(W) if E is None else np.array(E, dtype=np.float64).reshape(c.K, d)
    Ug = np.zeros(d) if Ug is None else np.array(Ug, dtype=np.float64).reshape(d)
    n = int(c.T - s0 if n_steps is None else n_steps)
    losses = np.zeros((n, c.K), dtype=np.float64)
    ng, nb = ctypes.c_int64(0), ctypes.c_int64(0)
    X, y, t = _f32(X), _i32(y), _f32(t)
    lib().oracle_run_ext(ctypes.byref(c), _p(X, ctypes.c_float), _p(y, ctypes.c_int32),
                         _p(t, ctypes.c_float), _p(W, ctypes.c_double), _p(U, ctypes.c_double),
                         _p(Wref, ctypes.c_double), _p(E, ctypes.c_double), _p(Ug, ctypes.c_double),
                         int(s0), n, _p(losses, ctypes.c_double), ctypes.byref(ng), ctypes.byref(nb))
    return W, U, Wref, E, Ug, losses, int(ng.value), int(nb.value)


def run(c: Cfg, X, y=None, t=None, W=None, U=None, s0=0, n_steps=None):
    """Local / post-local SGD; W, U are [K, d] (defaults: He init broadcast, zero momentum)."""
    d = num_params(c)
    if W is None:
        W = np.tile(init_params(c), (c.K, 1))
    W = np.array(W, dtype=np.float64).reshape(c.K, d)
    U = np.zeros_like(W) if U is None else np.array(U, dtype=np.float64).reshape(c.K, d)
    n = int(c.T - s0 if n_steps is None else n_steps)
    losses = np.zeros((n, c.K), dtype=np.float64)
    syncs = ctypes.c_int64(0)
    X, y, t = _f32(X), _i32(y), _f32(t)
    lib().oracle_run(ctypes.byref(c), _p(X, ctypes.c_float), _p(y, ctypes.c_int32),
                     _p(t, ctypes.c_float), _p(W, ctypes.c_double), _p(U, ctypes.c_double),
                     int(s0), n, _p(losses, ctypes.c_double), ctypes.byref(syncs))
    return W, U, losses, int(syncs.value)


def run_minibatch(c: Cfg, X, y=None, t=None, w=None, u=None, s0=0, n_steps=None):
    """Mini-batch SGD of Eq. 1 on one model with the union of the K workers' mini-batches."""
    d = num_params(c)
    w = init_params(c) if w is None else np.array(w, dtype=np.float64).reshape(d)
    u = np.zeros_like(w) if u is None else np.array(u, dtype=np.float64).reshape(d)
    n = int(c.T - s0 if n_steps is None else n_steps)
    losses = np.zeros(n, dtype=np.float64)
    X, y, t = _f32(X), _i32(y), _f32(t)
    lib().oracle_run_minibatch(ctypes.byref(c), _p(X, ctypes.c_float), _p(y, ctypes.c_int32),
                               _p(t, ctypes.c_float), _p(w, ctypes.c_double),
                               _p(u, ctypes.c_double), int(s0), n, _p(losses, ctypes.c_double))
    return w, u, losses


def eval_loss(c: Cfg, w, X, y=None, t=None, n=None) -> float:
    w = np.ascontiguousarray(w, dtype=np.float64)
    X, y, t = _f32(X), _i32(y), _f32(t)
    n = int(X.shape[0] if n is None else n)
    return float(lib().oracle_eval_loss(ctypes.byref(c), _p(w, ctypes.c_double),
                                        _p(X, ctypes.c_float), _p(y, ctypes.c_int32),
                                        _p(t, ctypes.c_float), n))


def bf16_round(x: float) -> float:
    return float(lib().oracle_bf16_round(float(x)))
