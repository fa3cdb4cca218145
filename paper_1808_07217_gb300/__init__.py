"""Python binding of liblsgd (include/lsgd.h): the GB300 hot path of local / post-local SGD.

Argument marshalling only -- every step of the method runs in the CUDA kernels of ``csrc/``.
Functions keep the C names; each raises :class:`LsgdError` when the C call returns a non-OK status.
PyTorch supplies device memory (its caching allocator, through the C allocator callbacks) and the
current CUDA stream.  There is no CPU fallback: if the library has not been built, every call
raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import _build

LIB_PATH = _build.LIB

MAX_LAYERS = 8
MLP, LSQ, RESNET20 = 0, 1, 2
FP32, BF16 = 0, 1
INIT_ZERO, INIT_HE = 0, 1
COMPRESS_NONE, COMPRESS_SIGN, COMPRESS_EF_SIGN = 0, 1, 2
STATE_WREF, STATE_ERROR, STATE_GLOBAL_MOMENTUM = 0, 1, 2
HWARM_NONE, HWARM_LINEAR, HWARM_EXPONENTIAL, HWARM_CONSTANT = 0, 1, 2, 3
SAMPLE_SHARDS, SAMPLE_RESHUFFLE = 0, 1

OK, EINVAL, ENOMEM, ECUDA, ESTATE, ENONFINITE, ETIMEOUT, EUNSUPPORTED, EIO = range(9)
_STATUS = {0: "OK", 1: "EINVAL", 2: "ENOMEM", 3: "ECUDA", 4: "ESTATE", 5: "ENONFINITE",
           6: "ETIMEOUT", 7: "EUNSUPPORTED", 8: "EIO"}

# Every symbol include/lsgd.h declares (checked by the tests).
EXPORTS = [
    "lsgd_create", "lsgd_destroy", "lsgd_set_dataset", "lsgd_set_targets", "lsgd_local_step",
    "lsgd_local_step_batch", "lsgd_sync_average", "lsgd_run", "lsgd_params", "lsgd_momentum",
    "lsgd_set_params", "lsgd_set_momentum", "lsgd_losses", "lsgd_debug_indices", "lsgd_eval_loss",
    "lsgd_check_finite", "lsgd_save", "lsgd_load", "lsgd_num_params", "lsgd_step_count",
    "lsgd_sync_count", "lsgd_total_steps", "lsgd_lr_at", "lsgd_kernel_launches", "lsgd_last_error",
    "lsgd_kway_average", "lsgd_sgd_update", "lsgd_sample_indices", "lsgd_profile_enable",
    "lsgd_profile_read", "lsgd_grouped_gemm_bf16", "lsgd_batchnorm_stats",
    "lsgd_batchnorm_stats_noalloc", "lsgd_block_average", "lsgd_block_sync_count",
    "lsgd_sync_state", "lsgd_set_sync_state", "lsgd_schedule", "lsgd_device_status",
    "lsgd_bounded_wait_selftest", "lsgd_losses_async", "lsgd_synchronize", "lsgd_set_step",
    "lsgd_conv_wgrad_bf16", "lsgd_conv3x3_bf16", "lsgd_conv3x3_bn_bf16", "lsgd_run_batch",
]
PHASES = ["input", "forward", "loss", "backward", "update", "average"]


class LsgdError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{_STATUS.get(status, status)}: {message}")
        self.status = status


class Model(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("n_layers", ctypes.c_int),
                ("widths", ctypes.c_int * (MAX_LAYERS + 1)), ("init", ctypes.c_int),
                ("in_h", ctypes.c_int), ("in_w", ctypes.c_int), ("in_c", ctypes.c_int),
                ("n_classes", ctypes.c_int), ("base_ch", ctypes.c_int), ("res_blocks", ctypes.c_int)]


class LrSchedule(ctypes.Structure):
    _fields_ = [("base_lr", ctypes.c_double), ("scale_by_K", ctypes.c_int),
                ("warmup_epochs", ctypes.c_double), ("n_milestones", ctypes.c_int),
                ("milestone_frac", ctypes.c_double * 4), ("decay", ctypes.c_double)]


class Profile(ctypes.Structure):
    _fields_ = [("count", ctypes.c_int64 * 6), ("ms", ctypes.c_double * 6)]


ALLOC_FN = ctypes.CFUNCTYPE(ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p)
FREE_FN = ctypes.CFUNCTYPE(None, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p)


class Allocator(ctypes.Structure):
    _fields_ = [("alloc", ALLOC_FN), ("free", FREE_FN), ("user", ctypes.c_void_p)]


class Config(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int), ("B_loc", ctypes.c_int), ("H", ctypes.c_int),
                ("t_switch", ctypes.c_int64), ("total_steps", ctypes.c_int64),
                ("epochs", ctypes.c_double), ("N", ctypes.c_int64), ("model", Model),
                ("lr", LrSchedule), ("momentum", ctypes.c_double), ("nesterov", ctypes.c_int),
                ("weight_decay", ctypes.c_double), ("seed", ctypes.c_uint64),
                ("precision", ctypes.c_int), ("fused_update", ctypes.c_int),
                ("hier_block", ctypes.c_int), ("hier_rounds", ctypes.c_int),
                ("compress", ctypes.c_int), ("global_momentum", ctypes.c_double),
                ("h_warmup", ctypes.c_int), ("h_warmup_epochs", ctypes.c_double),
                ("sampling", ctypes.c_int)]


def make_config(K=1, B_loc=1, H=1, t_switch=-1, total_steps=0, epochs=0.0, N=1, kind=MLP,
                widths=(3072, 10), init=INIT_HE, in_hwc=(32, 32, 3), n_classes=10, base_ch=16,
                res_blocks=3, base_lr=0.1, scale_by_K=False, warmup_epochs=0.0, milestones=(),
                decay=0.1, momentum=0.0, nesterov=False, weight_decay=0.0, seed=0,
                precision=FP32, fused_update=False, hier_block=0, hier_rounds=1, compress=0,
                global_momentum=0.0, h_warmup=0, h_warmup_epochs=0.0, sampling=0) -> Config:
    c = Config()
    c.K, c.B_loc, c.H = int(K), int(B_loc), int(H)
    c.t_switch, c.total_steps, c.epochs, c.N = int(t_switch), int(total_steps), float(epochs), int(N)
    c.model.kind = int(kind)
    if kind != RESNET20:
        c.model.n_layers = len(widths) - 1
        for i, w in enumerate(widths):
            c.model.widths[i] = int(w)
    c.model.init = int(init)
    c.model.in_h, c.model.in_w, c.model.in_c = (int(v) for v in in_hwc)
    c.model.n_classes, c.model.base_ch, c.model.res_blocks = int(n_classes), int(base_ch), int(res_blocks)
    c.lr.base_lr = float(base_lr)
    c.lr.scale_by_K = int(bool(scale_by_K))
    c.lr.warmup_epochs = float(warmup_epochs)
    c.lr.n_milestones = len(milestones)
    for i, m in enumerate(milestones):
        c.lr.milestone_frac[i] = float(m)
    c.lr.decay = float(decay)
    c.momentum, c.nesterov, c.weight_decay = float(momentum), int(bool(nesterov)), float(weight_decay)
    c.seed = int(seed)
    c.precision = int(precision)
    c.fused_update = int(bool(fused_update))
    c.hier_block, c.hier_rounds = int(hier_block), int(hier_rounds)
    c.compress, c.global_momentum = int(compress), float(global_momentum)
    c.h_warmup, c.h_warmup_epochs = int(h_warmup), float(h_warmup_epochs)
    c.sampling = int(sampling)
    return c


_lib = None


def lib():
    """Load liblsgd.so (built by ``__graft_entry__.build()``); raises if it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"CUDA library not built: {LIB_PATH} is missing "
                               "(run __graft_entry__.build())")
        L = ctypes.CDLL(LIB_PATH)
        P = ctypes.POINTER
        vp, i64, st = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        sig = {
            "lsgd_create": ([P(Config), P(Allocator), vp, P(vp)], st),
            "lsgd_destroy": ([vp], None),
            "lsgd_set_dataset": ([vp, vp, vp, i64], st),
            "lsgd_set_targets": ([vp, vp, vp, i64], st),
            "lsgd_local_step": ([vp], st),
            "lsgd_local_step_batch": ([vp, vp, vp, ctypes.c_int], st),
            "lsgd_sync_average": ([vp], st),
            "lsgd_run": ([vp, i64], st),
            "lsgd_params": ([vp, ctypes.c_int, vp, ctypes.c_int, ctypes.c_size_t], st),
            "lsgd_momentum": ([vp, ctypes.c_int, vp, ctypes.c_int, ctypes.c_size_t], st),
            "lsgd_set_params": ([vp, ctypes.c_int, vp, ctypes.c_size_t], st),
            "lsgd_set_momentum": ([vp, ctypes.c_int, vp, ctypes.c_size_t], st),
            "lsgd_sync_state": ([vp, ctypes.c_int, ctypes.c_int, vp, ctypes.c_size_t], st),
            "lsgd_schedule": ([P(Config), i64, vp, vp], st),
            "lsgd_device_status": ([vp], st),
            "lsgd_bounded_wait_selftest": ([ctypes.c_int, ctypes.c_double, vp], st),
            "lsgd_set_sync_state": ([vp, ctypes.c_int, ctypes.c_int, vp, ctypes.c_size_t], st),
            "lsgd_losses": ([vp, vp, i64], st),
            "lsgd_losses_async": ([vp, vp, i64], st),
            "lsgd_synchronize": ([vp], st),
            "lsgd_debug_indices": ([vp, i64, vp], st),
            "lsgd_eval_loss": ([vp, ctypes.c_int, i64, P(ctypes.c_double)], st),
            "lsgd_check_finite": ([vp], st),
            "lsgd_save": ([vp, ctypes.c_char_p], st),
            "lsgd_load": ([vp, ctypes.c_char_p], st),
            "lsgd_num_params": ([vp], i64),
            "lsgd_step_count": ([vp], i64),
            "lsgd_set_step": ([vp, i64], st),
            "lsgd_conv_wgrad_bf16": ([vp, vp, vp] + [ctypes.c_int] * 7 + [vp], st),
            "lsgd_conv3x3_bf16": ([ctypes.c_int, vp, vp, vp] + [ctypes.c_int] * 7 + [vp], st),
            "lsgd_conv3x3_bn_bf16": ([vp] * 5 + [ctypes.c_int] * 7 + [vp], st),
            "lsgd_run_batch": ([vp, vp, vp, ctypes.c_int], st),
            "lsgd_sync_count": ([vp], i64),
            "lsgd_block_sync_count": ([vp], i64),
            "lsgd_block_average": ([vp], st),
            "lsgd_total_steps": ([vp], i64),
            "lsgd_lr_at": ([vp, i64], ctypes.c_double),
            "lsgd_kernel_launches": ([vp], i64),
            "lsgd_last_error": ([vp], ctypes.c_char_p),
            "lsgd_kway_average": ([vp, vp, ctypes.c_int, i64, vp], st),
            "lsgd_sgd_update": ([vp, vp, vp, vp, i64, ctypes.c_float, ctypes.c_float, ctypes.c_int,
                                 ctypes.c_float, i64, i64, vp], st),
            "lsgd_sample_indices": ([vp, ctypes.c_uint64, i64, ctypes.c_int, ctypes.c_int, i64, vp], st),
            "lsgd_profile_enable": ([vp, ctypes.c_int], st),
            "lsgd_batchnorm_stats": ([vp, i64, ctypes.c_int, ctypes.c_int, vp, vp, vp], st),
            "lsgd_batchnorm_stats_noalloc": ([vp, i64, ctypes.c_int, ctypes.c_int, vp, vp, vp], st),
            "lsgd_grouped_gemm_bf16": ([vp, ctypes.c_int, vp, ctypes.c_int, vp, ctypes.c_int,
                                        ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, vp], st),
            "lsgd_profile_read": ([vp, P(Profile)], st),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _check(status, ctx=None):
    if status != OK:
        h = ctx.handle if isinstance(ctx, Ctx) else None
        msg = lib().lsgd_last_error(h)
        raise LsgdError(status, msg.decode() if msg else "")


def _ptr(a):
    """Data pointer of a numpy array or torch tensor."""
    if a is None:
        return None
    if hasattr(a, "data_ptr"):
        return ctypes.c_void_p(a.data_ptr())
    return ctypes.c_void_p(a.ctypes.data)


def _current_stream():
    import torch

    return torch.cuda.current_stream().cuda_stream


class Ctx:
    """Owns an lsgd_ctx handle and the allocator callbacks that must outlive it."""

    def __init__(self, handle, callbacks, stream):
        self.handle = handle
        self._callbacks = callbacks
        self.stream = stream

    def __del__(self):
        try:
            lsgd_destroy(self)
        except Exception:
            pass


def torch_allocator(device=None):
    """An lsgd_allocator backed by PyTorch's CUDA caching allocator."""
    import torch

    dev = torch.cuda.current_device() if device is None else device

    def _alloc(user, nbytes, stream):
        try:
            return torch.cuda.caching_allocator_alloc(int(nbytes), dev, stream)
        except Exception:
            return None

    def _free(user, p, stream):
        torch.cuda.caching_allocator_delete(p)

    cb = (ALLOC_FN(_alloc), FREE_FN(_free))
    a = Allocator(cb[0], cb[1], None)
    return a, cb


def lsgd_create(cfg: Config, allocator="torch", stream=None) -> Ctx:
    if stream is None:
        stream = _current_stream()
    cbs = None
    ap = None
    if allocator == "torch":
        a, cbs = torch_allocator()
        ap = ctypes.byref(a)
        cbs = (a, cbs)
    elif allocator is not None:
        ap = ctypes.byref(allocator)
        cbs = allocator
    h = ctypes.c_void_p()
    _check(lib().lsgd_create(ctypes.byref(cfg), ap, ctypes.c_void_p(stream), ctypes.byref(h)))
    return Ctx(h, cbs, stream)


def lsgd_destroy(ctx: Ctx):
    if ctx.handle:
        lib().lsgd_destroy(ctx.handle)
        ctx.handle = None


def lsgd_set_dataset(ctx: Ctx, X, labels):
    X = np.ascontiguousarray(X, dtype=np.float32)
    y = np.ascontiguousarray(labels, dtype=np.int32)
    _check(lib().lsgd_set_dataset(ctx.handle, _ptr(X), _ptr(y), X.shape[0]), ctx)


def lsgd_set_targets(ctx: Ctx, X, targets):
    X = np.ascontiguousarray(X, dtype=np.float32)
    t = np.ascontiguousarray(targets, dtype=np.float32)
    _check(lib().lsgd_set_targets(ctx.handle, _ptr(X), _ptr(t), X.shape[0]), ctx)


def lsgd_local_step(ctx: Ctx):
    _check(lib().lsgd_local_step(ctx.handle), ctx)


def lsgd_local_step_batch(ctx: Ctx, x, labels_or_targets):
    """x [K, B, D] fp32 and labels [K, B] int32 (targets fp32 for LSQ): numpy / host tensors
    (pinned memory copies asynchronously) or CUDA tensors."""
    on_dev = int(hasattr(x, "is_cuda") and x.is_cuda)
    _check(lib().lsgd_local_step_batch(ctx.handle, _ptr(x), _ptr(labels_or_targets), on_dev), ctx)


def lsgd_run_batch(ctx: Ctx, x, labels_or_targets):
    """One step of lsgd_run's schedule (local step + the average ending it, if any) on a
    caller-supplied mini-batch, arguments as lsgd_local_step_batch."""
    on_dev = int(hasattr(x, "is_cuda") and x.is_cuda)
    _check(lib().lsgd_run_batch(ctx.handle, _ptr(x), _ptr(labels_or_targets), on_dev), ctx)


def lsgd_sync_average(ctx: Ctx):
    _check(lib().lsgd_sync_average(ctx.handle), ctx)


def lsgd_run(ctx: Ctx, n_steps: int):
    _check(lib().lsgd_run(ctx.handle, int(n_steps)), ctx)


def lsgd_num_params(ctx: Ctx) -> int:
    return int(lib().lsgd_num_params(ctx.handle))


def _get(fn, ctx, k, dst):
    d = lsgd_num_params(ctx)
    if dst is None:
        dst = np.empty(d, dtype=np.float32)
        _check(fn(ctx.handle, int(k), _ptr(dst), 0, d), ctx)
        return dst
    on_dev = int(hasattr(dst, "is_cuda") and dst.is_cuda)
    _check(fn(ctx.handle, int(k), _ptr(dst), on_dev, d), ctx)
    return dst


def lsgd_params(ctx: Ctx, k: int = -1, dst=None):
    return _get(lib().lsgd_params, ctx, k, dst)


def lsgd_momentum(ctx: Ctx, k: int = -1, dst=None):
    return _get(lib().lsgd_momentum, ctx, k, dst)


def lsgd_set_params(ctx: Ctx, k: int, w):
    w = np.ascontiguousarray(w, dtype=np.float32)
    _check(lib().lsgd_set_params(ctx.handle, int(k), _ptr(w), w.size), ctx)


def lsgd_set_momentum(ctx: Ctx, k: int, u):
    u = np.ascontiguousarray(u, dtype=np.float32)
    _check(lib().lsgd_set_momentum(ctx.handle, int(k), _ptr(u), u.size), ctx)


def lsgd_device_status(ctx: Ctx = None) -> int:
    """OK, or ETIMEOUT if a bounded device wait ran out since the last check (flag cleared)."""
    return int(lib().lsgd_device_status(ctx.handle if ctx is not None else None))


def lsgd_bounded_wait_selftest(arrive: bool, limit_ms: float, stream=None) -> int:
    """Status of one bounded wait that completes only if `arrive`: OK or ETIMEOUT."""
    stream = _current_stream() if stream is None else stream
    return int(lib().lsgd_bounded_wait_selftest(int(bool(arrive)), float(limit_ms), stream))


def lsgd_schedule(cfg: Config, n_steps: int):
    """(lr[s], sync_kind[s]) for s < n_steps, computed on the host (no GPU needed)."""
    lr = np.zeros(int(n_steps), dtype=np.float64)
    kinds = np.zeros(int(n_steps), dtype=np.int32)
    st = lib().lsgd_schedule(ctypes.byref(cfg), int(n_steps), _ptr(lr), _ptr(kinds))
    if st != OK:
        raise RuntimeError(f"lsgd_schedule: status {st}: {lib().lsgd_last_error(None).decode()}")
    return lr, kinds


def lsgd_sync_state(ctx: Ctx, which: int, k: int = 0):
    out = np.empty(lsgd_num_params(ctx), dtype=np.float32)
    _check(lib().lsgd_sync_state(ctx.handle, int(which), int(k), _ptr(out), out.size), ctx)
    return out


def lsgd_set_sync_state(ctx: Ctx, which: int, k: int, v):
    v = np.ascontiguousarray(v, dtype=np.float32)
    _check(lib().lsgd_set_sync_state(ctx.handle, int(which), int(k), _ptr(v), v.size), ctx)


def lsgd_losses(ctx: Ctx, n_steps: int, K: int):
    out = np.empty((int(n_steps), int(K)), dtype=np.float32)
    _check(lib().lsgd_losses(ctx.handle, _ptr(out), int(n_steps)), ctx)
    return out


def lsgd_losses_async(ctx: Ctx, out, n_steps: int):
    """Enqueue the read of the last n_steps steps' losses into `out` ([n_steps, K] fp32 host
    array or pinned tensor the caller keeps alive); valid after lsgd_synchronize."""
    _check(lib().lsgd_losses_async(ctx.handle, _ptr(out), int(n_steps)), ctx)


def lsgd_synchronize(ctx: Ctx):
    _check(lib().lsgd_synchronize(ctx.handle), ctx)


def lsgd_debug_indices(ctx: Ctx, step: int, K: int, B: int):
    out = np.empty((int(K), int(B)), dtype=np.int32)
    _check(lib().lsgd_debug_indices(ctx.handle, int(step), _ptr(out)), ctx)
    return out


def lsgd_eval_loss(ctx: Ctx, k: int, n: int) -> float:
    v = ctypes.c_double()
    _check(lib().lsgd_eval_loss(ctx.handle, int(k), int(n), ctypes.byref(v)), ctx)
    return float(v.value)


def lsgd_check_finite(ctx: Ctx) -> bool:
    s = lib().lsgd_check_finite(ctx.handle)
    if s == ENONFINITE:
        return False
    _check(s, ctx)
    return True


def lsgd_save(ctx: Ctx, path: str):
    _check(lib().lsgd_save(ctx.handle, os.fsencode(path)), ctx)


def lsgd_load(ctx: Ctx, path: str):
    _check(lib().lsgd_load(ctx.handle, os.fsencode(path)), ctx)


def lsgd_step_count(ctx: Ctx) -> int:
    return int(lib().lsgd_step_count(ctx.handle))


def lsgd_set_step(ctx: Ctx, step: int):
    _check(lib().lsgd_set_step(ctx.handle, int(step)), ctx)


def lsgd_sync_count(ctx: Ctx) -> int:
    return int(lib().lsgd_sync_count(ctx.handle))


def lsgd_block_sync_count(ctx: Ctx) -> int:
    return int(lib().lsgd_block_sync_count(ctx.handle))


def lsgd_block_average(ctx: Ctx):
    _check(lib().lsgd_block_average(ctx.handle), ctx)


def lsgd_total_steps(ctx: Ctx) -> int:
    return int(lib().lsgd_total_steps(ctx.handle))


def lsgd_lr_at(ctx: Ctx, step: int) -> float:
    return float(lib().lsgd_lr_at(ctx.handle, int(step)))


def lsgd_kernel_launches(ctx: Ctx) -> int:
    return int(lib().lsgd_kernel_launches(ctx.handle))


def lsgd_last_error(ctx: Ctx | None = None) -> str:
    m = lib().lsgd_last_error(ctx.handle if ctx else None)
    return m.decode() if m else ""


def lsgd_kway_average(W, Wb, K: int, d: int, stream=None):
    """W: CUDA float32 tensor [K, d]; Wb: CUDA bfloat16/int16 tensor [K, d] or None."""
    stream = _current_stream() if stream is None else stream
    _check(lib().lsgd_kway_average(_ptr(W), _ptr(Wb), int(K), int(d), ctypes.c_void_p(stream)))


def lsgd_sgd_update(w, u, g, Wb, n, lr, momentum=0.0, nesterov=False, weight_decay=0.0,
                    period=0, decay_end=0, stream=None):
    stream = _current_stream() if stream is None else stream
    _check(lib().lsgd_sgd_update(_ptr(w), _ptr(u), _ptr(g), _ptr(Wb), int(n), float(lr),
                                 float(momentum), int(bool(nesterov)), float(weight_decay),
                                 int(period), int(decay_end), ctypes.c_void_p(stream)))


def lsgd_sample_indices(dst, seed: int, step: int, K: int, B: int, N: int, stream=None):
    stream = _current_stream() if stream is None else stream
    _check(lib().lsgd_sample_indices(_ptr(dst), int(seed), int(step), int(K), int(B), int(N),
                                     ctypes.c_void_p(stream)))


def lsgd_profile_enable(ctx: Ctx, enable: bool = True):
    _check(lib().lsgd_profile_enable(ctx.handle, int(bool(enable))), ctx)


def lsgd_profile_read(ctx: Ctx) -> dict:
    """{phase: (count, total_ms)} accumulated since profiling was enabled."""
    p = Profile()
    _check(lib().lsgd_profile_read(ctx.handle, ctypes.byref(p)), ctx)
    return {name: (int(p.count[i]), float(p.ms[i])) for i, name in enumerate(PHASES)}


def lsgd_grouped_gemm_bf16(A, a_mn: bool, B, b_mn: bool, C, M: int, N: int, Kd: int, G: int,
                           engine: int = 0, stream=None):
    """C[g] = A[g] B[g]^T on CUDA tensors (A, B bfloat16; C float32); engine 0 tcgen05, 1 SIMT."""
    stream = _current_stream() if stream is None else stream
    _check(lib().lsgd_grouped_gemm_bf16(_ptr(A), int(bool(a_mn)), _ptr(B), int(bool(b_mn)), _ptr(C),
                                        int(M), int(N), int(Kd), int(G), int(engine),
                                        ctypes.c_void_p(stream)))


def lsgd_conv_wgrad_bf16(x, dy, dW, G: int, B: int, Hout: int, Wout: int, Cin: int, Cout: int,
                         stride: int, stream=None):
    """dW [G, Cout, 3, 3, Cin] float32 = the 3x3 (pad 1, stride) convolution weight gradient of
    NHWC bfloat16 CUDA tensors x [G, B, stride Hout, stride Wout, Cin] and dy [G, B, Hout, Wout, Cout]."""
    stream = _current_stream() if stream is None else stream
    _check(lib().lsgd_conv_wgrad_bf16(_ptr(x), _ptr(dy), _ptr(dW), int(G), int(B), int(Hout),
                                      int(Wout), int(Cin), int(Cout), int(stride),
                                      ctypes.c_void_p(stream)))


CONV_FORWARD, CONV_DGRAD = 0, 1


def lsgd_conv3x3_bf16(mode: int, inp, W, out, G: int, B: int, Hin: int, Win: int, Cin: int,
                      Cout: int, stride: int, stream=None):
    """3x3 (pad 1, stride) convolution of NHWC bfloat16 CUDA tensors on the implicit-GEMM kernel:
    mode CONV_FORWARD: out [G, B, Hout, Wout, Cout] float32 from inp = x [G, B, Hin, Win, Cin];
    mode CONV_DGRAD: out = dx [G, B, Hin, Win, Cin] float32 from inp = dy [G, B, Hout, Wout, Cout];
    W [G, Cout, 3, 3, Cin] bfloat16."""
    stream = _current_stream() if stream is None else stream
    _check(lib().lsgd_conv3x3_bf16(int(mode), _ptr(inp), _ptr(W), _ptr(out), int(G), int(B),
                                   int(Hin), int(Win), int(Cin), int(Cout), int(stride),
                                   ctypes.c_void_p(stream)))


def lsgd_conv3x3_bn_bf16(x, W, y, mean, rstd, G: int, B: int, Hin: int, Win: int, Cin: int,
                         Cout: int, stride: int, stream=None):
    """Forward 3x3 convolution (CONV_FORWARD of lsgd_conv3x3_bf16) with the per-group BatchNorm
    statistics of its output from the convolution's epilogue: y [G, B, Hout, Wout, Cout] float32,
    mean and rstd [G, Cout] float32."""
    stream = _current_stream() if stream is None else stream
    _check(lib().lsgd_conv3x3_bn_bf16(_ptr(x), _ptr(W), _ptr(y), _ptr(mean), _ptr(rstd), int(G),
                                      int(B), int(Hin), int(Win), int(Cin), int(Cout), int(stride),
                                      ctypes.c_void_p(stream)))


def lsgd_batchnorm_stats(y, P: int, C: int, G: int, mean, rstd, stream=None):
    """Per-replica BatchNorm statistics of a CUDA float32 tensor y [G, P, C] into mean, rstd [G, C]."""
    stream = _current_stream() if stream is None else stream
    _check(lib().lsgd_batchnorm_stats(_ptr(y), int(P), int(C), int(G), _ptr(mean), _ptr(rstd),
                                      ctypes.c_void_p(stream)))


def lsgd_batchnorm_stats_noalloc(y, P: int, C: int, G: int, mean, rstd, stream=None):
    """lsgd_batchnorm_stats without any device allocation (fixed 4 MiB scratch inside the library),
    for callers whose device memory is all spoken for; see include/lsgd.h for the limit and the
    shared-scratch rules."""
    stream = _current_stream() if stream is None else stream
    _check(lib().lsgd_batchnorm_stats_noalloc(_ptr(y), int(P), int(C), int(G), _ptr(mean),
                                              _ptr(rstd), ctypes.c_void_p(stream)))
