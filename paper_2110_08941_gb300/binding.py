"""Python binding of libhs (include/hs.h): argument marshalling only.

Every function keeps the C name.  Tensors are torch tensors; the binding passes
their data pointers and the current CUDA stream to the library and does no
arithmetic of its own.  The shared library is built in-tree by
``python -m paper_2110_08941_gb300.build``; importing this package when it is
missing raises ImportError - there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_double, c_float, c_int32, c_int64, c_uint64, c_void_p
from typing import List, Optional, Sequence

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libhs.so")

HS_OK, HS_ERR_INVALID_ARG, HS_ERR_CUDA, HS_ERR_OOM, HS_ERR_UNSUPPORTED, HS_ERR_DEVICE_CHECK = range(6)
HS_MLP, HS_CNN = 0, 1
HS_BF16, HS_FP32_CHECK = 0, 1
HS_SYNC_MEAN, HS_SYNC_CP_WEIGHTED, HS_SYNC_CP_LITERAL = 0, 1, 2
HS_GEMM_FWD_RELU, HS_GEMM_FWD_LOGITS, HS_GEMM_DGRAD, HS_GEMM_WGRAD = 0, 1, 2, 3
HS_GEMM_FORM_SINGLE, HS_GEMM_FORM_PAIR = 0x100, 0x200
HS_GEMM_TEST_STALL = 0x1000

EXPORTED = ("hs_partition_sizes", "hs_param_count", "hs_init", "hs_partition", "hs_step", "hs_sync_params",
            "hs_set_debug", "hs_debug_grads", "hs_worker_losses", "hs_destroy", "hs_status_string",
            "hs_last_error", "hs_last_init_error", "hs_debug_gemm_bf16", "hs_set_profiling", "hs_read_profile",
            "hs_partition_noalloc", "hs_set_optimizer", "hs_optimizer_state", "hs_cosine_lr",
            "hs_set_cp_history", "hs_set_fused_sync", "hs_stage_inputs", "hs_debug_wgrad_avg")
HS_CP_LAST, HS_CP_EMA, HS_CP_WINDOW = 0, 1, 2
PHASES = ("cast", "forward", "loss", "wgrad", "biasgrad", "dgrad", "update")


class HsError(RuntimeError):
    def __init__(self, status: int, msg: str):
        self.status = status
        super().__init__(f"{_status_name(status)}: {msg}")


class hs_model_desc(ctypes.Structure):
    _fields_ = [("arch", c_int32), ("n_layers", c_int32), ("dims", POINTER(c_int32)),
                ("precision", c_int32), ("sync", c_int32)]


class hs_partition_t(ctypes.Structure):
    _fields_ = [("M", c_int32), ("N", c_int32), ("counts_host", POINTER(c_int32)),
                ("offsets_host", POINTER(c_int32)), ("index_map_dev", c_void_p),
                ("weights_host", POINTER(c_double)), ("cp_host", POINTER(c_double)), ("version", c_uint64)]


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libhs.so not built at {LIB_PATH}; run `python -m paper_2110_08941_gb300.build`")
    lib = ctypes.CDLL(LIB_PATH)
    S = c_int32
    sig = {
        "hs_partition_sizes": (S, [c_int32, c_int32, POINTER(c_double), POINTER(c_int32)]),
        "hs_partition_noalloc": (S, [c_int32, c_int32, POINTER(c_double), POINTER(c_int32), c_void_p, c_void_p]),
        "hs_param_count": (S, [POINTER(hs_model_desc), POINTER(c_int64)]),
        "hs_init": (S, [POINTER(hs_model_desc), c_int32, POINTER(c_double), c_int32, POINTER(c_void_p)]),
        "hs_partition": (S, [c_void_p, POINTER(c_double), POINTER(c_int32), c_void_p, c_void_p,
                             POINTER(hs_partition_t)]),
        "hs_step": (S, [c_void_p, c_void_p, c_void_p, c_void_p, POINTER(hs_partition_t), c_float, c_void_p,
                        POINTER(c_float)]),
        "hs_sync_params": (S, [c_void_p, c_void_p, c_void_p]),
        "hs_stage_inputs": (S, [c_void_p, c_void_p, c_void_p, c_void_p, POINTER(c_void_p), POINTER(c_void_p)]),
        "hs_set_debug": (S, [c_void_p, c_int32]),
        "hs_set_profiling": (S, [c_void_p, c_int32]),
        "hs_set_optimizer": (S, [c_void_p, c_float, c_float]),
        "hs_set_cp_history": (S, [c_void_p, c_int32, c_double]),
        "hs_set_fused_sync": (S, [c_void_p, c_int32]),
        "hs_optimizer_state": (S, [c_void_p, c_void_p, c_int32, c_void_p]),
        "hs_cosine_lr": (c_double, [c_double, c_double, c_int64, c_int64]),
        "hs_read_profile": (S, [c_void_p, POINTER(c_double), POINTER(c_int64)]),
        "hs_debug_grads": (S, [c_void_p, c_void_p, c_void_p, c_void_p]),
        "hs_worker_losses": (S, [c_void_p, POINTER(c_float)]),
        "hs_destroy": (None, [c_void_p]),
        "hs_status_string": (ctypes.c_char_p, [c_int32]),
        "hs_last_error": (ctypes.c_char_p, [c_void_p]),
        "hs_last_init_error": (ctypes.c_char_p, []),
        "hs_debug_gemm_bf16": (S, [c_int32, c_int32, c_int32, c_int32, c_void_p, c_int64, c_void_p, c_int64,
                                   c_void_p, c_int64, c_void_p, c_void_p, c_int64, POINTER(c_int32), c_int32,
                                   c_int64, c_void_p]),
        "hs_debug_wgrad_avg": (S, [c_int32, c_int32, c_void_p, c_int64, c_void_p, c_int64, POINTER(c_int32), c_int32,
                                   c_void_p, ctypes.c_float, c_void_p, c_int64, c_void_p, c_int64, c_int32, c_void_p]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = _load()


def _status_name(s: int) -> str:
    return _lib.hs_status_string(s).decode()


def _check(status: int, ctx_ptr=None, init: bool = False):
    if status == HS_OK:
        return
    if init or ctx_ptr is None:
        msg = _lib.hs_last_init_error().decode()
    else:
        msg = _lib.hs_last_error(ctx_ptr).decode()
    raise HsError(status, msg)


def _stream_ptr(stream) -> int:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


def _desc(arch: int, dims: Sequence[int], precision: int, sync: int):
    arr = (c_int32 * len(dims))(*[int(d) for d in dims])
    n_layers = len(dims) - 1 if arch == HS_MLP else 0
    return hs_model_desc(arch, n_layers, ctypes.cast(arr, POINTER(c_int32)), precision, sync), arr


# ------------------------------------------------------------------------------- host-only calls
def hs_partition_sizes(cp: Sequence[float], n: int) -> List[int]:
    m = len(cp)
    cpa = (c_double * max(m, 1))(*[float(v) for v in cp])
    out = (c_int32 * max(m, 1))()
    _check(_lib.hs_partition_sizes(m, int(n), cpa, out))
    return list(out[:m])


def _check_index_map(index_map_out, n: int):
    """The library writes n int32 through index_map_out's pointer: reject anything else first."""
    import torch
    if not (isinstance(index_map_out, torch.Tensor) and index_map_out.is_cuda
            and index_map_out.dtype == torch.int32 and index_map_out.is_contiguous()
            and index_map_out.numel() == n and index_map_out.device.index == torch.cuda.current_device()):
        raise ValueError(f"index_map_out must be a contiguous int32 CUDA tensor of {n} elements on the current device")


def hs_partition_noalloc(cp: Sequence[float], n: int, index_map_out, stream=None) -> List[int]:
    """Partition sizes and the device index map without a context or any device allocation."""
    _check_index_map(index_map_out, int(n))
    m = len(cp)
    cpa = (c_double * max(m, 1))(*[float(v) for v in cp])
    out = (c_int32 * max(m, 1))()
    _check(_lib.hs_partition_noalloc(m, int(n), cpa, out, c_void_p(index_map_out.data_ptr()),
                                     c_void_p(_stream_ptr(stream))))
    return list(out[:m])


def hs_param_count(arch: int, dims: Sequence[int]) -> int:
    d, keep = _desc(arch, dims, HS_BF16, HS_SYNC_MEAN)
    p = c_int64()
    _check(_lib.hs_param_count(ctypes.byref(d), ctypes.byref(p)))
    return p.value


# ------------------------------------------------------------------------------- context
class Partition:
    """Snapshot of hs_partition_t (host arrays copied out)."""

    def __init__(self, raw: hs_partition_t):
        self.raw = raw
        self.M, self.N, self.version = raw.M, raw.N, raw.version
        self.counts = [raw.counts_host[i] for i in range(raw.M)]
        self.offsets = [raw.offsets_host[i] for i in range(raw.M + 1)]
        self.weights = [raw.weights_host[i] for i in range(raw.M)]
        self.cp = [raw.cp_host[i] for i in range(raw.M)]
        self.index_map_dev = raw.index_map_dev


class Context:
    def __init__(self, ptr: int, arch: int, dims, M: int, N: int, P: int, precision: int, sync: int):
        self.ptr = c_void_p(ptr)
        self.arch, self.dims, self.M, self.N, self.P = arch, tuple(dims), M, N, P
        self.precision, self.sync = precision, sync
        self.partition: Optional[Partition] = None

    def close(self):
        if self.ptr and self.ptr.value:
            _lib.hs_destroy(self.ptr)
            self.ptr = c_void_p(0)

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def hs_init(arch: int, dims: Sequence[int], M: int, global_batch: int, compute_weights=None,
            precision: int = HS_BF16, sync: int = HS_SYNC_CP_WEIGHTED) -> Context:
    d, keep = _desc(arch, dims, precision, sync)
    cw = None
    if compute_weights is not None:
        cw = (c_double * M)(*[float(v) for v in compute_weights])
    out = c_void_p()
    _check(_lib.hs_init(ctypes.byref(d), int(M), cw, int(global_batch), ctypes.byref(out)), init=True)
    ctx = Context(out.value, arch, dims, M, global_batch, hs_param_count(arch, dims), precision, sync)
    ctx.partition = hs_partition(ctx)
    return ctx


def hs_partition(ctx: Context, measured_throughputs=None, index_map_out=None, stream=None) -> Partition:
    tp = None
    if measured_throughputs is not None:
        tp = (c_double * ctx.M)(*[float(v) for v in measured_throughputs])
    raw = hs_partition_t()
    im = None
    if index_map_out is not None:
        _check_index_map(index_map_out, ctx.N)
        im = c_void_p(index_map_out.data_ptr())
    s = c_void_p(_stream_ptr(stream)) if (tp is not None or im is not None) else c_void_p(0)
    _check(_lib.hs_partition(ctx.ptr, tp, None, im, s, ctypes.byref(raw)), ctx.ptr)
    ctx.partition = Partition(raw)
    return ctx.partition


class StagedInputs:
    """One step's x and y in a context staging slot (device pointers from hs_stage_inputs); pass it
    to hs_step as x (y omitted).  Holds the host tensors until then."""

    def __init__(self, x_ptr: int, y_ptr: int, host):
        self.x_ptr, self.y_ptr, self._host = x_ptr, y_ptr, host


def hs_stage_inputs(ctx: Context, x_host, y_host, stream=None) -> StagedInputs:
    import torch
    assert x_host.dtype == torch.float32 and x_host.is_contiguous() and not x_host.is_cuda
    assert y_host.dtype == torch.int32 and y_host.is_contiguous() and not y_host.is_cuda
    xp, yp = c_void_p(), c_void_p()
    _check(_lib.hs_stage_inputs(ctx.ptr, c_void_p(x_host.data_ptr()), c_void_p(y_host.data_ptr()),
                                c_void_p(_stream_ptr(stream)), ctypes.byref(xp), ctypes.byref(yp)), ctx.ptr)
    return StagedInputs(xp.value, yp.value, (x_host, y_host))


def hs_step(ctx: Context, params, x, y=None, part: Optional[Partition] = None, lr: float = 0.01, stream=None,
            want_loss: bool = True) -> Optional[float]:
    import torch
    assert params.dtype == torch.float32 and params.is_contiguous() and params.is_cuda
    if isinstance(x, StagedInputs):
        assert y is None
        xp, yp = x.x_ptr, x.y_ptr
    else:
        assert x.dtype == torch.float32 and x.is_contiguous()
        assert y.dtype == torch.int32 and y.is_contiguous()
        xp, yp = x.data_ptr(), y.data_ptr()
    loss = c_float()
    raw = ctypes.byref(part.raw) if part is not None else None
    _check(_lib.hs_step(ctx.ptr, c_void_p(params.data_ptr()), c_void_p(xp), c_void_p(yp), raw, float(lr),
                        c_void_p(_stream_ptr(stream)), ctypes.byref(loss) if want_loss else None), ctx.ptr)
    return loss.value if want_loss else None


def hs_sync_params(ctx: Context, params, stream=None):
    _check(_lib.hs_sync_params(ctx.ptr, c_void_p(params.data_ptr()), c_void_p(_stream_ptr(stream))), ctx.ptr)


def hs_set_debug(ctx: Context, enable: bool = True):
    _check(_lib.hs_set_debug(ctx.ptr, 1 if enable else 0), ctx.ptr)


def hs_set_fused_sync(ctx: Context, enable: bool = True):
    _check(_lib.hs_set_fused_sync(ctx.ptr, 1 if enable else 0), ctx.ptr)


def hs_set_cp_history(ctx: Context, mode: int, param: float = 0.0):
    _check(_lib.hs_set_cp_history(ctx.ptr, int(mode), float(param)), ctx.ptr)


def hs_set_optimizer(ctx: Context, momentum: float, weight_decay: float):
    _check(_lib.hs_set_optimizer(ctx.ptr, float(momentum), float(weight_decay)), ctx.ptr)


def hs_optimizer_state(ctx: Context, buf, save: bool, stream=None):
    _check(_lib.hs_optimizer_state(ctx.ptr, c_void_p(buf.data_ptr()), 1 if save else 0,
                                   c_void_p(_stream_ptr(stream))), ctx.ptr)


def hs_cosine_lr(eta0: float, eta_min: float, t: int, T: int) -> float:
    return _lib.hs_cosine_lr(float(eta0), float(eta_min), int(t), int(T))


def hs_set_profiling(ctx: Context, enable: bool = True):
    _check(_lib.hs_set_profiling(ctx.ptr, 1 if enable else 0), ctx.ptr)


def hs_read_profile(ctx: Context):
    """{phase: (ms, launches)} summed since the last read (waits for the recorded events)."""
    ms = (c_double * len(PHASES))()
    n = (c_int64 * len(PHASES))()
    _check(_lib.hs_read_profile(ctx.ptr, ms, n), ctx.ptr)
    return {name: (ms[i], n[i]) for i, name in enumerate(PHASES)}


def hs_debug_grads(ctx: Context, g_out=None, slabs_out=None, stream=None):
    _check(_lib.hs_debug_grads(ctx.ptr, c_void_p(g_out.data_ptr() if g_out is not None else 0),
                               c_void_p(slabs_out.data_ptr() if slabs_out is not None else 0),
                               c_void_p(_stream_ptr(stream))), ctx.ptr)


def hs_worker_losses(ctx: Context) -> List[float]:
    out = (c_float * ctx.M)()
    _check(_lib.hs_worker_losses(ctx.ptr, out), ctx.ptr)
    return list(out)


def hs_destroy(ctx: Context):
    ctx.close()


def hs_debug_wgrad_avg(A, B, k_offsets, wavg, lr: float, theta, shadow, test_stall: bool = False, stream=None):
    """theta -= lr * sum_g wavg[g] A[k_g]^T B[k_g]; shadow = bf16(theta) (test hook, include/hs_debug.h).
    A: bf16 [K, M], B: bf16 [K, N], wavg: fp32 [groups], theta: fp32 [M, N], shadow: bf16 [M, N]
    (device tensors); k_offsets: groups + 1 row offsets."""
    ko = (c_int32 * len(k_offsets))(*[int(v) for v in k_offsets])
    M, N = int(theta.shape[0]), int(theta.shape[1])
    _check(_lib.hs_debug_wgrad_avg(M, N, c_void_p(A.data_ptr()), int(A.stride(0)), c_void_p(B.data_ptr()),
                                   int(B.stride(0)), ko, len(k_offsets) - 1, c_void_p(wavg.data_ptr()), float(lr),
                                   c_void_p(theta.data_ptr()), int(theta.stride(0)), c_void_p(shadow.data_ptr()),
                                   int(shadow.stride(0)), 1 if test_stall else 0, c_void_p(_stream_ptr(stream))))


def hs_debug_gemm_bf16(mode: int, M: int, N: int, K: int, A, B, D, bias=None, Z=None, k_offsets=None,
                       d_gstride: int = 0, stream=None):
    """Run one product through the tensor-core kernel (test hook, include/hs_debug.h)."""
    ko = None
    groups = 1
    if k_offsets is not None:
        groups = len(k_offsets) - 1
        ko = (c_int32 * len(k_offsets))(*[int(v) for v in k_offsets])
    _check(_lib.hs_debug_gemm_bf16(
        int(mode), int(M), int(N), int(K), c_void_p(A.data_ptr()), int(A.stride(0)), c_void_p(B.data_ptr()),
        int(B.stride(0)), c_void_p(D.data_ptr()), int(D.stride(0)),
        c_void_p(bias.data_ptr() if bias is not None else 0), c_void_p(Z.data_ptr() if Z is not None else 0),
        int(Z.stride(0)) if Z is not None else 0, ko, groups, int(d_gstride), c_void_p(_stream_ptr(stream))))
