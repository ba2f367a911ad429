"""Python binding of the GB300 DP-SGD step library (``libdpstep.so``).

Argument marshalling only: every function here forwards to the C entry point
of the same name declared in ``include/dp_step.h`` (device pointers, sizes,
the CUDA stream handle).  All arithmetic of the step runs in the library's
CUDA kernels; there is no CPU fallback, and importing a function whose
library is missing raises :class:`LibraryNotBuilt`.

PyTorch appears here only as the owner of device memory and streams.
"""

from __future__ import annotations

import ctypes
import os
from typing import Iterable, Optional, Sequence

import numpy as np

__all__ = [
    "DPError", "LibraryNotBuilt", "lib", "lib_path",
    "DP_OK", "DP_F32", "DP_BF16",
    "DP_NORM_AUTO", "DP_NORM_RANK1", "DP_NORM_GHOST", "DP_NORM_MATERIALISED",
    "DP_NO_NOISE", "DP_NOISE_ONLY", "DP_ACCUMULATE", "DP_WRITE_GRAD", "dp_adamw", "dp_noise_adamw",
    "DP_LAYER_DENSE", "DP_LAYER_CONV2D",
    "dp_layer", "dp_config", "make_config",
    "dp_step_init", "dp_layer_norms", "dp_layer_norms_batch", "dp_clip_factors",
    "dp_clipped_sum_noise", "dp_clipped_sum_noise_batch",
    "dp_audit_emit", "audit_dtype", "dp_audit_record_bytes", "dp_layer_norm_mode", "dp_layer_path",
    "dp_set_noise_key", "dp_step_destroy",
    "dp_last_error", "dp_kernel_launches", "dp_debug_philox", "dp_debug_gaussian",
    "dp_layer_sqnorms_noalloc", "dp_conv2d", "make_conv", "dp_conv2d_dims", "dp_conv2d_unfold",
    "EXPORTED_SYMBOLS",
]

HERE = os.path.dirname(os.path.abspath(__file__))
lib_path = os.path.join(HERE, "libdpstep.so")

DP_OK = 0
DP_F32, DP_BF16 = 0, 1
DP_NORM_AUTO, DP_NORM_RANK1, DP_NORM_GHOST, DP_NORM_MATERIALISED = 0, 1, 2, 3
DP_NO_NOISE, DP_NOISE_ONLY, DP_ACCUMULATE, DP_WRITE_GRAD = 0x1, 0x2, 0x4, 0x8
DP_LAYER_DENSE, DP_LAYER_CONV2D = 0, 1

STATUS_NAMES = {0: "DP_OK", 1: "DP_ERR_ARG", 2: "DP_ERR_SHAPE", 3: "DP_ERR_DTYPE",
                4: "DP_ERR_ORDER", 5: "DP_ERR_NONFINITE", 6: "DP_ERR_CUDA",
                7: "DP_ERR_TIMEOUT", 8: "DP_ERR_OOM", 9: "DP_ERR_UNSUPPORTED"}

# every symbol include/dp_step.h declares
EXPORTED_SYMBOLS = ["dp_step_init", "dp_layer_norms", "dp_layer_norms_batch", "dp_clip_factors",
                    "dp_clipped_sum_noise", "dp_clipped_sum_noise_batch",
                    "dp_audit_emit", "dp_audit_record_bytes", "dp_layer_norm_mode",
                    "dp_layer_path", "dp_set_noise_key", "dp_step_destroy", "dp_last_error",
                    "dp_status_string", "dp_kernel_launches", "dp_conv2d_dims",
                    "dp_conv2d_unfold",
                    "dp_debug_philox", "dp_debug_gaussian", "dp_debug_bounded_wait",
                    "dp_layer_sqnorms_noalloc", "dp_noise_adamw", "dp_partial_sqnorms",
                    "dp_clip_factors_from", "dp_noise_add_range"]


class DPError(RuntimeError):
    def __init__(self, status: int, msg: str):
        self.status = status
        self.name = STATUS_NAMES.get(status, str(status))
        super().__init__(f"{self.name}: {msg}")


class LibraryNotBuilt(ImportError):
    pass


class dp_conv2d(ctypes.Structure):
    _fields_ = [("H", ctypes.c_int32), ("W", ctypes.c_int32), ("C_in", ctypes.c_int32),
                ("kh", ctypes.c_int32), ("kw", ctypes.c_int32), ("stride_h", ctypes.c_int32),
                ("stride_w", ctypes.c_int32), ("pad_h", ctypes.c_int32), ("pad_w", ctypes.c_int32)]


class dp_layer(ctypes.Structure):
    _fields_ = [("d_in", ctypes.c_int64), ("d_out", ctypes.c_int64), ("T", ctypes.c_int32),
                ("kind", ctypes.c_int32)]


class dp_adamw(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("eps", ctypes.c_float), ("weight_decay", ctypes.c_float), ("t", ctypes.c_int64)]


class dp_config(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("T", ctypes.c_int32), ("n_layers", ctypes.c_int32),
                ("layers", ctypes.POINTER(dp_layer)), ("dtype", ctypes.c_int32),
                ("clip_C", ctypes.c_float), ("sigma", ctypes.c_float),
                ("out_scale", ctypes.c_float), ("seed", ctypes.c_uint64),
                ("step", ctypes.c_uint64), ("norm_mode", ctypes.c_int32),
                ("audit_capacity", ctypes.c_int32), ("convs", ctypes.POINTER(dp_conv2d)),
                ("param_base", ctypes.c_uint64)]


_LIB = None


def lib() -> ctypes.CDLL:
    """Load ``libdpstep.so`` (once).  Raises LibraryNotBuilt if it is missing."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if not os.path.exists(lib_path):
        raise LibraryNotBuilt(
            f"{lib_path} is missing: build it with `python -c 'import __graft_entry__ as g; "
            f"g.build()'` (nvcc, sm_103a)")
    L = ctypes.CDLL(lib_path)
    vp, i32, i64, u32, u64 = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32,
                              ctypes.c_uint64)
    sig = {
        "dp_step_init": ([ctypes.POINTER(vp), ctypes.POINTER(dp_config), vp], i32),
        "dp_layer_norms": ([vp, i32, vp, vp], i32),
        "dp_layer_norms_batch": ([vp, i32, vp, vp, vp], i32),
        "dp_clip_factors": ([vp, vp, vp], i32),
        "dp_clipped_sum_noise": ([vp, i32, vp, vp, vp, u32], i32),
        "dp_clipped_sum_noise_batch": ([vp, i32, vp, vp, vp, vp, u32], i32),
        "dp_audit_emit": ([vp, vp, i32, vp], i32),
        "dp_audit_record_bytes": ([i32], i64),
        "dp_layer_norm_mode": ([vp, i32, ctypes.POINTER(i32)], i32),
        "dp_layer_path": ([vp, i32, ctypes.POINTER(i32), ctypes.POINTER(i32)], i32),
        "dp_set_noise_key": ([vp, u64, u64], i32),
        "dp_step_destroy": ([vp], None),
        "dp_last_error": ([], ctypes.c_char_p),
        "dp_status_string": ([i32], ctypes.c_char_p),
        "dp_kernel_launches": ([ctypes.POINTER(i64)], i32),
        "dp_conv2d_dims": ([ctypes.POINTER(dp_conv2d), ctypes.POINTER(i32), ctypes.POINTER(i64)], i32),
        "dp_conv2d_unfold": ([ctypes.POINTER(dp_conv2d), i32, i32, vp, vp, vp], i32),
        "dp_debug_philox": ([u64, u64, u64, i64, vp, vp], i32),
        "dp_debug_gaussian": ([u64, u64, u64, i64, vp, vp], i32),
        "dp_debug_bounded_wait": ([vp, i64], i32),
        "dp_partial_sqnorms": ([vp, vp], i32),
        "dp_clip_factors_from": ([vp, vp, vp, vp], i32),
        "dp_noise_add_range": ([vp, u64, i64, vp], i32),
        "dp_layer_sqnorms_noalloc": ([vp, vp, i32, i32, i64, i64, i32, vp, vp], i32),
        "dp_noise_adamw": ([vp, i32, vp, vp, vp, vp, ctypes.POINTER(dp_adamw), u32], i32),
    }
    for name, (args, res) in sig.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = res
    _LIB = L
    return L


def _check(st: int):
    if st != DP_OK:
        raise DPError(st, lib().dp_last_error().decode())


def _ptr(x) -> Optional[int]:
    """Device pointer of a torch tensor (contiguity checked), an int, or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("tensor arguments must be contiguous")
        return x.data_ptr()
    raise TypeError(f"cannot take a pointer of {type(x)}")


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_config(layers: Sequence[Sequence[int]], B: int, T: int, dtype: str, C: float,
                sigma: float, out_scale: float = 1.0, seed: int = 0, step: int = 0,
                norm_mode: int = DP_NORM_AUTO, audit_capacity: int = 0,
                convs: Optional[Sequence[Optional[dp_conv2d]]] = None,
                param_base: int = 0) -> dp_config:
    """A layer is (d_in, d_out) or (d_in, d_out, T); T = 0 takes the config's
    T.  convs, when given, has one entry per layer: a dp_conv2d makes that
    layer a DP_LAYER_CONV2D layer (its A is then the NHWC input), None keeps
    it dense.  param_base: global parameter index of the first layer's first
    element (layers split over ranks)."""
    kinds = [DP_LAYER_CONV2D if convs is not None and convs[i] is not None else DP_LAYER_DENSE
             for i in range(len(layers))]
    arr = (dp_layer * len(layers))(*[dp_layer(int(ly[0]), int(ly[1]),
                                              int(ly[2]) if len(ly) > 2 else 0, kinds[i])
                                     for i, ly in enumerate(layers)])
    carr = None
    if convs is not None and any(k == DP_LAYER_CONV2D for k in kinds):
        carr = (dp_conv2d * len(layers))(*[cv if cv is not None else dp_conv2d() for cv in convs])
    cfg = dp_config(B=B, T=T, n_layers=len(layers), layers=arr,
                    dtype=DP_BF16 if dtype == "bf16" else DP_F32, clip_C=C, sigma=sigma,
                    out_scale=out_scale, seed=seed & (2 ** 64 - 1), step=step & (2 ** 64 - 1),
                    norm_mode=norm_mode, audit_capacity=audit_capacity,
                    convs=ctypes.cast(carr, ctypes.POINTER(dp_conv2d)) if carr is not None else None,
                    param_base=param_base & (2 ** 64 - 1))
    cfg._keep = (arr, carr)  # keep the arrays alive with the struct
    return cfg


def dp_step_init(cfg: dp_config, stream=None, ctx: Optional[int] = None) -> int:
    """Create a context (ctx None) or re-key an existing one; returns the handle."""
    h = ctypes.c_void_p(ctx)
    _check(lib().dp_step_init(ctypes.byref(h), ctypes.byref(cfg), _stream(stream)))
    return h.value


def dp_layer_norms(ctx: int, layer: int, A, D) -> None:
    _check(lib().dp_layer_norms(ctx, layer, _ptr(A), _ptr(D)))


def dp_layer_norms_batch(ctx: int, layers: Sequence[int], A_list, D_list) -> None:
    n = len(layers)
    ids = (ctypes.c_int32 * n)(*layers)
    a = (ctypes.c_void_p * n)(*[_ptr(x) for x in A_list])
    d = (ctypes.c_void_p * n)(*[_ptr(x) for x in D_list])
    _check(lib().dp_layer_norms_batch(ctx, n, ids, a, d))


def dp_clip_factors(ctx: int, sqnorm_out=None, clip_out=None) -> None:
    _check(lib().dp_clip_factors(ctx, _ptr(sqnorm_out), _ptr(clip_out)))


def dp_clipped_sum_noise(ctx: int, layer: int, A, D, out, flags: int = 0) -> None:
    _check(lib().dp_clipped_sum_noise(ctx, layer, _ptr(A), _ptr(D), _ptr(out), flags))


def dp_clipped_sum_noise_batch(ctx: int, layers: Sequence[int], A_list, D_list, outs,
                               flags: int = 0) -> None:
    n = len(layers)
    ids = (ctypes.c_int32 * n)(*layers)
    a = (ctypes.c_void_p * n)(*[_ptr(x) for x in A_list]) if A_list is not None else None
    d = (ctypes.c_void_p * n)(*[_ptr(x) for x in D_list]) if D_list is not None else None
    o = (ctypes.c_void_p * n)(*[_ptr(x) for x in outs])
    _check(lib().dp_clipped_sum_noise_batch(ctx, n, ids, a, d, o, flags))


def dp_audit_record_bytes(n_layers: int) -> int:
    return int(lib().dp_audit_record_bytes(n_layers))


def audit_dtype(n_layers: int) -> np.dtype:
    """numpy layout of one audit record (12 + 4 L bytes, see dp_step.h)."""
    return np.dtype([("example", "<i4"), ("total_sqnorm", "<f4"), ("clip_factor", "<f4"),
                     ("layer_sqnorm", "<f4", (n_layers,))])


def dp_audit_emit(ctx: int, idx: Iterable[int], n_layers: int) -> np.ndarray:
    """Records for the listed examples as a numpy structured array with fields
    example, total_sqnorm, clip_factor and layer_sqnorm [L]."""
    idx = np.ascontiguousarray(np.asarray(list(idx), dtype=np.int32))
    n = int(idx.size)
    recs = np.zeros(max(n, 1), dtype=audit_dtype(n_layers))
    st = lib().dp_audit_emit(ctx, idx.ctypes.data if n else None, n, recs.ctypes.data)
    _check(st)
    return recs[:n]


def dp_layer_norm_mode(ctx: int, layer: int) -> int:
    m = ctypes.c_int32(0)
    _check(lib().dp_layer_norm_mode(ctx, layer, ctypes.byref(m)))
    return m.value


def dp_layer_path(ctx: int, layer: int):
    """(norm path, sum path) of a layer: 1 = tensor cores, 0 = CUDA cores,
    norm path 2 = thin layer with stored per-example gradients."""
    a, b = ctypes.c_int32(0), ctypes.c_int32(0)
    _check(lib().dp_layer_path(ctx, layer, ctypes.byref(a), ctypes.byref(b)))
    return a.value, b.value


def dp_set_noise_key(ctx: int, seed: int, step: int) -> None:
    _check(lib().dp_set_noise_key(ctx, seed & (2 ** 64 - 1), step & (2 ** 64 - 1)))


def dp_step_destroy(ctx: Optional[int]) -> None:
    if ctx:
        lib().dp_step_destroy(ctx)


def dp_last_error() -> str:
    return lib().dp_last_error().decode()


def dp_kernel_launches() -> int:
    """Kernels the library has issued in this process (host-side count)."""
    n = ctypes.c_int64(0)
    _check(lib().dp_kernel_launches(ctypes.byref(n)))
    return n.value


def dp_debug_philox(seed: int, step: int, first_quad: int, n_quads: int, out, stream=None):
    _check(lib().dp_debug_philox(seed & (2 ** 64 - 1), step & (2 ** 64 - 1),
                                 first_quad & (2 ** 64 - 1), n_quads, _ptr(out), _stream(stream)))


def dp_debug_gaussian(seed: int, step: int, first_index: int, n: int, out, stream=None):
    _check(lib().dp_debug_gaussian(seed & (2 ** 64 - 1), step & (2 ** 64 - 1),
                                   first_index & (2 ** 64 - 1), n, _ptr(out), _stream(stream)))


def dp_partial_sqnorms(ctx: int, s_local) -> None:
    """This context's layers' share of every example's squared norm into
    ``s_local`` [B] (layers split over ranks; no clip factors yet)."""
    _check(lib().dp_partial_sqnorms(ctx, _ptr(s_local)))


def dp_clip_factors_from(ctx: int, s_total, sqnorm_out=None, clip_out=None) -> None:
    """Clip factors from squared norms summed over every rank's layers."""
    _check(lib().dp_clip_factors_from(ctx, _ptr(s_total), _ptr(sqnorm_out), _ptr(clip_out)))


def dp_noise_add_range(ctx: int, p_first: int, n: int, out) -> None:
    """out[e] += out_scale * sigma * C * z_{p_first + e} for e < n."""
    _check(lib().dp_noise_add_range(ctx, p_first & (2 ** 64 - 1), n, _ptr(out)))


def dp_debug_bounded_wait(ctx: int, limit_ns: int) -> int:
    """Run one bounded device wait that nothing satisfies; returns the status
    (DP_ERR_TIMEOUT when it gave up, as it should).  Test export."""
    return lib().dp_debug_bounded_wait(ctx, limit_ns)


def make_conv(H: int, W: int, C_in: int, kh: int, kw: int, stride=(1, 1), pad=(0, 0)) -> dp_conv2d:
    return dp_conv2d(H=H, W=W, C_in=C_in, kh=kh, kw=kw, stride_h=stride[0], stride_w=stride[1],
                     pad_h=pad[0], pad_w=pad[1])


def dp_conv2d_dims(conv: dp_conv2d):
    """(T, K) of a convolution: T = H_out * W_out, K = kh * kw * C_in."""
    T, K = ctypes.c_int32(0), ctypes.c_int64(0)
    _check(lib().dp_conv2d_dims(ctypes.byref(conv), ctypes.byref(T), ctypes.byref(K)))
    return T.value, K.value


def dp_conv2d_unfold(conv: dp_conv2d, B: int, dtype: str, x, a_out, stream=None) -> None:
    """Patch rows a_out [B][T][K] of the NHWC input x [B][H][W][C_in]."""
    _check(lib().dp_conv2d_unfold(ctypes.byref(conv), B, DP_BF16 if dtype == "bf16" else DP_F32,
                                  _ptr(x), _ptr(a_out), _stream(stream)))


def dp_layer_sqnorms_noalloc(A, D, B: int, T: int, d_in: int, d_out: int, dtype: str, out,
                             stream=None) -> None:
    """Per-example squared norms of one layer into ``out`` [B] without any
    allocation by the library (for callers that cannot allocate at the point
    of use; see include/dp_step.h)."""
    _check(lib().dp_layer_sqnorms_noalloc(_ptr(A), _ptr(D), B, T, d_in, d_out,
                                          DP_BF16 if dtype == "bf16" else DP_F32, _ptr(out),
                                          _stream(stream)))


def dp_noise_adamw(ctx: int, layer: int, grad, theta, m, v, lr: float, beta1: float,
                   beta2: float, eps: float, weight_decay: float, t: int, flags: int = 0) -> None:
    """Noisy gradient from the committed average, then AdamW on theta, m, v
    in place (see include/dp_step.h)."""
    hp = dp_adamw(lr=lr, beta1=beta1, beta2=beta2, eps=eps, weight_decay=weight_decay, t=t)
    _check(lib().dp_noise_adamw(ctx, layer, _ptr(grad), _ptr(theta), _ptr(m), _ptr(v),
                                ctypes.byref(hp), flags))


def run_step(ctx: int, A_list, D_list, outs, flags: int = 0) -> None:
    """The calls of one step in order (norms of every layer in one batched
    call, clip, clipped sum + noise of every layer); audit is left to the
    caller."""
    ids = list(range(len(A_list)))
    dp_layer_norms_batch(ctx, ids, A_list, D_list)
    dp_clip_factors(ctx)
    dp_clipped_sum_noise_batch(ctx, ids, A_list, D_list, outs, flags)
