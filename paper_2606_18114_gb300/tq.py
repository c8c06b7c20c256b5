"""ctypes binding of libtq (include/tq.h), with the same entry-point names.

Argument marshalling only: torch supplies device memory and the current CUDA
stream, every step of the computation runs in libtq's sm_103a kernels. There is
no fallback: if libtq.so is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

__all__ = [
    "TqError",
    "load",
    "quantize",
    "quantize_with_transpose",
    "quantize_batched",
    "quant_batch",
    "linear_fwd",
    "linear_bwd",
    "linear_bwd_noalloc",
    "codes_transpose",
    "linear_fwd_batched",
    "fwd_batch",
    "device_status",
    "adamw_requantize",
    "quantize_decoupled",
    "alpha_grad",
    "quantize_with_scales",
    "scale_grad",
    "adamw_requantize_with_scales",
    "adamw",
    "test_hooks",
    "AdamwHparams",
    "version",
    "OUT_F32",
    "OUT_BF16",
    "EXPORTS",
]

OUT_F32 = 0
OUT_BF16 = 1
IN_F16 = 0x100  # flag: fp16 activations (x, dy) instead of bf16
STATUS = {0: "TQ_OK", 1: "TQ_ERR_INVALID_ARG", 2: "TQ_ERR_UNSUPPORTED", 3: "TQ_ERR_CUDA",
          4: "TQ_ERR_TIMEOUT"}
# Every symbol include/tq.h declares.
EXPORTS = ("tq_quantize", "tq_quantize_with_transpose", "tq_quantize_batched", "tq_linear_fwd", "tq_linear_bwd",
           "tq_linear_bwd_noalloc", "tq_codes_transpose", "tq_linear_fwd_batched",
           "tq_adamw_requantize", "tq_quantize_decoupled", "tq_alpha_grad",
           "tq_quantize_with_scales", "tq_scale_grad", "tq_adamw_requantize_with_scales",
           "tq_adamw", "tq_device_status", "tq_test_hooks", "tq_last_error", "tq_version")

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libtq.so")
_lib = None


class TqError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status


class QuantDesc(ctypes.Structure):
    _fields_ = [
        ("w", ctypes.c_void_p),
        ("codes", ctypes.c_void_p),
        ("scales", ctypes.c_void_p),
        ("zero_counts", ctypes.c_void_p),
        ("n", ctypes.c_int64),
        ("k", ctypes.c_int64),
    ]


class AdamwHparams(ctypes.Structure):
    """tq_adamw_hparams of include/tq.h."""
    _fields_ = [
        ("lr", ctypes.c_double),
        ("beta1", ctypes.c_double),
        ("beta2", ctypes.c_double),
        ("eps", ctypes.c_double),
        ("weight_decay", ctypes.c_double),
        ("grad_scale", ctypes.c_double),
        ("step", ctypes.c_int64),
    ]


class FwdDesc(ctypes.Structure):
    _fields_ = [
        ("x", ctypes.c_void_p),
        ("codes", ctypes.c_void_p),
        ("scales", ctypes.c_void_p),
        ("y", ctypes.c_void_p),
        ("n", ctypes.c_int64),
        ("k", ctypes.c_int64),
        ("g", ctypes.c_int32),
        ("y_dtype", ctypes.c_int32),
    ]


def load(path: Optional[str] = None):
    """Load libtq.so (built by ``paper_2606_18114_gb300.build``) once."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or _LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"libtq.so not found at {p}; run paper_2606_18114_gb300.build.build()")
    lib = ctypes.CDLL(p)
    i64, i32, vp = ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p
    lib.tq_quantize.argtypes = [vp, i64, i64, i32, vp, vp, vp, vp]
    lib.tq_quantize_with_transpose.argtypes = [vp, i64, i64, i32, vp, vp, vp, vp, vp]
    lib.tq_quantize_batched.argtypes = [ctypes.POINTER(QuantDesc), i32, i32, vp]
    lib.tq_linear_fwd.argtypes = [vp, i64, i64, vp, vp, i64, i32, vp, i32, vp]
    lib.tq_linear_bwd.argtypes = [vp, vp, i64, i64, i64, vp, vp, vp, i32, vp, i32, vp, i32, vp]
    lib.tq_linear_bwd_noalloc.argtypes = [vp, vp, i64, i64, i64, vp, vp, i32, vp, i32, vp, i32,
                                          vp]
    lib.tq_codes_transpose.argtypes = [vp, i64, i64, vp, vp]
    lib.tq_linear_fwd_batched.argtypes = [ctypes.POINTER(FwdDesc), i32, i64, vp]
    lib.tq_device_status.argtypes = [vp]
    lib.tq_quantize_decoupled.argtypes = [vp, i64, i64, i32, vp, vp, vp, vp, vp]
    lib.tq_alpha_grad.argtypes = [vp, vp, i64, i64, i32, vp, vp]
    lib.tq_adamw_requantize.argtypes = [vp, vp, vp, vp, i64, i64, i32, ctypes.POINTER(AdamwHparams),
                                        vp, vp, vp, vp]
    lib.tq_quantize_with_scales.argtypes = [vp, i64, i64, i32, vp, vp, vp, vp]
    lib.tq_scale_grad.argtypes = [vp, vp, vp, vp, i64, i64, i32, vp, vp]
    lib.tq_adamw_requantize_with_scales.argtypes = [vp, vp, vp, vp, i64, i64, i32,
                                                    ctypes.POINTER(AdamwHparams), vp, vp, vp, vp]
    lib.tq_adamw.argtypes = [vp, vp, vp, vp, i64, ctypes.POINTER(AdamwHparams), vp]
    lib.tq_test_hooks.argtypes = [i64, ctypes.c_uint32]
    for name in ("tq_quantize", "tq_quantize_with_transpose", "tq_quantize_batched", "tq_linear_fwd", "tq_linear_bwd",
                 "tq_linear_bwd_noalloc", "tq_codes_transpose", "tq_linear_fwd_batched",
                 "tq_device_status", "tq_test_hooks"):
        getattr(lib, name).restype = ctypes.c_int
    lib.tq_last_error.restype = ctypes.c_char_p
    lib.tq_last_error.argtypes = []
    lib.tq_version.restype = ctypes.c_char_p
    lib.tq_version.argtypes = []
    _lib = lib
    return lib


def _check(status: int):
    if status != 0:
        raise TqError(status, load().tq_last_error().decode())


def _stream(stream=None) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors passed to libtq must be contiguous")
    return t.data_ptr() or None


def version() -> str:
    return load().tq_version().decode()


def device_status(stream=None) -> None:
    """Synchronise the stream and raise if a kernel's bounded wait ran out."""
    _check(load().tq_device_status(_stream(stream)))


def test_hooks(wait_limit_ns: int = 0, flags: int = 0) -> None:
    """Timeout-path testing only (include/tq.h, tq_test_hooks): the kernels' wait
    limit on this device (0: the default) and the withhold-one-arrival flags."""
    _check(load().tq_test_hooks(int(wait_limit_ns), int(flags)))


def quantize(w: torch.Tensor, g: int, out=None, stream=None):
    """§3.1 quantiser on a CUDA fp32 ``w [N, K]``.

    Returns ``(codes uint32-as-int32 [N, K/16], scales fp32 [N, K/g],
    zero_counts int32 [N, K/g])``. ``codes`` is an int32 tensor holding the
    uint32 bit patterns.
    """
    n, k = w.shape
    if out is None:
        codes = torch.empty((n, k // 16), dtype=torch.int32, device=w.device)
        scales = torch.empty((n, k // g), dtype=torch.float32, device=w.device)
        zeros = torch.empty((n, k // g), dtype=torch.int32, device=w.device)
    else:
        codes, scales, zeros = out
    _check(load().tq_quantize(_ptr(w), n, k, g, _ptr(codes), _ptr(scales), _ptr(zeros),
                              _stream(stream)))
    return codes, scales, zeros


def quantize_with_transpose(w: torch.Tensor, g: int, out=None, stream=None):
    """``quantize`` and ``codes_transpose`` of its codes in one launch.

    Returns ``(codes, scales, zero_counts, codes_t)``, ``codes_t`` int32
    ``[K, 4 * ceil(N / 64)]``; ``out`` may supply all four.
    """
    n, k = w.shape
    if out is None:
        codes = torch.empty((n, k // 16), dtype=torch.int32, device=w.device)
        scales = torch.empty((n, k // g), dtype=torch.float32, device=w.device)
        zeros = torch.empty((n, k // g), dtype=torch.int32, device=w.device)
        codes_t = torch.empty((k, 4 * ((n + 63) // 64)), dtype=torch.int32, device=w.device)
    else:
        codes, scales, zeros, codes_t = out
    _check(load().tq_quantize_with_transpose(_ptr(w), n, k, g, _ptr(codes), _ptr(scales),
                                             _ptr(zeros), _ptr(codes_t), _stream(stream)))
    return codes, scales, zeros, codes_t


def adamw_requantize(w: torch.Tensor, grad: torch.Tensor, m: torch.Tensor, v: torch.Tensor,
                     g: int, lr: float, step: int, beta1: float = 0.9, beta2: float = 0.95,
                     eps: float = 1e-8, weight_decay: float = 0.01, grad_scale: float = 1.0,
                     out=None, stream=None):
    """One AdamW step on the fp32 latent ``w`` (``m``, ``v`` its moments; all three
    updated in place) fused with the requantization of the new weights.

    Returns ``(codes, scales, zero_counts)`` as :func:`quantize` does."""
    n, k = w.shape
    if out is None:
        codes = torch.empty((n, k // 16), dtype=torch.int32, device=w.device)
        scales = torch.empty((n, k // g), dtype=torch.float32, device=w.device)
        zeros = torch.empty((n, k // g), dtype=torch.int32, device=w.device)
    else:
        codes, scales, zeros = out
    hp = AdamwHparams(lr, beta1, beta2, eps, weight_decay, grad_scale, step)
    _check(load().tq_adamw_requantize(_ptr(w), _ptr(grad), _ptr(m), _ptr(v), n, k, g,
                                      ctypes.byref(hp), _ptr(codes), _ptr(scales), _ptr(zeros),
                                      _stream(stream)))
    return codes, scales, zeros


def quantize_decoupled(w: torch.Tensor, g: int, row_factor: Optional[torch.Tensor] = None,
                       out=None, stream=None):
    """The decoupled quantizer: codes against ``row_factor[n] * absmean`` (``None``: 1).
    Returns ``(codes, absmean scales, zero_counts)`` like :func:`quantize`."""
    n, k = w.shape
    if out is None:
        codes = torch.empty((n, k // 16), dtype=torch.int32, device=w.device)
        scales = torch.empty((n, k // g), dtype=torch.float32, device=w.device)
        zeros = torch.empty((n, k // g), dtype=torch.int32, device=w.device)
    else:
        codes, scales, zeros = out
    rf = None if row_factor is None else _ptr(row_factor)
    _check(load().tq_quantize_decoupled(_ptr(w), n, k, g, rf, _ptr(codes), _ptr(scales),
                                        _ptr(zeros), _stream(stream)))
    return codes, scales, zeros


def alpha_grad(dw: torch.Tensor, codes: torch.Tensor, g: int, out: Optional[torch.Tensor] = None,
               stream=None) -> torch.Tensor:
    """Gradient of the decoupled quantizer's magnitude: per group, sum of dW * code."""
    n, k = dw.shape
    if out is None:
        out = torch.empty((n, k // g), dtype=torch.float32, device=dw.device)
    _check(load().tq_alpha_grad(_ptr(dw), _ptr(codes), n, k, g, _ptr(out), _stream(stream)))
    return out


def quantize_with_scales(w: torch.Tensor, g: int, scales: torch.Tensor, out=None, stream=None):
    """The learnable-scale variant's quantizer: codes against the given per-group
    ``scales`` (fp32 ``[N, K/g]``, any sign). Returns ``(codes, zero_counts)``."""
    n, k = w.shape
    if out is None:
        codes = torch.empty((n, k // 16), dtype=torch.int32, device=w.device)
        zeros = torch.empty((n, k // g), dtype=torch.int32, device=w.device)
    else:
        codes, zeros = out
    _check(load().tq_quantize_with_scales(_ptr(w), n, k, g, _ptr(scales), _ptr(codes),
                                          _ptr(zeros), _stream(stream)))
    return codes, zeros


def scale_grad(w: torch.Tensor, dw: torch.Tensor, codes: torch.Tensor, scales: torch.Tensor,
               g: int, out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Gradient of the learnable scales (include/tq.h, tq_scale_grad)."""
    n, k = w.shape
    if out is None:
        out = torch.empty((n, k // g), dtype=torch.float32, device=w.device)
    _check(load().tq_scale_grad(_ptr(w), _ptr(dw), _ptr(codes), _ptr(scales), n, k, g, _ptr(out),
                                _stream(stream)))
    return out


def adamw_requantize_with_scales(w: torch.Tensor, grad: torch.Tensor, m: torch.Tensor,
                                 v: torch.Tensor, g: int, scales: torch.Tensor, lr: float,
                                 step: int, beta1: float = 0.9, beta2: float = 0.95,
                                 eps: float = 1e-8, weight_decay: float = 0.01,
                                 grad_scale: float = 1.0, out=None, stream=None):
    """:func:`adamw_requantize` with the codes of the new ``w`` decided against the
    given ``scales``. Returns ``(codes, zero_counts)``."""
    n, k = w.shape
    if out is None:
        codes = torch.empty((n, k // 16), dtype=torch.int32, device=w.device)
        zeros = torch.empty((n, k // g), dtype=torch.int32, device=w.device)
    else:
        codes, zeros = out
    hp = AdamwHparams(lr, beta1, beta2, eps, weight_decay, grad_scale, step)
    _check(load().tq_adamw_requantize_with_scales(_ptr(w), _ptr(grad), _ptr(m), _ptr(v), n, k, g,
                                                  ctypes.byref(hp), _ptr(scales), _ptr(codes),
                                                  _ptr(zeros), _stream(stream)))
    return codes, zeros


def adamw(p: torch.Tensor, grad: torch.Tensor, m: torch.Tensor, v: torch.Tensor, lr: float,
          step: int, beta1: float = 0.9, beta2: float = 0.95, eps: float = 1e-8,
          weight_decay: float = 0.01, grad_scale: float = 1.0, stream=None) -> None:
    """One AdamW step on a flat fp32 array ``p`` (numel a multiple of 16); ``p``, ``m``
    and ``v`` are updated in place."""
    hp = AdamwHparams(lr, beta1, beta2, eps, weight_decay, grad_scale, step)
    _check(load().tq_adamw(_ptr(p), _ptr(grad), _ptr(m), _ptr(v), p.numel(), ctypes.byref(hp),
                           _stream(stream)))


def quant_batch(items: Sequence[tuple]):
    """Descriptor array for ``quantize_batched`` (build once, call many times).

    ``items``: tuples ``(w, codes, scales, zero_counts)`` of allocated tensors
    (outputs written in place). The tensors must outlive the array's use.
    """
    arr = (QuantDesc * len(items))()
    for i, (w, codes, scales, zeros) in enumerate(items):
        arr[i] = QuantDesc(_ptr(w), _ptr(codes), _ptr(scales), _ptr(zeros), w.shape[0],
                           w.shape[1])
    return arr


def quantize_batched(items, g: int, stream=None) -> None:
    """``quantize`` of many fp32 matrices with one group size in one launch
    (``items`` as for ``quant_batch``, or an array that it returned)."""
    arr = items if isinstance(items, ctypes.Array) else quant_batch(items)
    _check(load().tq_quantize_batched(arr, len(arr), g, _stream(stream)))


def _out_code(dtype) -> int:
    if dtype == torch.float32:
        return OUT_F32
    if dtype == torch.bfloat16:
        return OUT_BF16
    raise ValueError(f"unsupported output dtype {dtype}")


def _in_flag(act: Optional[torch.Tensor]) -> int:
    """IN_F16 for fp16 activations, 0 for bf16 (the activation type rides on the
    output-type word of the C calls)."""
    if act is None or act.dtype == torch.bfloat16:
        return 0
    if act.dtype == torch.float16:
        return IN_F16
    raise ValueError(f"unsupported activation dtype {act.dtype}")


def linear_fwd(x: torch.Tensor, codes: torch.Tensor, scales: torch.Tensor, g: int,
               out_dtype=torch.float32, y: Optional[torch.Tensor] = None, stream=None):
    """W1.58A16 forward ``y = x W^T`` for bf16 (or fp16) ``x [M, K]``; returns ``y [M, N]``."""
    m, k = x.shape
    n = codes.shape[0]
    if y is None:
        y = torch.empty((m, n), dtype=out_dtype, device=x.device)
    _check(load().tq_linear_fwd(_ptr(x), m, k, _ptr(codes), _ptr(scales), n, g, _ptr(y),
                                _out_code(y.dtype) | _in_flag(x), _stream(stream)))
    return y


def codes_transpose(codes: torch.Tensor, k: int, out: Optional[torch.Tensor] = None, stream=None):
    """Packed codes of W^T (uint32 bit patterns in int32) ``[K, 4 * ceil(N / 64)]``."""
    n = codes.shape[0]
    if out is None:
        out = torch.empty((k, 4 * ((n + 63) // 64)), dtype=torch.int32, device=codes.device)
    _check(load().tq_codes_transpose(_ptr(codes), n, k, _ptr(out), _stream(stream)))
    return out


def linear_bwd(dy: torch.Tensor, x: Optional[torch.Tensor], codes: torch.Tensor,
               scales: torch.Tensor, k: int, g: int, want_dx: bool = True, want_dw: bool = True,
               dx_dtype=torch.float32, dx: Optional[torch.Tensor] = None,
               dw: Optional[torch.Tensor] = None, accumulate_dw: bool = False,
               codes_t: Optional[torch.Tensor] = None, stream=None):
    """STE backward; returns ``(dx [M, K] or None, dw fp32 [N, K] or None)``.

    ``codes_t`` (from ``codes_transpose``) selects the faster dX path."""
    m, n = dy.shape
    if want_dx and dx is None:
        dx = torch.empty((m, k), dtype=dx_dtype, device=dy.device)
    if want_dw and dw is None:
        dw = torch.empty((n, k), dtype=torch.float32, device=dy.device)
    if not want_dx:
        dx = None
    if not want_dw:
        dw = None
    _check(load().tq_linear_bwd(_ptr(dy), _ptr(x), m, n, k, _ptr(codes), _ptr(codes_t),
                                _ptr(scales), g,
                                _ptr(dx), (_out_code(dx.dtype) if dx is not None else OUT_F32)
                                | _in_flag(dy),
                                _ptr(dw), int(accumulate_dw), _stream(stream)))
    return dx, dw


def linear_bwd_noalloc(dy: torch.Tensor, x: Optional[torch.Tensor], codes: torch.Tensor,
                       scales: torch.Tensor, k: int, g: int, want_dx: bool = True,
                       want_dw: bool = True, dx_dtype=torch.float32,
                       dx: Optional[torch.Tensor] = None, dw: Optional[torch.Tensor] = None,
                       accumulate_dw: bool = False, stream=None):
    """``linear_bwd`` on the transposed-codes dX path with the library's own
    scratch for the transposed codes (nothing allocated for them)."""
    m, n = dy.shape
    if want_dx and dx is None:
        dx = torch.empty((m, k), dtype=dx_dtype, device=dy.device)
    if want_dw and dw is None:
        dw = torch.empty((n, k), dtype=torch.float32, device=dy.device)
    if not want_dx:
        dx = None
    if not want_dw:
        dw = None
    _check(load().tq_linear_bwd_noalloc(_ptr(dy), _ptr(x), m, n, k, _ptr(codes), _ptr(scales), g,
                                        _ptr(dx), (_out_code(dx.dtype) if dx is not None else OUT_F32)
                                        | _in_flag(dy),
                                        _ptr(dw), int(accumulate_dw), _stream(stream)))
    return dx, dw


def fwd_batch(items: Sequence[dict]):
    """Descriptor array for ``linear_fwd_batched`` (build once, call many times).

    ``items``: dicts with ``x, codes, scales, y, g`` (tensors already allocated,
    ``y`` written in place). The tensors must outlive the array's use.
    """
    arr = (FwdDesc * len(items))()
    for i, it in enumerate(items):
        codes = it["codes"]
        arr[i] = FwdDesc(_ptr(it["x"]), _ptr(codes), _ptr(it["scales"]), _ptr(it["y"]),
                         codes.shape[0], codes.shape[1] * 16, it["g"],
                         _out_code(it["y"].dtype) | _in_flag(it["x"]))
    return arr


def linear_fwd_batched(items, m: int, stream=None) -> None:
    """Decode forward over many matrices in one call (``items`` as for ``fwd_batch``,
    or an array that ``fwd_batch`` returned)."""
    arr = items if isinstance(items, ctypes.Array) else fwd_batch(items)
    _check(load().tq_linear_fwd_batched(arr, len(arr), m, _stream(stream)))
