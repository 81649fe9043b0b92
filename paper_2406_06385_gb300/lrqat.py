"""Python binding of liblrqat (the C ABI in include/lrqat.h).

Argument marshalling only: every function here forwards torch tensor pointers
and the current CUDA stream to the C entry point of the same name and raises
``LrqatError`` on a non-OK status.  All computation happens in the library's
CUDA kernels; there is no fallback when the library is missing.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "_lib", "liblrqat.so")

PHI_QFIXED = 0
PHI_INT_PACKED = 1
PHI_BF16 = 2
PHI_FP16 = 3
PHI_FP8_E4M3 = 4
PHI_FP8_E5M2 = 5

STATUS = {0: "LRQAT_OK", -1: "LRQAT_ERR_INVALID_ARG", -2: "LRQAT_ERR_UNSUPPORTED", -3: "LRQAT_ERR_ALIGNMENT",
          -4: "LRQAT_ERR_WORKSPACE", -5: "LRQAT_ERR_CUDA", -6: "LRQAT_ERR_TIMEOUT"}


class LrqatError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status


class Layer(ctypes.Structure):
    """Mirror of the C struct lrqat_layer."""
    _fields_ = [("m", ctypes.c_int64), ("k", ctypes.c_int64), ("r", ctypes.c_int32), ("alpha", ctypes.c_float),
                ("bits", ctypes.c_int32), ("group_size", ctypes.c_int32), ("phi_format", ctypes.c_int32),
                ("act_bits", ctypes.c_int32), ("zero", ctypes.c_void_p), ("act_per_token", ctypes.c_int32),
                ("u_bf16", ctypes.c_int32)]

    @classmethod
    def from_spec(cls, spec, zero: int = 0) -> "Layer":
        """`zero`: device address of the zero offsets (asymmetric weights), 0 for none."""
        return cls(spec.m, spec.k, spec.r, spec.alpha, spec.bits, spec.group_size, spec.phi_format, spec.act_bits,
                   zero or None, int(getattr(spec, "act_per_token", False)), int(getattr(spec, "u_bf16", False)))


class AdamW(ctypes.Structure):
    """Mirror of lrqat_adamw (App. B, Table B1 defaults)."""
    _fields_ = [("lr_ab", ctypes.c_float), ("lr_s", ctypes.c_float), ("beta1", ctypes.c_float),
                ("beta2", ctypes.c_float), ("eps", ctypes.c_float), ("weight_decay_ab", ctypes.c_float),
                ("weight_decay_s", ctypes.c_float), ("max_grad_norm", ctypes.c_float), ("step", ctypes.c_int32)]

    @classmethod
    def make(cls, lr_ab: float, lr_s: float, step: int, beta1: float = 0.9, beta2: float = 0.95, eps: float = 1e-8,
             weight_decay_ab: float = 0.0, weight_decay_s: float = 0.0, max_grad_norm: float = 1.0) -> "AdamW":
        return cls(lr_ab, lr_s, beta1, beta2, eps, weight_decay_ab, weight_decay_s, max_grad_norm, step)


class AdamWState(ctypes.Structure):
    """Mirror of lrqat_adamw_state: device addresses of the fp32 masters and moments."""
    _fields_ = [(n, ctypes.c_void_p) for n in ("A32", "B32", "mA", "vA", "mB", "vB", "ms", "vs")]


_lib = None


def lib() -> ctypes.CDLL:
    """Loads liblrqat.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -m paper_2406_06385_gb300.build`")
        L = ctypes.CDLL(LIB_PATH)
        vp, i64, sz, ip = ctypes.c_void_p, ctypes.c_int64, ctypes.c_size_t, ctypes.c_int
        lp = ctypes.POINTER(Layer)
        L.lrqat_last_error.restype = ctypes.c_char_p
        L.lrqat_last_error.argtypes = []
        sigs = {
            "lrqat_range_minmax": [lp, vp, vp, vp],
            "lrqat_downcast": [lp, vp, vp, vp, vp],
            "lrqat_linear_fwd": [lp, i64, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp],
            "lrqat_linear_fwd_noalloc": [lp, i64, vp, vp, vp, vp, vp, vp, vp, vp],
            "lrqat_linear_bwd": [lp, i64, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, ip, vp, sz, vp],
            "lrqat_linear_fwd_quantized": [lp, i64, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp],
            "lrqat_linear_bwd_quantized": [lp, i64, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, ip, vp, sz, vp],
            "lrqat_merge": [lp, vp, vp, vp, vp, vp],
            "lrqat_get_device_status": [vp],
            "lrqat_grad_sqnorm": [lp, vp, vp, vp, vp, vp],
            "lrqat_range_lp": [lp, vp, ctypes.c_float, ctypes.c_int32, vp, vp],
            "lrqat_act_quant": [lp, ctypes.c_int64, vp, vp, vp, vp, vp],
            "lrqat_adamw_step": [lp, ctypes.POINTER(AdamW), vp, vp, vp, vp, ctypes.POINTER(AdamWState), vp, vp, vp,
                                 vp],
        }
        for name, args in sigs.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        for name in ("lrqat_get_gemm_variant", "lrqat_get_dw_schedule", "lrqat_get_lowrank_path"):
            getattr(L, name).argtypes = []
            getattr(L, name).restype = ctypes.c_int
        L.lrqat_set_gemm_variant.argtypes = [ip]
        L.lrqat_set_gemm_variant.restype = ctypes.c_int
        L.lrqat_set_dw_schedule.argtypes = [ip]
        L.lrqat_set_dw_schedule.restype = ctypes.c_int
        L.lrqat_set_lowrank_path.argtypes = [ip]
        L.lrqat_set_lowrank_path.restype = ctypes.c_int
        L.lrqat_trace_enable.argtypes = [ip]
        L.lrqat_trace_enable.restype = ctypes.c_int
        L.lrqat_trace_read.argtypes = [ip, ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(ctypes.c_int64),
                                       ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int)]
        L.lrqat_trace_read.restype = ctypes.c_int
        for name in ("lrqat_fwd_workspace_bytes", "lrqat_bwd_workspace_bytes"):
            fn = getattr(L, name)
            fn.argtypes = [lp, i64]
            fn.restype = ctypes.c_size_t
        _lib = L
    return _lib


def _check(status: int) -> None:
    if status != 0:
        raise LrqatError(status, lib().lrqat_last_error().decode())


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is not None:
        return stream if isinstance(stream, int) else stream.cuda_stream
    import torch
    return torch.cuda.current_stream().cuda_stream


def last_error() -> str:
    return lib().lrqat_last_error().decode()


def range_minmax(layer: Layer, W0, s0, stream=None) -> None:
    _check(lib().lrqat_range_minmax(ctypes.byref(layer), _ptr(W0), _ptr(s0), _stream(stream)))


def downcast(layer: Layer, W0, s0, Phi0, stream=None) -> None:
    _check(lib().lrqat_downcast(ctypes.byref(layer), _ptr(W0), _ptr(s0), _ptr(Phi0), _stream(stream)))


def fwd_workspace_bytes(layer: Layer, T: int) -> int:
    return int(lib().lrqat_fwd_workspace_bytes(ctypes.byref(layer), T))


def bwd_workspace_bytes(layer: Layer, T: int) -> int:
    return int(lib().lrqat_bwd_workspace_bytes(ctypes.byref(layer), T))


def linear_fwd(layer: Layer, T: int, X, Phi0, s, A, B, s_x, Y, workspace, stream=None) -> None:
    nbytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().lrqat_linear_fwd(ctypes.byref(layer), T, _ptr(X), _ptr(Phi0), _ptr(s), _ptr(A), _ptr(B), _ptr(s_x),
                                  _ptr(Y), _ptr(workspace), nbytes, _stream(stream)))


def linear_fwd_noalloc(layer: Layer, T: int, X, Phi0, s, A, B, s_x, Y, stream=None) -> None:
    """Forward that takes its scratch from the library's fixed device array (no workspace argument)."""
    _check(lib().lrqat_linear_fwd_noalloc(ctypes.byref(layer), T, _ptr(X), _ptr(Phi0), _ptr(s), _ptr(A), _ptr(B),
                                          _ptr(s_x), _ptr(Y), _stream(stream)))


def linear_bwd(layer: Layer, T: int, dY, X, Phi0, s, A, B, s_x, dX, dA, dB, ds, accumulate: bool, workspace,
               stream=None) -> None:
    nbytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().lrqat_linear_bwd(ctypes.byref(layer), T, _ptr(dY), _ptr(X), _ptr(Phi0), _ptr(s), _ptr(A), _ptr(B),
                                  _ptr(s_x), _ptr(dX), _ptr(dA), _ptr(dB), _ptr(ds), 1 if accumulate else 0,
                                  _ptr(workspace), nbytes, _stream(stream)))


def linear_fwd_quantized(layer: Layer, T: int, X_q, Phi0, s, A, B, s_x, Y, workspace, stream=None) -> None:
    """Forward on the output of act_quant (per tensor: codes; per token: X_hat)."""
    nbytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().lrqat_linear_fwd_quantized(ctypes.byref(layer), T, _ptr(X_q), _ptr(Phi0), _ptr(s), _ptr(A), _ptr(B),
                                            _ptr(s_x), _ptr(Y), _ptr(workspace), nbytes, _stream(stream)))


def linear_bwd_quantized(layer: Layer, T: int, dY, X_q, mask, Phi0, s, A, B, s_x, dX, dA, dB, ds, accumulate: bool,
                         workspace, stream=None) -> None:
    """Backward on the output of act_quant and its clip mask (per tensor; None per token)."""
    nbytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().lrqat_linear_bwd_quantized(ctypes.byref(layer), T, _ptr(dY), _ptr(X_q), _ptr(mask), _ptr(Phi0),
                                            _ptr(s), _ptr(A), _ptr(B), _ptr(s_x), _ptr(dX), _ptr(dA), _ptr(dB),
                                            _ptr(ds), 1 if accumulate else 0, _ptr(workspace), nbytes,
                                            _stream(stream)))


def merge(layer: Layer, Phi0, A, B, W_Z, stream=None) -> None:
    _check(lib().lrqat_merge(ctypes.byref(layer), _ptr(Phi0), _ptr(A), _ptr(B), _ptr(W_Z), _stream(stream)))


def act_quant(layer: Layer, T: int, X, s_x, X_out, mask=None, stream=None) -> None:
    """Activation quantizer on its own (per tensor: codes + optional mask; per token: X_hat)."""
    _check(lib().lrqat_act_quant(ctypes.byref(layer), T, _ptr(X), _ptr(s_x), _ptr(X_out), _ptr(mask),
                                 _stream(stream)))


def range_lp(layer: Layer, W0, s0, p_norm: float, n_candidates: int = 100, stream=None) -> None:
    """L^p range setting over n_candidates scaled min-max scales (symmetric grids)."""
    _check(lib().lrqat_range_lp(ctypes.byref(layer), _ptr(W0), p_norm, n_candidates, _ptr(s0), _stream(stream)))


def grad_sqnorm(layer: Layer, dA, dB, ds, sqnorm, stream=None) -> None:
    """Adds the squared L2 norm of the layer's gradients to the device scalar sqnorm."""
    _check(lib().lrqat_grad_sqnorm(ctypes.byref(layer), _ptr(dA), _ptr(dB), _ptr(ds), _ptr(sqnorm), _stream(stream)))


def adamw_step(layer: Layer, opt: AdamW, sqnorm, dA, dB, ds, state: dict, s, A, B, stream=None) -> None:
    """One clipped AdamW step; `state` maps A32, B32, mA, vA, mB, vB, ms, vs to device tensors."""
    st = AdamWState(*[_ptr(state[n]) for n, _ in AdamWState._fields_])
    _check(lib().lrqat_adamw_step(ctypes.byref(layer), ctypes.byref(opt), _ptr(sqnorm), _ptr(dA), _ptr(dB), _ptr(ds),
                                  ctypes.byref(st), _ptr(s), _ptr(A), _ptr(B), _stream(stream)))


def get_device_status(stream=None) -> None:
    _check(lib().lrqat_get_device_status(_stream(stream)))


DW_SCHEDULES = {"auto": 0, "split": 1, "tail": 2}


def set_dw_schedule(schedule: str) -> None:
    """Process-wide schedule of the weight-gradient work: "auto", "split" or "tail"."""
    _check(lib().lrqat_set_dw_schedule(DW_SCHEDULES[schedule]))


GEMM_VARIANTS = {"auto": 0, "single": 1, "pair": 2}


def set_gemm_variant(variant: str) -> None:
    """Process-wide kernels of the forward, dX and dW GEMMs: "auto" (CTA pairs where they were
    measured faster, the default), "single" (one SM per tile) or "pair" (CTA pairs wherever
    the shapes allow)."""
    _check(lib().lrqat_set_gemm_variant(GEMM_VARIANTS[variant]))


def gemm_variant() -> str:
    return {v: k for k, v in GEMM_VARIANTS.items()}[lib().lrqat_get_gemm_variant()]


def dw_schedule() -> str:
    return {v: k for k, v in DW_SCHEDULES.items()}[lib().lrqat_get_dw_schedule()]


LOWRANK_PATHS = {"auto": 0, "tile": 1, "codes": 2}


def set_lowrank_path(path: str) -> None:
    """Process-wide source of the low-rank term in the forward and dX GEMMs: "auto" (the
    default), "tile" (computed inside each GEMM stage; ranks up to 64) or "codes" (one pass per
    call writes the codes of every weight, which the GEMMs read)."""
    _check(lib().lrqat_set_lowrank_path(LOWRANK_PATHS[path]))


def lowrank_path() -> str:
    return {v: k for k, v in LOWRANK_PATHS.items()}[lib().lrqat_get_lowrank_path()]


def trace_enable(enable: bool = True) -> None:
    _check(lib().lrqat_trace_enable(1 if enable else 0))


def trace_read(max_entries: int = 32):
    """Per-kernel {name: (launches, total_ms)} recorded since trace_enable(True)."""
    names = (ctypes.c_char_p * max_entries)()
    launches = (ctypes.c_int64 * max_entries)()
    ms = (ctypes.c_double * max_entries)()
    count = ctypes.c_int(0)
    _check(lib().lrqat_trace_read(max_entries, names, launches, ms, ctypes.byref(count)))
    return {names[i].decode(): (int(launches[i]), float(ms[i])) for i in range(min(count.value, max_entries))}
