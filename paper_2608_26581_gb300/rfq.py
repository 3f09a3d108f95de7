"""ctypes binding of ``librfq.so`` (declared in ``include/rfq.h``).

Argument marshalling only: every step of the RFQ path runs in the library's
CUDA kernels.  PyTorch provides device memory and streams.  There is no CPU
fallback: if the library is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
# the library (RFQ_LIBRARY names another build of it, e.g. librfq_debug.so)
LIB_PATH = os.environ.get("RFQ_LIBRARY") or os.path.join(_HERE, "librfq.so")

RFQ_OK = 0
RFQ_FMT_MXFP4, RFQ_FMT_HIF4, RFQ_FMT_BF16, RFQ_FMT_MXFP8 = 0, 1, 2, 3
RFQ_SCALE_ROWMAJOR, RFQ_SCALE_MMA = 0, 1
RFQ_FALLBACK_NONE, RFQ_FALLBACK_ALL, RFQ_FALLBACK_AMAX = 0, 1, 2
RFQ_OUT_F32, RFQ_OUT_BF16 = 0, 1
(RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT, RFQ_ERR_UNSUPPORTED, RFQ_ERR_CUDA, RFQ_ERR_TIMEOUT,
 RFQ_ERR_DEVICE, RFQ_ERR_NONFINITE) = range(1, 9)
STATUS_NAMES = {0: "RFQ_OK", 1: "RFQ_ERR_INVALID_ARG", 2: "RFQ_ERR_SHAPE", 3: "RFQ_ERR_ALIGNMENT",
                4: "RFQ_ERR_UNSUPPORTED", 5: "RFQ_ERR_CUDA", 6: "RFQ_ERR_TIMEOUT", 7: "RFQ_ERR_DEVICE",
                8: "RFQ_ERR_NONFINITE"}

EXPORTED = ("rfq_status_string", "rfq_qtensor_bytes", "rfq_quantize_weight", "rfq_quantize_act",
            "rfq_linear_workspace_bytes", "rfq_linear", "rfq_workspace_status", "rfq_dequant",
            "rfq_linear_noalloc", "rfq_linear_fused", "rfq_convert", "rfq_linear_grouped", "rfq_check_finite",
            "rfq_quantize_act_expand", "rfq_fp4_mma_peak", "rfq_linear_fused_workspace_bytes",
            "rfq_linear_profile", "rfq_debug_bounds", "rfq_linear_mixed", "rfq_linear_host")


class RFQError(RuntimeError):
    def __init__(self, status: int, call: str):
        self.status = status
        super().__init__(f"{call}: {STATUS_NAMES.get(status, status)}")


class _QT(ctypes.Structure):
    _fields_ = [("fmt", ctypes.c_int32), ("scale_layout", ctypes.c_int32), ("rows", ctypes.c_int64),
                ("k", ctypes.c_int64), ("codes", ctypes.c_void_p), ("scales", ctypes.c_void_p)]


class _FB(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int32), ("tau", ctypes.c_float), ("p_s", ctypes.c_int32),
                ("r_s", ctypes.c_int32)]


_lib = None


def load_library(path: str = LIB_PATH):
    """Load librfq.so; raises if it has not been built (no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build it with paper_2608_26581_gb300._build.build()")
        lib = ctypes.CDLL(path)
        P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
        QTP = ctypes.POINTER(_QT)
        lib.rfq_status_string.restype = ctypes.c_char_p
        lib.rfq_status_string.argtypes = [I32]
        lib.rfq_qtensor_bytes.restype = I32
        lib.rfq_qtensor_bytes.argtypes = [I32, I32, I64, I64, ctypes.POINTER(SZ), ctypes.POINTER(SZ)]
        lib.rfq_quantize_weight.restype = I32
        lib.rfq_quantize_weight.argtypes = [P, I64, I64, QTP, P]
        lib.rfq_quantize_act.restype = I32
        lib.rfq_quantize_act.argtypes = [P, I64, I64, ctypes.POINTER(_FB), QTP, QTP, P, P]
        lib.rfq_quantize_act_expand.restype = I32
        lib.rfq_quantize_act_expand.argtypes = [P, I64, I64, ctypes.POINTER(_FB), QTP, QTP, P, QTP, QTP, P]
        lib.rfq_linear_workspace_bytes.restype = SZ
        lib.rfq_linear_workspace_bytes.argtypes = []
        lib.rfq_linear.restype = I32
        lib.rfq_linear.argtypes = [QTP, QTP, P, I32, QTP, P, I32, P, P]
        lib.rfq_workspace_status.restype = I32
        lib.rfq_workspace_status.argtypes = [P, I32, P]
        lib.rfq_dequant.restype = I32
        lib.rfq_dequant.argtypes = [QTP, P, I32, P]
        lib.rfq_linear_noalloc.restype = I32
        lib.rfq_linear_noalloc.argtypes = [QTP, QTP, P, I32, QTP, P, I32, P]
        lib.rfq_linear_fused.restype = I32
        lib.rfq_linear_fused.argtypes = [P, I64, I64, QTP, ctypes.POINTER(_FB), P, I32, P, P]
        lib.rfq_convert.restype = I32
        lib.rfq_convert.argtypes = [QTP, QTP, P]
        lib.rfq_check_finite.restype = I32
        lib.rfq_check_finite.argtypes = [P, I64, I64, P, P]
        lib.rfq_linear_grouped.restype = I32
        lib.rfq_linear_grouped.argtypes = [QTP, QTP, P, I32, P, I32, QTP, I64, P, I32, P, P]
        lib.rfq_linear_fused_workspace_bytes.restype = SZ
        lib.rfq_linear_fused_workspace_bytes.argtypes = [I64, I64, ctypes.POINTER(_FB)]
        lib.rfq_linear_mixed.restype = I32
        lib.rfq_linear_mixed.argtypes = [QTP, QTP, P, I32, QTP, P, I32, P, P]
        lib.rfq_linear_host.restype = I32
        lib.rfq_linear_host.argtypes = [P, I64, I64, ctypes.POINTER(_FB), QTP, P, I32, I64, P, QTP, QTP, P, P, P, P]
        lib.rfq_debug_bounds.restype = I32
        lib.rfq_debug_bounds.argtypes = [ctypes.POINTER(I32), I32]
        lib.rfq_linear_profile.restype = I32
        lib.rfq_linear_profile.argtypes = [QTP, QTP, QTP, P, I32, P, P]
        lib.rfq_fp4_mma_peak.restype = I32
        lib.rfq_fp4_mma_peak.argtypes = [I32, I64, P, ctypes.POINTER(ctypes.c_double), P]
        _lib = lib
    return _lib


def _check(status: int, call: str):
    if status != RFQ_OK:
        raise RFQError(status, call)


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


@dataclass
class QTensor:
    """A quantized rows x k matrix: device ``codes`` and ``scales`` tensors."""
    fmt: int
    scale_layout: int
    rows: int
    k: int
    codes: torch.Tensor
    scales: torch.Tensor

    def c(self) -> _QT:
        return _QT(self.fmt, self.scale_layout, self.rows, self.k,
                   self.codes.data_ptr(), None if self.scales is None else self.scales.data_ptr())


def rfq_status_string(status: int) -> str:
    return load_library().rfq_status_string(status).decode()


def rfq_qtensor_bytes(fmt: int, scale_layout: int, rows: int, k: int):
    cb, sb = ctypes.c_size_t(), ctypes.c_size_t()
    _check(load_library().rfq_qtensor_bytes(fmt, scale_layout, rows, k, ctypes.byref(cb), ctypes.byref(sb)),
           "rfq_qtensor_bytes")
    return cb.value, sb.value


def empty_qtensor(fmt: int, scale_layout: int, rows: int, k: int, device="cuda") -> QTensor:
    """Allocate (with torch) the buffers of a quantized matrix."""
    cb, sb = rfq_qtensor_bytes(fmt, scale_layout, rows, k)
    return QTensor(fmt, scale_layout, rows, k,
                   torch.empty(max(cb, 16), dtype=torch.uint8, device=device),
                   torch.empty(max(sb, 16), dtype=torch.uint8, device=device))


def empty_bf16_operand(rows: int, k: int, device="cuda") -> QTensor:
    return bf16_operand(torch.empty(rows, k, dtype=torch.bfloat16, device=device))


def rfq_quantize_weight(w: torch.Tensor, out: QTensor, stream=None):
    K, N = w.shape
    qt = out.c()
    _check(load_library().rfq_quantize_weight(_ptr(w), K, N, ctypes.byref(qt), _stream(stream)),
           "rfq_quantize_weight")


def rfq_quantize_act(x: torch.Tensor, xq: QTensor, xr: QTensor | None, phi: torch.Tensor | None = None,
                     mode: int = RFQ_FALLBACK_ALL, tau: float = 0.0, p_s: int = 128, r_s: int = 256,
                     stream=None):
    M, K = x.shape
    fb = _FB(mode, tau, p_s, r_s)
    q = xq.c()
    r = xr.c() if xr is not None else None
    _check(load_library().rfq_quantize_act(_ptr(x), M, K, ctypes.byref(fb), ctypes.byref(q),
                                           ctypes.byref(r) if r is not None else None, _ptr(phi),
                                           _stream(stream)), "rfq_quantize_act")


def rfq_quantize_act_expand(x: torch.Tensor, xq: QTensor, xr: QTensor | None, xq_op: QTensor,
                            xr_op: QTensor | None, phi: torch.Tensor | None = None, mode: int = RFQ_FALLBACK_ALL,
                            tau: float = 0.0, p_s: int = 128, r_s: int = 256, stream=None):
    """Activation quantization that also writes X~ (and X^) in the form the
    GEMM multiplies, in the same pass: the exact bf16 values for HiF4 (xq_op,
    xr_op), X~ re-encoded as MXFP8 for an MXFP4 main pathway under an MXFP8
    residual (xq_op; xr_op None)."""
    M, K = x.shape
    fb = _FB(mode, tau, p_s, r_s)
    q, qo = xq.c(), xq_op.c()
    r = xr.c() if xr is not None else None
    ro = xr_op.c() if xr_op is not None else None
    _check(load_library().rfq_quantize_act_expand(
        _ptr(x), M, K, ctypes.byref(fb), ctypes.byref(q), ctypes.byref(r) if r is not None else None, _ptr(phi),
        ctypes.byref(qo), ctypes.byref(ro) if ro is not None else None, _stream(stream)),
        "rfq_quantize_act_expand")


def rfq_linear_workspace_bytes() -> int:
    return load_library().rfq_linear_workspace_bytes()


def rfq_linear(xq: QTensor, xr: QTensor | None, phi: torch.Tensor | None, phi_r_s: int, wq: QTensor,
               y: torch.Tensor, out_dtype: int, workspace: torch.Tensor, stream=None):
    q, w = xq.c(), wq.c()
    r = xr.c() if xr is not None else None
    _check(load_library().rfq_linear(ctypes.byref(q), ctypes.byref(r) if r is not None else None, _ptr(phi),
                                     phi_r_s, ctypes.byref(w), _ptr(y), out_dtype, _ptr(workspace),
                                     _stream(stream)), "rfq_linear")


def rfq_linear_mixed(xq: QTensor, xr: QTensor, phi: torch.Tensor | None, phi_r_s: int, wq: QTensor,
                     y: torch.Tensor, out_dtype: int, workspace: torch.Tensor, stream=None):
    """The FP4-to-FP8 RFQ with the main product at the FP4 rate: X~ (MXFP4),
    X^ (MXFP8), W~ (MXFP4; see include/rfq.h)."""
    q, r, w = xq.c(), xr.c(), wq.c()
    _check(load_library().rfq_linear_mixed(ctypes.byref(q), ctypes.byref(r), _ptr(phi), phi_r_s, ctypes.byref(w),
                                           _ptr(y), out_dtype, _ptr(workspace), _stream(stream)),
           "rfq_linear_mixed")


def rfq_linear_host(x_host: torch.Tensor, wq: QTensor, y_host: torch.Tensor, out_dtype: int, x_dev: torch.Tensor,
                    xq: QTensor, xr: QTensor | None, phi: torch.Tensor | None, y_dev: torch.Tensor,
                    workspace: torch.Tensor, mode: int = RFQ_FALLBACK_ALL, tau: float = 0.0, r_s: int = 256,
                    chunk_rows: int = 0, stream=None):
    """The RFQ linear layer from host memory: x_host (CPU bf16 [M][K],
    pinned for overlapped copies) in, y_host (CPU [M][N]) out; x_dev, xq,
    xr, phi, y_dev and workspace are the caller's device scratch (see
    include/rfq.h)."""
    M, K = x_host.shape
    fb = _FB(mode, tau, 128, r_s)
    w, q = wq.c(), xq.c()
    r = xr.c() if xr is not None else None
    _check(load_library().rfq_linear_host(_ptr(x_host), M, K, ctypes.byref(fb), ctypes.byref(w), _ptr(y_host),
                                          out_dtype, chunk_rows, _ptr(x_dev), ctypes.byref(q),
                                          ctypes.byref(r) if r is not None else None, _ptr(phi), _ptr(y_dev),
                                          _ptr(workspace), _stream(stream)), "rfq_linear_host")


def rfq_workspace_status(workspace: torch.Tensor, clear: bool = False, stream=None) -> int:
    return load_library().rfq_workspace_status(_ptr(workspace), 1 if clear else 0, _stream(stream))


def rfq_dequant(q: QTensor, out: torch.Tensor, out_dtype: int | None = None, stream=None):
    if out_dtype is None:
        out_dtype = RFQ_OUT_BF16 if out.dtype == torch.bfloat16 else RFQ_OUT_F32
    qt = q.c()
    _check(load_library().rfq_dequant(ctypes.byref(qt), _ptr(out), out_dtype, _stream(stream)), "rfq_dequant")


def rfq_check_finite(x: torch.Tensor, workspace: torch.Tensor, stream=None):
    """Records RFQ_ERR_NONFINITE in the workspace if the bf16 matrix x holds an
    Inf or NaN (read it back with rfq_workspace_status)."""
    rows, k = x.shape
    _check(load_library().rfq_check_finite(_ptr(x), rows, k, _ptr(workspace), _stream(stream)), "rfq_check_finite")


def rfq_linear_grouped(xq: QTensor, xr: QTensor | None, phi: torch.Tensor | None, phi_r_s: int,
                       group_off: torch.Tensor, wq: QTensor, N: int, y: torch.Tensor, out_dtype: int,
                       workspace: torch.Tensor, stream=None):
    """Grouped RFQ GEMM (one launch over all groups).  group_off: device int32
    [groups + 1] row offsets (group starts multiples of 128); wq holds the
    groups' weights stacked, rows = groups * N."""
    a = xq.c()
    r = xr.c() if xr is not None else None
    w = wq.c()
    groups = group_off.numel() - 1
    _check(load_library().rfq_linear_grouped(ctypes.byref(a), ctypes.byref(r) if r is not None else None, _ptr(phi),
                                             phi_r_s, _ptr(group_off), groups, ctypes.byref(w), N, _ptr(y), out_dtype,
                                             _ptr(workspace), _stream(stream)), "rfq_linear_grouped")


def rfq_convert(src: QTensor, dst: QTensor, stream=None):
    """Exact re-encoding of an MXFP4 tensor as MXFP8 (E4M3 codes of the same
    values, the same scales)."""
    a, b = src.c(), dst.c()
    _check(load_library().rfq_convert(ctypes.byref(a), ctypes.byref(b), _stream(stream)), "rfq_convert")


def bf16_operand(t: torch.Tensor) -> QTensor:
    """A bf16 [rows, k] tensor as an RFQ_FMT_BF16 operand (e.g. the exact
    expansion of a HiF4 weight written by rfq_dequant)."""
    rows, k = t.shape
    return QTensor(RFQ_FMT_BF16, RFQ_SCALE_ROWMAJOR, rows, k, t, t)


def rfq_linear_noalloc(xq: QTensor, xr: QTensor | None, phi: torch.Tensor | None, phi_r_s: int, wq: QTensor,
                       y: torch.Tensor, out_dtype: int, stream=None):
    """rfq_linear for callers that cannot allocate device memory: the GEMM's
    workspace is a fixed array inside the library (see include/rfq.h)."""
    q, w = xq.c(), wq.c()
    r = xr.c() if xr is not None else None
    _check(load_library().rfq_linear_noalloc(ctypes.byref(q), ctypes.byref(r) if r is not None else None,
                                             _ptr(phi), phi_r_s, ctypes.byref(w), _ptr(y), out_dtype,
                                             _stream(stream)), "rfq_linear_noalloc")


def rfq_linear_fused_workspace_bytes(M: int, K: int, mode: int = RFQ_FALLBACK_ALL) -> int:
    fb = _FB(mode, 0.0, 128, 256)
    return load_library().rfq_linear_fused_workspace_bytes(M, K, ctypes.byref(fb))


def fused_workspace(M: int, K: int, mode: int = RFQ_FALLBACK_ALL, device="cuda") -> torch.Tensor:
    """A zeroed workspace for rfq_linear_fused (int32 words)."""
    n = rfq_linear_fused_workspace_bytes(M, K, mode)
    return torch.zeros((n + 3) // 4, dtype=torch.int32, device=device)


def rfq_linear_fused(x: torch.Tensor, wq: QTensor, y: torch.Tensor, out_dtype: int, workspace: torch.Tensor,
                     mode: int = RFQ_FALLBACK_ALL, stream=None):
    """Y = Q(X) W~ + phi Q(X - Q(X)) W~ with X (bf16 [M, K]) quantized inside
    the GEMM; mode RFQ_FALLBACK_ALL or RFQ_FALLBACK_NONE."""
    M, K = x.shape
    fb = _FB(mode, 0.0, 128, 256)
    need = rfq_linear_fused_workspace_bytes(M, K, mode)
    if workspace.numel() * workspace.element_size() < need:
        raise ValueError(f"rfq_linear_fused needs a workspace of {need} bytes (rfq_linear_fused_workspace_bytes)")
    w = wq.c()
    _check(load_library().rfq_linear_fused(_ptr(x), M, K, ctypes.byref(w), ctypes.byref(fb), _ptr(y), out_dtype,
                                           _ptr(workspace), _stream(stream)), "rfq_linear_fused")


def rfq_fp4_mma_peak(cta_pair: bool, iters: int, workspace: torch.Tensor, stream=None) -> float:
    """Launches the MMA-only FP4 rate measurement (see include/rfq.h) on the
    stream; returns the launch's MMA work in FLOP (time it with events)."""
    flop = ctypes.c_double(0.0)
    _check(load_library().rfq_fp4_mma_peak(1 if cta_pair else 0, iters, _ptr(workspace), ctypes.byref(flop),
                                           _stream(stream)), "rfq_fp4_mma_peak")
    return flop.value


PROFILE_KEYS = ("cycles", "ns", "wait_acc_cycles", "wait_copies_cycles", "wait_scales_cycles", "stages", "pairs",
                "tiles")


def rfq_linear_profile(xq: QTensor, xr: QTensor, wq: QTensor, y: torch.Tensor, out_dtype: int,
                       workspace: torch.Tensor, stream=None) -> dict:
    """rfq_linear on the CTA-pair kernel's measuring build: returns the MMA
    threads' summed counters (see include/rfq.h); synchronizes."""
    workspace.view(torch.uint8)[32:96].zero_()
    q, r, w = xq.c(), xr.c(), wq.c()
    _check(load_library().rfq_linear_profile(ctypes.byref(q), ctypes.byref(r), ctypes.byref(w), _ptr(y), out_dtype,
                                             _ptr(workspace), _stream(stream)), "rfq_linear_profile")
    torch.cuda.synchronize(workspace.device)
    v = workspace.view(torch.uint8)[32:96].cpu().view(torch.int64).tolist()
    return dict(zip(PROFILE_KEYS, v))


def rfq_debug_bounds(clear: bool = False) -> tuple[int, int]:
    """(status, source line) of the debug build's first out-of-range store
    (see include/rfq.h); the normal build returns RFQ_ERR_UNSUPPORTED."""
    line = ctypes.c_int32(0)
    st = load_library().rfq_debug_bounds(ctypes.byref(line), 1 if clear else 0)
    return st, line.value
