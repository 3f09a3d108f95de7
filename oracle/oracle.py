"""ctypes wrapper around ``rfq_oracle.c``, the plain fp64 CPU oracle of RFQ.

TEST INFRASTRUCTURE ONLY (see the package docstring).  Every function here
only marshals numpy arrays into the C oracle; the arithmetic lives in
``rfq_oracle.c`` where each step cites the paper's section or equation.

Layouts (shared with the library's public contract, not with its code):
  codes   MXFP4 / HiF4: uint8 [rows, k/2], element 2j in the low nibble, 2j+1
          in the high one; MXFP8: uint8 E4M3 [rows, k]
  scales  MXFP4 / MXFP8: uint8 E8M0 [rows, k/32]; HiF4: uint32 metadata [rows, k/64]
  phi     uint8 [ceil(M/p_s), ceil(K/r_s)]
"""
from __future__ import annotations

import ctypes
import os
import platform
import subprocess

import numpy as np

FMT_MXFP4 = 0
FMT_HIF4 = 1
FMT_MXFP8 = 2
PHI_NONE = 0
PHI_ALL = 1
PHI_AMAX = 2

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rfq_oracle.c")
_LIB = os.path.join(_HERE, f"librfq_oracle.{platform.machine()}.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math, no FMA contraction, so x86
    and Arm hosts compute bit-identical results)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
             "-fno-fast-math", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        I64 = ctypes.c_int64
        I = ctypes.c_int
        D = ctypes.c_double
        lib.rfq_o_bf16_to_double.restype = D
        lib.rfq_o_bf16_to_double.argtypes = [ctypes.c_uint16]
        lib.rfq_o_e2m1_decode.restype = D
        lib.rfq_o_e2m1_decode.argtypes = [I]
        lib.rfq_o_e2m1_encode.restype = I
        lib.rfq_o_e2m1_encode.argtypes = [D]
        lib.rfq_o_mx_scale_exp.restype = I
        lib.rfq_o_mx_scale_exp.argtypes = [D]
        lib.rfq_o_e4m3_decode.restype = D
        lib.rfq_o_e4m3_decode.argtypes = [I]
        lib.rfq_o_e4m3_encode.restype = I
        lib.rfq_o_e4m3_encode.argtypes = [D]
        lib.rfq_o_mx8_scale_exp.restype = I
        lib.rfq_o_mx8_scale_exp.argtypes = [D]
        lib.rfq_o_mxfp8_quantize.argtypes = [P, I64, I64, P, P]
        lib.rfq_o_mxfp8_dequant.argtypes = [P, P, I64, I64, P]
        lib.rfq_o_quantize_act2.argtypes = [P, I64, I64, I, I, I, D, I64, I64, P, P, P, P, P]
        lib.rfq_o_linear2.argtypes = [I, I, I, P, P, P, P, I64, I64, P, P, I64, P]
        lib.rfq_o_ue6m2_decode.restype = D
        lib.rfq_o_ue6m2_decode.argtypes = [I]
        lib.rfq_o_s1p2_decode.restype = D
        lib.rfq_o_s1p2_decode.argtypes = [I]
        lib.rfq_o_hif4_decode.restype = D
        lib.rfq_o_hif4_decode.argtypes = [ctypes.c_uint32, I, I]
        lib.rfq_o_mxfp4_quantize.argtypes = [P, I64, I64, P, P]
        lib.rfq_o_mxfp4_dequant.argtypes = [P, P, I64, I64, P]
        lib.rfq_o_hif4_quantize.argtypes = [P, I64, I64, P, P]
        lib.rfq_o_hif4_dequant.argtypes = [P, P, I64, I64, P]
        lib.rfq_o_dequant.argtypes = [I, P, P, I64, I64, P]
        lib.rfq_o_phi.argtypes = [P, I64, I64, I, D, I64, I64, P]
        lib.rfq_o_quantize_act.argtypes = [P, I64, I64, I, I, D, I64, I64, P, P, P, P, P]
        lib.rfq_o_quantize_weight.argtypes = [P, I64, I64, I, P, P]
        lib.rfq_o_linear.argtypes = [I, P, P, P, P, I64, I64, P, P, I64, P]
        _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _scale_shape(fmt, rows, k):
    return (rows, k // 64) if fmt == FMT_HIF4 else (rows, k // 32)


def _code_shape(fmt, rows, k):
    return (rows, k) if fmt == FMT_MXFP8 else (rows, k // 2)


def _scale_dtype(fmt):
    return np.uint32 if fmt == FMT_HIF4 else np.uint8


# ---- scalar helpers ---------------------------------------------------------

def bf16_to_double(bits: int) -> float:
    return _load().rfq_o_bf16_to_double(int(bits))


def e2m1_decode(code: int) -> float:
    return _load().rfq_o_e2m1_decode(int(code))


def e2m1_encode(y: float) -> int:
    return _load().rfq_o_e2m1_encode(float(y))


def mx_scale_exp(amax: float) -> int:
    return _load().rfq_o_mx_scale_exp(float(amax))


def e4m3_decode(code: int) -> float:
    return _load().rfq_o_e4m3_decode(int(code))


def e4m3_encode(y: float) -> int:
    return _load().rfq_o_e4m3_encode(float(y))


def mx8_scale_exp(amax: float) -> int:
    return _load().rfq_o_mx8_scale_exp(float(amax))


def ue6m2_decode(byte: int) -> float:
    return _load().rfq_o_ue6m2_decode(int(byte))


def s1p2_decode(code: int) -> float:
    return _load().rfq_o_s1p2_decode(int(code))


def hif4_decode(meta: int, i: int, code: int) -> float:
    return _load().rfq_o_hif4_decode(int(meta), int(i), int(code))


# ---- array functions ---------------------------------------------------------

def quantize(fmt: int, x: np.ndarray):
    """Quantize an fp64 [rows, k] array along k: returns (codes, scales)."""
    x = _c(x, np.float64)
    rows, k = x.shape
    codes = np.zeros(_code_shape(fmt, rows, k), np.uint8)
    scales = np.zeros(_scale_shape(fmt, rows, k), _scale_dtype(fmt))
    if fmt == FMT_HIF4:
        _load().rfq_o_hif4_quantize(_p(x), rows, k, _p(codes), _p(scales))
    elif fmt == FMT_MXFP8:
        _load().rfq_o_mxfp8_quantize(_p(x), rows, k, _p(codes), _p(scales))
    else:
        _load().rfq_o_mxfp4_quantize(_p(x), rows, k, _p(codes), _p(scales))
    return codes, scales


def dequant(fmt: int, codes: np.ndarray, scales: np.ndarray, rows: int, k: int) -> np.ndarray:
    codes = _c(codes, np.uint8)
    scales = _c(scales, _scale_dtype(fmt))
    out = np.empty((rows, k), np.float64)
    _load().rfq_o_dequant(fmt, _p(codes), _p(scales), rows, k, _p(out))
    return out


def phi(x: np.ndarray, mode: int, tau: float, p_s: int, r_s: int) -> np.ndarray:
    x = _c(x, np.float64)
    M, K = x.shape
    out = np.zeros(((M + p_s - 1) // p_s, (K + r_s - 1) // r_s), np.uint8)
    _load().rfq_o_phi(_p(x), M, K, mode, float(tau), p_s, r_s, _p(out))
    return out


def quantize_act(x_bf16: np.ndarray, fmt: int = FMT_MXFP4, mode: int = PHI_ALL,
                 tau: float = 0.0, p_s: int = 128, r_s: int = 256, res_fmt: int | None = None):
    """RFQ activation decomposition (Sec. 4.3).  ``x_bf16``: uint16 bf16 bit
    patterns [M, K].  ``res_fmt``: the residual pathway's format (default: the
    main one; FMT_MXFP8 under an MXFP4 main pathway is the FP4-to-FP8
    variant).  Returns dict(main_codes, main_scales, res_codes, res_scales,
    phi); the residual entries are None for mode PHI_NONE."""
    x = _c(x_bf16, np.uint16)
    M, K = x.shape
    res_fmt = fmt if res_fmt is None else res_fmt
    mc = np.zeros(_code_shape(fmt, M, K), np.uint8)
    ms = np.zeros(_scale_shape(fmt, M, K), _scale_dtype(fmt))
    has_res = mode != PHI_NONE
    rc = np.zeros(_code_shape(res_fmt, M, K), np.uint8) if has_res else None
    rs = np.zeros(_scale_shape(res_fmt, M, K), _scale_dtype(res_fmt)) if has_res else None
    ph = np.zeros(((M + p_s - 1) // p_s, (K + r_s - 1) // r_s), np.uint8)
    _load().rfq_o_quantize_act2(_p(x), M, K, fmt, res_fmt, mode, float(tau), p_s, r_s,
                                _p(mc), _p(ms), _p(rc), _p(rs), _p(ph))
    return dict(main_codes=mc, main_scales=ms, res_codes=rc, res_scales=rs, phi=ph)


def quantize_weight(w_bf16: np.ndarray, fmt: int = FMT_MXFP4):
    """Weight quantization of bf16 W [K, N] along K; returns K-major
    (codes [N, K/2], scales [N, K/32] or [N, K/64])."""
    w = _c(w_bf16, np.uint16)
    K, N = w.shape
    codes = np.zeros(_code_shape(fmt, N, K), np.uint8)
    scales = np.zeros(_scale_shape(fmt, N, K), _scale_dtype(fmt))
    _load().rfq_o_quantize_weight(_p(w), K, N, fmt, _p(codes), _p(scales))
    return codes, scales


def linear(fmt: int, xm_codes, xm_scales, xr_codes, xr_scales, w_codes, w_scales,
           M: int, K: int, N: int, res_fmt: int | None = None, w_fmt: int | None = None) -> np.ndarray:
    """RFQ GEMM (Algorithm 1, Eq. rfq) in fp64; returns Y [M, N] float64.
    ``res_fmt`` / ``w_fmt``: the residual's and the weight's formats (default:
    ``fmt``)."""
    res_fmt = fmt if res_fmt is None else res_fmt
    w_fmt = fmt if w_fmt is None else w_fmt
    xm_codes = _c(xm_codes, np.uint8)
    xm_scales = _c(xm_scales, _scale_dtype(fmt))
    if xr_codes is not None:
        xr_codes = _c(xr_codes, np.uint8)
        xr_scales = _c(xr_scales, _scale_dtype(res_fmt))
    w_codes = _c(w_codes, np.uint8)
    w_scales = _c(w_scales, _scale_dtype(w_fmt))
    Y = np.empty((M, N), np.float64)
    _load().rfq_o_linear2(fmt, res_fmt, w_fmt, _p(xm_codes), _p(xm_scales), _p(xr_codes), _p(xr_scales),
                          M, K, _p(w_codes), _p(w_scales), N, _p(Y))
    return Y


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns exactly (a bf16 is the top half of a binary32)."""
    b = np.ascontiguousarray(bits, np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)
