"""Pins for the MXFP8 (E4M3) part of the CPU oracle and its FP4-to-FP8
residual pathway (Sec. 3.2.1, Eq. 1; Sec. 4.2 / 4.3, readings R11, R12).

The E4M3 element is checked against PyTorch's float8_e4m3fn (a library
implementation of the OCP E4M3 format, independent of the oracle): every
one of the 256 codes decodes to the same value, and every finite bf16 input
inside the range rounds to the same value as PyTorch's round-to-nearest-even
conversion.  The scale rule is checked by brute force and the residual
pathway by the error bounds the two grids imply.
"""
import math

import numpy as np
import pytest
import torch

from paper_2608_26581_gb300.synth import f32_to_bf16_bits


def _torch_e4m3_values(codes):
    return torch.from_numpy(np.asarray(codes, np.uint8)).view(torch.float8_e4m3fn).float().numpy()


def test_e4m3_decode_matches_library_for_every_code(orc):
    codes = np.arange(256)
    ref = _torch_e4m3_values(codes)
    for c in codes:
        got = orc.e4m3_decode(int(c))
        if math.isnan(ref[c]):
            assert math.isnan(got), c
        else:
            assert got == ref[c] and math.copysign(1, got) == math.copysign(1, ref[c]), (c, got, ref[c])
    # closed forms of the format: largest finite, smallest normal, smallest subnormal
    assert orc.e4m3_decode(0x7E) == 448.0
    assert orc.e4m3_decode(0x08) == 2.0 ** -6
    assert orc.e4m3_decode(0x01) == 2.0 ** -9
    assert math.isnan(orc.e4m3_decode(0x7F)) and math.isnan(orc.e4m3_decode(0xFF))


def test_e4m3_encode_every_finite_bf16_in_range(orc):
    """All 65536 bf16 patterns: inside [-448, 448] the code's value is the
    library's RNE conversion; beyond it the code saturates to +-448; the sign
    of the input is kept (also for values that round to zero)."""
    bits = np.arange(65536, dtype=np.uint32)
    x = (bits << 16).view(np.float32)
    fin = np.isfinite(x)
    xs = x[fin]
    codes = np.array([orc.e4m3_encode(float(v)) for v in xs], np.int64)
    vals = np.array([orc.e4m3_decode(int(c)) for c in codes])
    inside = np.abs(xs) <= 448.0
    ref = torch.from_numpy(xs[inside].copy()).to(torch.float8_e4m3fn).float().numpy()
    assert np.array_equal(vals[inside], ref)
    assert np.all(np.abs(vals[~inside]) == 448.0)
    assert np.all(np.signbit(vals) == np.signbit(xs))


@pytest.mark.parametrize("y,code", [
    (0.0, 0x00), (-0.0, 0x80), (2.0 ** -10, 0x00), (2.0 ** -10 + 2.0 ** -30, 0x01),   # subnormal midpoint
    (3 * 2.0 ** -10, 0x02),                              # tie between codes 1 and 2 -> even (2)
    (2.0 ** -6 - 2.0 ** -11, 0x08),                     # rounds up into the first normal binade
    (1.0 + 1.0 / 16, 0x38), (1.0 + 3.0 / 16, 0x3A),     # ties to even mantissa (0 and 2)
    (448.0, 0x7E), (464.0, 0x7E), (470.0, 0x7E), (1e30, 0x7E), (-1e30, 0xFE),
])
def test_e4m3_midpoints(orc, y, code):
    assert orc.e4m3_encode(y) == code


def test_mx8_scale_rule_brute_force(orc):
    """The exponent is the unique e with 256 <= amax 2^-e < 512 (the block's
    largest element lands in E4M3's top binade), clamped to [-127, 127]."""
    for b in range(1, 0x7F80, 7):
        amax = float((np.uint32(b) << 16).view(np.float32))
        e = orc.mx8_scale_exp(amax)
        cands = [c for c in range(-127, 128) if 256.0 <= amax * 2.0 ** -c < 512.0]
        if cands:
            assert e == cands[0], (amax, e, cands)
        else:
            assert e == -127 and amax * 2.0 ** 127 < 256.0
    assert orc.mx8_scale_exp(0.0) == -127


def _blocks(rng, rows=64, k=256, spread=True):
    x = rng.standard_normal((rows, k))
    if spread:                                         # rows across 40 binades
        x *= np.exp2(rng.integers(-20, 20, size=(rows, 1)))
    x[:, 5] *= 300.0                                   # an outlier channel
    bits = f32_to_bf16_bits(x.astype(np.float32))
    return bits, orc_f64(bits)


def orc_f64(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _e4m3_bound(y):
    """Largest |y - q| for q the E4M3 value of y >= 0: half an ulp
    (2^(floor(log2 y) - 4) for normal y, 2^-10 below 2^-6) up to 464, the
    midpoint above 448; beyond it the value saturates to 448."""
    half = np.where(y >= 2.0 ** -6, np.exp2(np.floor(np.log2(np.maximum(y, 2.0 ** -6))) - 4), 2.0 ** -10)
    return np.where(y <= 464.0, half, y - 448.0)


def test_mxfp8_element_error_bound(orc):
    """|x - x~| 2^-e is within the E4M3 rounding bound of |x| 2^-e.  The
    scale rule puts the block maximum in [256, 512), so maxima above 464
    saturate to 448 (an error below 64 2^e)."""
    rng = np.random.default_rng(3)
    bits, x = _blocks(rng)
    codes, scales = orc.quantize(orc.FMT_MXFP8, x)
    xq = orc.dequant(orc.FMT_MXFP8, codes, scales, *x.shape)
    e = scales.astype(np.int64).repeat(32, axis=1) - 127
    y = np.abs(x) * np.exp2(-e)
    assert np.all(np.abs(x - xq) * np.exp2(-e) <= _e4m3_bound(y))
    assert np.all(np.abs(xq) <= 448.0 * np.exp2(e)) and np.all(y < 512.0)


def test_mxfp8_roundtrip_of_grid_values(orc):
    """A block whose values all lie on the E4M3 grid at its own scale is
    reproduced exactly."""
    codes = np.array([0x7E, 0x01, 0x08, 0x38, 0xBC, 0x44, 0x00, 0x80] * 4, np.uint8)
    vals = _torch_e4m3_values(codes).astype(np.float64) * 2.0 ** 5
    c, s = orc.quantize(orc.FMT_MXFP8, vals.reshape(1, 32))
    assert s[0, 0] == 127 + 5
    back = orc.dequant(orc.FMT_MXFP8, c, s, 1, 32)[0]
    assert np.array_equal(back, vals)


def test_fp8_residual_pathway_bounds(orc):
    """FP4-to-FP8 residual (R12): x^ = Q_MXFP8(x - x~), so x - x~ - x^ is
    the E4M3 rounding error of the residual r = x - x~ in its own block
    (exponent e_R).  |r| < 2^(e+1) for the MXFP4 block exponent e, so
    e_R <= e - 8 and the RFQ error stays below 2^(e_R + 6) <= 2^(e - 2),
    against 2^(e - 1) for the MXFP4 residual."""
    rng = np.random.default_rng(4)
    bits, x = _blocks(rng)
    M, K = x.shape
    q = orc.quantize_act(bits, orc.FMT_MXFP4, orc.PHI_ALL, res_fmt=orc.FMT_MXFP8)
    assert q["res_codes"].shape == (M, K) and q["main_codes"].shape == (M, K // 2)
    xm = orc.dequant(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], M, K)
    xr = orc.dequant(orc.FMT_MXFP8, q["res_codes"], q["res_scales"], M, K)
    e = q["main_scales"].astype(np.int64).repeat(32, axis=1) - 127
    er = q["res_scales"].astype(np.int64).repeat(32, axis=1) - 127
    err = np.abs(x - xm - xr)
    assert np.all(er <= e - 8)
    assert np.all(err * np.exp2(-er) <= _e4m3_bound(np.abs(x - xm) * np.exp2(-er)))
    assert np.all(err < np.exp2(e - 2))
    # the residual pathway is the MXFP8 quantization of the exact fp64 residual
    rc, rs = orc.quantize(orc.FMT_MXFP8, x - xm)
    assert np.array_equal(rc, q["res_codes"]) and np.array_equal(rs, q["res_scales"])


def test_fp8_residual_phi_zero_blocks_and_none(orc):
    rng = np.random.default_rng(5)
    bits, x = _blocks(rng, rows=256, k=512, spread=False)
    q = orc.quantize_act(bits, orc.FMT_MXFP4, orc.PHI_AMAX, tau=50.0, p_s=128, r_s=128, res_fmt=orc.FMT_MXFP8)
    ph = q["phi"]
    assert 0 < ph.sum() < ph.size
    for p in range(ph.shape[0]):
        for r in range(ph.shape[1]):
            blk = q["res_codes"][128 * p:128 * (p + 1), 128 * r:128 * (r + 1)]
            sc = q["res_scales"][128 * p:128 * (p + 1), 4 * r:4 * (r + 1)]
            if ph[p, r] == 0:
                assert not blk.any() and not sc.any()
    q0 = orc.quantize_act(bits, orc.FMT_MXFP4, orc.PHI_NONE, res_fmt=orc.FMT_MXFP8)
    q4 = orc.quantize_act(bits, orc.FMT_MXFP4, orc.PHI_NONE)
    assert q0["res_codes"] is None and np.array_equal(q0["main_codes"], q4["main_codes"])


def test_mixed_format_gemm_is_the_fp64_product(orc):
    """linear with an MXFP8 residual (and with an MXFP8 activation against an
    MXFP4 or MXFP8 weight) equals the fp64 product of the dequantized
    operands, the library matmul standing in for the sum over k."""
    rng = np.random.default_rng(6)
    M, K, N = 24, 256, 40
    bits, x = _blocks(rng, rows=M, k=K)
    wbits = f32_to_bf16_bits((rng.standard_normal((K, N)) * 0.02).astype(np.float32))
    q = orc.quantize_act(bits, orc.FMT_MXFP4, orc.PHI_ALL, res_fmt=orc.FMT_MXFP8)
    wc, ws = orc.quantize_weight(wbits, orc.FMT_MXFP4)
    w = orc.dequant(orc.FMT_MXFP4, wc, ws, N, K)
    xm = orc.dequant(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], M, K)
    xr = orc.dequant(orc.FMT_MXFP8, q["res_codes"], q["res_scales"], M, K)
    y = orc.linear(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"], wc, ws,
                   M, K, N, res_fmt=orc.FMT_MXFP8)
    assert np.allclose(y, (xm + xr) @ w.T, rtol=1e-12, atol=1e-12 * np.abs(y).max())
    # W4A8 and W8A8 (MXFP8 activation, no residual)
    a = orc.quantize_act(bits, orc.FMT_MXFP8, orc.PHI_NONE)
    xa = orc.dequant(orc.FMT_MXFP8, a["main_codes"], a["main_scales"], M, K)
    y48 = orc.linear(orc.FMT_MXFP8, a["main_codes"], a["main_scales"], None, None, wc, ws, M, K, N,
                     w_fmt=orc.FMT_MXFP4)
    assert np.allclose(y48, xa @ w.T, rtol=1e-12, atol=1e-12 * np.abs(y48).max())
    w8c, w8s = orc.quantize_weight(wbits, orc.FMT_MXFP8)
    assert w8c.shape == (N, K)
    w8 = orc.dequant(orc.FMT_MXFP8, w8c, w8s, N, K)
    y88 = orc.linear(orc.FMT_MXFP8, a["main_codes"], a["main_scales"], None, None, w8c, w8s, M, K, N)
    assert np.allclose(y88, xa @ w8.T, rtol=1e-12, atol=1e-12 * np.abs(y88).max())
