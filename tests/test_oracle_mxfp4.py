"""Pins for the MXFP4 part of the CPU oracle.

Each test checks the oracle against something fixed outside it: the E2M1
value table of the MX format (Sec. 3.2.2), hand-worked blocks under
tests/golden/, brute force over every code or scale byte, and error bounds
that follow from the grid spacing.
"""
import math

import numpy as np
import pytest

from conftest import read_golden
from paper_2608_26581_gb300.synth import f32_to_bf16_bits


# E2M1 code -> value, the OCP MX element table for 1 sign / 2 exponent /
# 1 mantissa bit, bias 1, subnormal at exponent field 0 (Sec. 3.2.2, Eq. 1).
E2M1_TABLE = {
    0b0000: 0.0, 0b0001: 0.5, 0b0010: 1.0, 0b0011: 1.5,
    0b0100: 2.0, 0b0101: 3.0, 0b0110: 4.0, 0b0111: 6.0,
    0b1000: -0.0, 0b1001: -0.5, 0b1010: -1.0, 0b1011: -1.5,
    0b1100: -2.0, 0b1101: -3.0, 0b1110: -4.0, 0b1111: -6.0,
}


def test_e2m1_value_table(orc):
    for code, v in E2M1_TABLE.items():
        got = orc.e2m1_decode(code)
        assert got == v and math.copysign(1, got) == math.copysign(1, v), (code, got, v)


# (input, code) pairs at and around every rounding midpoint of the E2M1 grid.
THRESHOLDS = [
    (0.0, 0x0), (-0.0, 0x8), (0.1, 0x0), (-0.1, 0x8),
    (0.25, 0x0), (0.2500001, 0x1), (0.5, 0x1), (0.7499999, 0x1),
    (0.75, 0x2), (1.0, 0x2), (1.25, 0x2), (1.2500001, 0x3), (1.5, 0x3),
    (1.7499999, 0x3), (1.75, 0x4), (2.0, 0x4), (2.5, 0x4), (2.5000001, 0x5),
    (3.0, 0x5), (3.4999999, 0x5), (3.5, 0x6), (4.0, 0x6), (5.0, 0x6),
    (5.0000001, 0x7), (6.0, 0x7), (7.0, 0x7), (8.0, 0x7), (1e30, 0x7),
    (-0.75, 0xA), (-5.0, 0xE), (-5.0000001, 0xF), (-100.0, 0xF),
]


@pytest.mark.parametrize("y,code", THRESHOLDS)
def test_e2m1_rounding_midpoints(orc, y, code):
    assert orc.e2m1_encode(y) == code


def _bruteforce_e2m1(y):
    """argmin over the 8 magnitudes; ties go to the even mantissa bit."""
    a = abs(y)
    best = None
    for c in range(8):
        d = abs(a - E2M1_TABLE[c])
        if best is None or d < best[0] or (d == best[0] and (c & 1) == 0 and (best[1] & 1) == 1):
            best = (d, c)
    return best[1] | (8 if math.copysign(1.0, y) < 0 else 0)


def _bruteforce_e2m1_vec(y):
    """_bruteforce_e2m1 over an array: the argmin over the 8 magnitudes, ties
    to the even mantissa bit, the sign bit of y."""
    mags = np.array([E2M1_TABLE[c] for c in range(8)])
    d = np.abs(np.abs(y)[:, None] - mags[None, :])
    best = d.min(axis=1, keepdims=True)
    tied = d == best
    # among the tied codes prefer an even one (at most two codes tie)
    even = tied & (np.arange(8)[None, :] % 2 == 0)
    code = np.where(even.any(axis=1), even.argmax(axis=1), tied.argmax(axis=1))
    return code | np.where(np.signbit(y), 8, 0)


def test_e2m1_encode_bruteforce_all_bf16(orc):
    # Every one of the 65 536 bf16 patterns that is finite, divided by each
    # power of two that moves it into (or near) the E2M1 range, must round
    # like the brute-force argmin.
    bits = np.arange(0, 1 << 16, dtype=np.uint32)
    f = (bits << 16).view(np.float32)
    vals = f[np.isfinite(f)].astype(np.float64)
    assert vals.size == 65536 - 2 * 128          # every pattern but the 128 Inf / NaN ones per sign
    ex = np.frexp(np.abs(vals))[1]
    ys = np.concatenate([np.where(vals == 0, vals, np.ldexp(vals, -(ex - 1) + s)) for s in range(-3, 5)])
    want = _bruteforce_e2m1_vec(ys)
    got = np.fromiter((orc.e2m1_encode(float(y)) for y in ys), np.int64, ys.size)
    bad = np.nonzero(got != want)[0]
    assert bad.size == 0, [(ys[i], got[i], want[i]) for i in bad[:5]]
    # the vectorised brute force agrees with the scalar one on a sample
    for y in ys[:: 4099]:
        assert _bruteforce_e2m1(y) == _bruteforce_e2m1_vec(np.array([y]))[0]


def test_scale_rule_bruteforce_all_bytes(orc):
    # The chosen E8M0 byte is the unique byte b in [0, 254] with
    # 4 <= amax / 2^(b-127) < 8 (the largest E2M1 binade), else the clamp.
    rng = np.random.default_rng(1)
    amaxes = [2.0 ** p for p in range(-133, 128)]
    amaxes += [1.5 * 2.0 ** p for p in range(-133, 127)]
    amaxes += list(np.abs(rng.standard_normal(300)) * 10.0 ** rng.integers(-30, 30, 300))
    for a in amaxes:
        e = orc.mx_scale_exp(a)
        hits = [b for b in range(255) if 4.0 <= a / 2.0 ** (b - 127) < 8.0]
        if hits:
            assert len(hits) == 1 and e + 127 == hits[0], (a, e, hits)
        else:
            assert a < 4.0 * 2.0 ** -127 and e == -127, (a, e)
    assert orc.mx_scale_exp(0.0) == -127


def _golden_block(orc, name):
    g = read_golden(name)
    x = np.array([float(v) for v in g["x"]], np.float32)
    xb = f32_to_bf16_bits(x)
    assert np.array_equal(orc.bf16_bits_to_f64(xb), x.astype(np.float64)), "fixture not bf16-exact"
    q = orc.quantize_act(xb.reshape(1, -1), orc.FMT_MXFP4, orc.PHI_ALL)
    assert q["main_scales"][0, 0] == int(g["main_scale"][0])
    assert q["main_codes"][0].tolist() == [int(h, 16) for h in g["main_codes_hex"]]
    assert q["res_scales"][0, 0] == int(g["res_scale"][0])
    assert q["res_codes"][0].tolist() == [int(h, 16) for h in g["res_codes_hex"]]


def test_golden_handworked_block(orc):
    _golden_block(orc, "mxfp4_block_handworked.txt")


def test_golden_subnormal_block(orc):
    _golden_block(orc, "mxfp4_block_subnormal.txt")


def _representable_blocks(rng, rows, k):
    """Blocks made of exact MXFP4 values: random codes times 2^e, with one
    element of magnitude 4 or 6 per block so the shared exponent is e."""
    mags = np.array([0, 0.5, 1, 1.5, 2, 3, 4, 6])
    codes = rng.integers(0, 8, (rows, k))
    sign = np.where(rng.random((rows, k)) < 0.5, -1.0, 1.0)
    x = mags[codes] * sign
    nb = k // 32
    lead = rng.integers(0, 32, (rows, nb))
    for r in range(rows):
        for b in range(nb):
            x[r, b * 32 + lead[r, b]] = rng.choice([4.0, 6.0, -4.0, -6.0])
    e = rng.integers(-100, 100, (rows, nb))
    x = x * np.repeat(2.0 ** e, 32, axis=1)
    return x


def test_zero_residual_on_representable_input(orc):
    rng = np.random.default_rng(2)
    x = _representable_blocks(rng, 16, 256)
    xb = f32_to_bf16_bits(x.astype(np.float32))
    assert np.array_equal(orc.bf16_bits_to_f64(xb), x)
    q = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_ALL)
    xt = orc.dequant(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], 16, 256)
    assert np.array_equal(xt, x)
    assert not q["res_codes"].any() and not q["res_scales"].any()


def _heavy_tailed(rng, rows, k):
    x = rng.standard_t(3, (rows, k)) * 10.0 ** rng.integers(-3, 4, (rows, 1))
    x[:, rng.choice(k, 3, replace=False)] *= 100.0
    return f32_to_bf16_bits(x.astype(np.float32))


def test_error_bounds_stage1_and_stage2(orc):
    # Stage 1: |x - x~| <= half the grid spacing of the binade x/2^e falls in
    # (0.25, 0.5, 1 times 2^e), and < 2^(e+1) when saturated at 6.
    # Stage 2 (RFQ): |x - x~ - x^| < 2^(e_R+1) <= 2^(e-1).
    rng = np.random.default_rng(3)
    xb = _heavy_tailed(rng, 64, 512)
    x = orc.bf16_bits_to_f64(xb)
    q = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_ALL)
    xt = orc.dequant(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], 64, 512)
    xh = orc.dequant(orc.FMT_MXFP4, q["res_codes"], q["res_scales"], 64, 512)
    e = np.repeat(q["main_scales"].astype(np.int64) - 127, 32, axis=1)
    eR = np.repeat(q["res_scales"].astype(np.int64) - 127, 32, axis=1)
    y = np.abs(x) / 2.0 ** e
    half = np.where(y < 2, 0.25, np.where(y < 4, 0.5, 1.0)) * 2.0 ** e
    err1 = np.abs(x - xt)
    sat = y > 6
    assert np.all(err1[~sat] <= half[~sat])
    assert np.all(err1[sat] < 2.0 ** (e[sat] + 1))
    err2 = np.abs(x - xt - xh)
    nz = q["res_scales"].repeat(32, axis=1) > 0
    assert np.all(err2[nz] < 2.0 ** (eR[nz] + 1))
    assert np.all(eR[nz] <= e[nz] - 2)
    # per block, the two-stage decomposition is never worse than stage 1
    b1 = (err1 ** 2).reshape(64, 16, 32).sum(-1)
    b2 = (err2 ** 2).reshape(64, 16, 32).sum(-1)
    assert np.all(b2 <= b1)
    assert b2.sum() < 0.05 * b1.sum()


def test_residual_is_exact_difference(orc):
    # Sec. 4.3: dX = X - X~.  Quantizing dX directly must give the stored
    # residual codes (the residual is exact in fp64).
    rng = np.random.default_rng(4)
    xb = _heavy_tailed(rng, 8, 256)
    x = orc.bf16_bits_to_f64(xb)
    q = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_ALL)
    xt = orc.dequant(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], 8, 256)
    rc, rs = orc.quantize(orc.FMT_MXFP4, x - xt)
    assert np.array_equal(rc, q["res_codes"]) and np.array_equal(rs, q["res_scales"])
    mc, ms = orc.quantize(orc.FMT_MXFP4, x)
    assert np.array_equal(mc, q["main_codes"]) and np.array_equal(ms, q["main_scales"])


def test_nibble_order_and_scale_index(orc):
    # One non-zero element at a time: its code lands in the nibble and the
    # scale byte the layout names (element 2j low nibble; block k // 32).
    x = np.zeros((3, 96))
    for pos in [0, 1, 31, 32, 33, 95]:
        x[:] = 0
        x[1, pos] = 6.0
        c, s = orc.quantize(orc.FMT_MXFP4, x)
        assert s[1, pos // 32] == 127 and s.sum() == 127
        assert c[1, pos // 2] == (0x70 if pos & 1 else 0x07) and int(c.sum()) == c[1, pos // 2]
