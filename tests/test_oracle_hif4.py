"""Pins for the HiF4 part of the CPU oracle (Sec. 3.3).

The decoder and the format's printed properties are pinned: the UE6M2 macro
scale with bias 48, the S1P2 element grid, the 4.81-binade intra-block range
and the 4.5 bits per element.  The encoder's choice of macro scale and
micro-exponents is a reading (the paper defines only the decoder): parity
unpinned for that choice; its consistency and optimality properties are
checked here, and a hand-worked block fixes the reading's output.
"""
import math

import numpy as np

from conftest import read_golden
from paper_2608_26581_gb300.synth import f32_to_bf16_bits


def test_ue6m2_table(orc):
    vals = [orc.ue6m2_decode(b) for b in range(256)]
    assert vals[0] == 2.0 ** -48            # E = 0, M = 0, bias 48
    assert vals[0xC0] == 1.0                # E = 48
    assert vals[0xC1] == 1.25 and vals[0xC2] == 1.5 and vals[0xC3] == 1.75
    assert vals[255] == 1.75 * 2.0 ** 15    # E = 63, M = 3
    assert all(a < b for a, b in zip(vals, vals[1:]))


def test_s1p2_grid(orc):
    assert [orc.s1p2_decode(c) for c in range(8)] == [k / 4 for k in range(8)]
    assert [orc.s1p2_decode(c | 8) for c in range(1, 8)] == [-k / 4 for k in range(1, 8)]


def test_intra_block_range_is_4_81_binades(orc):
    # Sec. 3.3: the micro-exponents widen the range inside one block to 4.81
    # binades: largest over smallest non-zero magnitude for a fixed S_macro.
    mags = []
    for e18 in (0, 1):
        for e116 in (0, 1):
            meta = 0xC0 | (e18 << 8) | (e116 << 16)
            mags += [abs(orc.hif4_decode(meta, 0, c)) for c in range(1, 8)]
    r = math.log2(max(mags) / min(mags))
    assert round(r, 2) == 4.81


def test_storage_is_4_5_bits_per_element():
    # Sec. 3.3: 64 elements with 32 bits of metadata -> 4.5 bits each.
    code_bytes, meta_bytes = 64 // 2, 4
    assert (code_bytes + meta_bytes) * 8 / 64 == 4.5


def test_golden_handworked_block(orc):
    g = read_golden("hif4_block_handworked.txt")
    x = np.array([float(v) for v in g["x"]], np.float32)
    xb = f32_to_bf16_bits(x)
    xd = orc.bf16_bits_to_f64(xb)
    assert np.array_equal(xd, x.astype(np.float64))
    c, m = orc.quantize(orc.FMT_HIF4, xd.reshape(1, 64))
    assert int(m[0, 0]) == int(g["meta_hex"][0], 16)
    assert c[0].tolist() == [int(h, 16) for h in g["codes_hex"]]
    dec = orc.dequant(orc.FMT_HIF4, c, m, 1, 64)[0]
    assert dec.tolist() == [float(v) for v in g["decoded"]]


def _decode_all(orc, meta, codes):
    return np.array([orc.hif4_decode(meta, i, int(codes[i])) for i in range(64)])


def test_encoder_rounds_to_nearest_on_its_grid(orc):
    # Given the chosen metadata, every element is the nearest point of its
    # grid {k * step, k = 0..7} (brute force), ties to even k.
    rng = np.random.default_rng(0)
    for trial in range(200):
        x = rng.standard_t(3, 64) * 10.0 ** rng.integers(-4, 4)
        x[rng.integers(0, 64)] *= 50
        xb = f32_to_bf16_bits(x.astype(np.float32))
        xd = orc.bf16_bits_to_f64(xb).reshape(1, 64)
        c, m = orc.quantize(orc.FMT_HIF4, xd)
        meta = int(m[0, 0])
        codes = [(c[0, i // 2] >> (4 * (i & 1))) & 0xF for i in range(64)]
        for i in range(64):
            grid = [abs(orc.hif4_decode(meta, i, k)) for k in range(8)]
            a = abs(xd[0, i])
            d = [abs(a - g) for g in grid]
            best = min(d)
            ks = [k for k in range(8) if d[k] == best]
            want = ks[0] if len(ks) == 1 else [k for k in ks if k % 2 == 0][0]
            assert codes[i] & 7 == want, (trial, i)
            assert (codes[i] >> 3) == (1 if math.copysign(1, xd[0, i]) < 0 else 0)


def test_encoder_choice_is_minimal_and_unsaturated(orc):
    # Reading R6: S is the smallest UE6M2 value with 7 S >= amax; each
    # sub-group's effective exponent is the smallest that keeps its amax
    # within 1.75 2^t S (or forced up by E1_8); no element saturates.
    rng = np.random.default_rng(1)
    for trial in range(300):
        x = rng.laplace(0, 0.3, 64) * 10.0 ** rng.integers(-6, 5)
        xb = f32_to_bf16_bits(x.astype(np.float32))
        xd = orc.bf16_bits_to_f64(xb)
        c, m = orc.quantize(orc.FMT_HIF4, xd.reshape(1, 64))
        meta = int(m[0, 0])
        sb = meta & 0xFF
        S = orc.ue6m2_decode(sb)
        amax = np.abs(xd).max()
        assert 7 * S >= amax
        if sb > 0:
            assert 7 * orc.ue6m2_decode(sb - 1) < amax
        e18 = (meta >> 8) & 0xFF
        e116 = meta >> 16
        for j in range(16):
            g = j // 2
            t = ((e18 >> g) & 1) + ((e116 >> j) & 1)
            a = np.abs(xd[4 * j:4 * j + 4]).max()
            assert a <= 1.75 * S * 2 ** t
            if (e18 >> g) & 1 == 0 and t > 0:
                assert a > 1.75 * S * 2 ** (t - 1)
        for g in range(8):
            if (e18 >> g) & 1:
                tmax = [np.abs(xd[4 * j:4 * j + 4]).max() for j in (2 * g, 2 * g + 1)]
                assert max(tmax) > 3.5 * S


def test_hif4_rfq_residual_shrinks_error(orc):
    rng = np.random.default_rng(2)
    x = rng.laplace(0, 0.3, (16, 256))
    x[:, [7, 100]] *= 50
    xb = f32_to_bf16_bits(x.astype(np.float32))
    xd = orc.bf16_bits_to_f64(xb)
    q = orc.quantize_act(xb, orc.FMT_HIF4, orc.PHI_ALL)
    xt = orc.dequant(orc.FMT_HIF4, q["main_codes"], q["main_scales"], 16, 256)
    xh = orc.dequant(orc.FMT_HIF4, q["res_codes"], q["res_scales"], 16, 256)
    rc, rs = orc.quantize(orc.FMT_HIF4, xd - xt)
    assert np.array_equal(rc, q["res_codes"]) and np.array_equal(rs, q["res_scales"])
    e1 = np.linalg.norm(xd - xt)
    e2 = np.linalg.norm(xd - xt - xh)
    assert e2 < 0.1 * e1
