"""Pins for the RFQ decomposition, phi and GEMM of the CPU oracle.

Checks: the GEMM against numpy's fp64 matmul of the dequantized operands
(a library routine on the same definition, Algorithm 1), phi = 0 reducing
RFQ to plain W4A4, linearity of Eq. (rfq) in its two terms, the K-major
weight layout, and the phi tiling against a numpy max over tiles.
"""
import numpy as np

from paper_2608_26581_gb300.synth import ActSpec, f32_to_bf16_bits, make_activation, make_weight


def _setup(orc, M=40, K=96, N=24, seed=0, fmt=0):
    xb = make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, seed=seed))
    wb = make_weight(K, N, seed=seed)
    wc, ws = orc.quantize_weight(wb, fmt)
    return xb, wb, wc, ws


def test_gemm_matches_numpy_matmul_of_dequantized_operands(orc):
    M, K, N = 40, 96, 24  # non-square so a transposed operand cannot pass
    xb, wb, wc, ws = _setup(orc, M, K, N)
    q = orc.quantize_act(xb)
    Y = orc.linear(0, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"],
                   wc, ws, M, K, N)
    xm = orc.dequant(0, q["main_codes"], q["main_scales"], M, K)
    xr = orc.dequant(0, q["res_codes"], q["res_scales"], M, K)
    w = orc.dequant(0, wc, ws, N, K)          # [N, K]
    ref = xm @ w.T + xr @ w.T
    assert np.allclose(Y, ref, rtol=1e-13, atol=1e-13 * np.abs(ref).max())


def test_gemm_close_to_unquantized_product(orc):
    # Sanity on scale: the RFQ product approximates X W far better than
    # plain W4A4 does (Sec. 4.3 two-stage decomposition), with the weight
    # quantization error left in both.
    M, K, N = 64, 256, 32
    xb, wb, wc, ws = _setup(orc, M, K, N, seed=3)
    q = orc.quantize_act(xb)
    w = orc.dequant(0, wc, ws, N, K)
    exact = orc.bf16_bits_to_f64(xb) @ w.T
    y_rfq = orc.linear(0, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"],
                       wc, ws, M, K, N)
    y_w4a4 = orc.linear(0, q["main_codes"], q["main_scales"], None, None, wc, ws, M, K, N)
    e_rfq = np.linalg.norm(y_rfq - exact)
    e_w4a4 = np.linalg.norm(y_w4a4 - exact)
    assert e_rfq < 0.25 * e_w4a4


def test_phi_zero_reduces_to_plain_w4a4(orc):
    M, K, N = 32, 128, 16
    xb, wb, wc, ws = _setup(orc, M, K, N, seed=1)
    q_none = orc.quantize_act(xb, mode=orc.PHI_NONE)
    q_amax = orc.quantize_act(xb, mode=orc.PHI_AMAX, tau=1e30, p_s=16, r_s=64)
    assert not q_amax["phi"].any()
    assert not q_amax["res_codes"].any() and not q_amax["res_scales"].any()
    y0 = orc.linear(0, q_none["main_codes"], q_none["main_scales"], None, None, wc, ws, M, K, N)
    y1 = orc.linear(0, q_amax["main_codes"], q_amax["main_scales"], q_amax["res_codes"],
                    q_amax["res_scales"], wc, ws, M, K, N)
    xm = orc.dequant(0, q_none["main_codes"], q_none["main_scales"], M, K)
    w = orc.dequant(0, wc, ws, N, K)
    assert np.array_equal(y0, y1)
    assert np.allclose(y0, xm @ w.T, rtol=1e-13, atol=1e-13 * np.abs(y0).max())


def test_rfq_is_linear_in_its_two_terms(orc):
    M, K, N = 24, 64, 40
    xb, wb, wc, ws = _setup(orc, M, K, N, seed=2)
    q = orc.quantize_act(xb)
    zero_c = np.zeros_like(q["main_codes"])
    zero_s = np.zeros_like(q["main_scales"])
    y = orc.linear(0, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"],
                   wc, ws, M, K, N)
    ym = orc.linear(0, q["main_codes"], q["main_scales"], None, None, wc, ws, M, K, N)
    yr = orc.linear(0, zero_c, zero_s, q["res_codes"], q["res_scales"], wc, ws, M, K, N)
    assert np.allclose(y, ym + yr, rtol=1e-12, atol=1e-12 * np.abs(y).max())


def test_weight_is_quantized_along_k(orc):
    # W [K, N] row-major; column n is quantized along K and stored as row n.
    rng = np.random.default_rng(5)
    K, N = 64, 6
    w = rng.standard_normal((K, N)).astype(np.float32)
    w[:, 2] *= 1000.0          # one loud column must not change the others' scales
    wb = f32_to_bf16_bits(w)
    wc, ws = orc.quantize_weight(wb)
    c2, s2 = orc.quantize(0, orc.bf16_bits_to_f64(wb).T)
    assert np.array_equal(wc, c2) and np.array_equal(ws, s2)
    assert ws[2].min() > ws[np.arange(N) != 2].max()


def test_phi_amax_tiles_match_numpy(orc):
    rng = np.random.default_rng(6)
    M, K = 37, 200            # ragged in both tile directions
    x = rng.standard_normal((M, K))
    x[5, 150] = 40.0
    x[36, 3] = -50.0
    # tau = 40 equals a tile maximum exactly: the criterion is strict (> tau)
    for p_s, r_s, tau in [(16, 64, 10.0), (8, 32, 3.0), (128, 256, 0.5), (16, 64, 40.0)]:
        ph = orc.phi(x, orc.PHI_AMAX, tau, p_s, r_s)
        npad = -(-M // p_s) * p_s, -(-K // r_s) * r_s
        xp = np.zeros(npad)
        xp[:M, :K] = np.abs(x)
        tmax = xp.reshape(npad[0] // p_s, p_s, npad[1] // r_s, r_s).max(axis=(1, 3))
        assert np.array_equal(ph, (tmax > tau).astype(np.uint8))


def test_residual_zero_where_phi_zero(orc):
    xb = make_activation(ActSpec(64, 256, "normal", chan_count=3, chan_scale=64.0, seed=7))
    q = orc.quantize_act(xb, mode=orc.PHI_AMAX, tau=20.0, p_s=16, r_s=64)
    ph = q["phi"]
    assert 0 < ph.sum() < ph.size
    full = orc.quantize_act(xb, mode=orc.PHI_ALL)
    for m in range(64):
        for b in range(256 // 32):
            on = ph[m // 16, (b * 32) // 64]
            cs = slice(b * 16, b * 16 + 16)
            if on:
                assert np.array_equal(q["res_codes"][m, cs], full["res_codes"][m, cs])
                assert q["res_scales"][m, b] == full["res_scales"][m, b]
            else:
                assert not q["res_codes"][m, cs].any() and q["res_scales"][m, b] == 0
