"""GPU parity of the HiF4 path (Sec. 3.3) against the CPU oracle: codes and
metadata words bit-exact, dequantized values exact, and the RFQ GEMM with
HiF4 activations within the Y tolerance."""
import numpy as np
import pytest
import torch

from gpu_util import DEV, check_y, qtensor_host, to_dev_bf16, guarded_full
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import WORKLOADS, ActSpec, f32_to_bf16_bits, make_activation, make_weight

pytestmark = pytest.mark.gpu
H = rfq.RFQ_FMT_HIF4


def _diff(a, b):
    idx = np.argwhere(a != b)
    return f"{len(idx)} mismatches, first at {idx[:5].tolist()}: gpu {a[tuple(idx[0])]:#x} ref {b[tuple(idx[0])]:#x}"


def _quant(xb, layout, mode=rfq.RFQ_FALLBACK_ALL, tau=0.0, p_s=128, r_s=256):
    M, K = xb.shape
    x = to_dev_bf16(xb)
    xq = rfq.empty_qtensor(H, layout, M, K)
    xr = rfq.empty_qtensor(H, layout, M, K) if mode != rfq.RFQ_FALLBACK_NONE else None
    for q in (xq, xr):
        if q is not None:
            q.codes.fill_(0xAB); q.scales.fill_(0xAB)
    phi = torch.empty(((M + p_s - 1) // p_s) * ((K + r_s - 1) // r_s), dtype=torch.uint8, device=DEV)
    rfq.rfq_quantize_act(x, xq, xr, phi, mode=mode, tau=tau, p_s=p_s, r_s=r_s)
    torch.cuda.synchronize()
    return xq, xr, phi


def _compare(orc, xb, layout, mode=rfq.RFQ_FALLBACK_ALL, tau=0.0, p_s=128, r_s=256):
    xq, xr, phi = _quant(xb, layout, mode, tau, p_s, r_s)
    ref = orc.quantize_act(xb, orc.FMT_HIF4, mode, tau, p_s, r_s)
    mc, mm = qtensor_host(xq)
    assert np.array_equal(mm, ref["main_scales"]), _diff(mm, ref["main_scales"])
    assert np.array_equal(mc, ref["main_codes"]), _diff(mc, ref["main_codes"])
    if xr is not None:
        rc, rm = qtensor_host(xr)
        assert np.array_equal(rm, ref["res_scales"]), _diff(rm, ref["res_scales"])
        assert np.array_equal(rc, ref["res_codes"]), _diff(rc, ref["res_codes"])
    return xq, xr


def test_every_bf16_pattern(orc):
    bits = np.arange(1 << 16, dtype=np.uint32)
    f = (bits << 16).view(np.float32)
    fin = bits[np.isfinite(f)].astype(np.uint16)
    rng = np.random.default_rng(0)
    shuffled = rng.permutation(fin)
    by_mag = fin[np.argsort(np.abs((fin.astype(np.uint32) << 16).view(np.float32)), kind="stable")]
    xs = np.concatenate([shuffled, by_mag])
    xs = xs[: len(xs) // 512 * 512].reshape(-1, 512)
    _compare(orc, xs, rfq.RFQ_SCALE_ROWMAJOR)


def test_scale_boundaries(orc):
    # blocks whose amax sits on and around every 7 S threshold of the macro
    # scale, across the whole UE6M2 range and beyond (saturation)
    rows = []
    for E in list(range(0, 64, 3)) + [63]:
        for Mm in range(4):
            S = 2.0 ** (E - 48) * (1 + Mm / 4)
            for f in (1.0, 1.0 + 2 ** -7, 1.0 - 2 ** -8, 0.5, 0.26, 0.125):
                blk = np.linspace(-1, 1, 64) * 7 * S * f
                blk[5] = 7 * S * f
                rows.append(blk)
    rows.append(np.full(64, 3.0e38))
    rows.append(np.full(64, 1e-40))
    x = np.array(rows).reshape(-1, 256).astype(np.float32) if len(rows) % 4 == 0 else \
        np.array(rows + [np.zeros(64)] * (4 - len(rows) % 4)).reshape(-1, 256).astype(np.float32)
    xb = f32_to_bf16_bits(x)
    _compare(orc, xb, rfq.RFQ_SCALE_ROWMAJOR)


@pytest.mark.parametrize("M,K", [(1, 64), (3, 192), (127, 256), (129, 640), (300, 12288)])
def test_shapes_both_layouts(orc, M, K):
    xb = make_activation(ActSpec(M, K, "laplace", body_scale=0.3, chan_count=max(1, K // 100), chan_scale=50.0,
                                 seed=M + K))
    _compare(orc, xb, rfq.RFQ_SCALE_ROWMAJOR)
    _compare(orc, xb, rfq.RFQ_SCALE_MMA)


def test_degenerate_blocks(orc):
    x = np.zeros((6, 256), np.float32)
    x[1] = -0.0
    x[2, :64] = 2.0
    x[3, 0] = 3.3895314e38; x[3, 1] = 1e-40
    x[4] = 2.0 ** -133
    x[5, ::2] = 0.125; x[5, 1::2] = -0.375
    _compare(orc, f32_to_bf16_bits(x), rfq.RFQ_SCALE_ROWMAJOR)


def _tie_blocks(seed=0):
    """64-element blocks whose elements sit on and next to the midpoints of
    the S1P2 grid: per block a macro scale S (one element 7 S, so S is that
    block's scale), the other elements +-(j + 1/2) or +-j steps of 0.25 S 2^ex
    for random j and ex in {0, 1, 2} (bf16-exact: at most 7 significant
    bits), some moved by one bf16 ulp; sub-groups then take exponents that
    make many of them exact ties of their own grid."""
    rng = np.random.default_rng(seed)
    rows = []
    for E in (0, 5, 20, 47, 48, 49, 60, 63):
        for Mm in range(4):
            S = 2.0 ** (E - 48) * (1 + Mm / 4)
            for _ in range(24):
                j = rng.integers(0, 7, 64)
                ex = rng.integers(0, 3, 64)
                half = rng.random(64) < 0.75
                blk = (j + np.where(half, 0.5, 0.0)) * 0.25 * S * 2.0 ** ex
                blk *= np.where(rng.random(64) < 0.5, -1.0, 1.0)
                blk[rng.integers(0, 64)] = 7 * S
                bits = f32_to_bf16_bits(blk.astype(np.float32)).astype(np.int32)
                nudge = rng.choice([-1, 0, 0, 0, 1], 64)
                nz = (bits & 0x7FFF) > 1
                bits = np.where(nz, bits + nudge, bits)
                rows.append(bits.astype(np.uint16))
    return np.array(rows).reshape(-1, 256)


def test_rounding_ties_to_even(orc):
    """Elements exactly halfway between two grid points round to the even k
    (the oracle's exact rounding), in both metadata layouts, for the
    activation quantizer (main and residual) and the weight quantizer."""
    xb = _tie_blocks()
    # the blocks do hold exact ties: |x| / step a half-integer for the
    # element's own step (decoded from the oracle's metadata words)
    ref = orc.quantize_act(xb, orc.FMT_HIF4, orc.PHI_ALL, 0.0, 128, 256)
    x = np.abs((xb.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
    meta = ref["main_scales"].reshape(xb.shape[0], -1).astype(np.int64)
    sb = meta & 0xFF
    S = np.exp2((sb >> 2) - 48.0) * (1 + (sb & 3) / 4)
    i = np.arange(256) % 64
    e18 = (np.repeat(meta, 64, axis=1) >> (8 + i // 8)) & 1
    e116 = (np.repeat(meta, 64, axis=1) >> (16 + i // 4)) & 1
    step = 0.25 * np.repeat(S, 64, axis=1) * np.exp2(e18 + e116)
    q = x / step
    ties = np.sum((q - np.floor(q) == 0.5) & (q < 7))
    assert ties > 1000, ties
    for layout in (rfq.RFQ_SCALE_ROWMAJOR, rfq.RFQ_SCALE_MMA):
        _compare(orc, xb, layout)
    # the same values as a weight [K x N] (quantized along K)
    wb = np.ascontiguousarray(xb[:64].T)
    wq = rfq.empty_qtensor(H, rfq.RFQ_SCALE_ROWMAJOR, 64, 256)
    rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
    torch.cuda.synchronize()
    c, m = qtensor_host(wq)
    rc, rm = orc.quantize_weight(wb, orc.FMT_HIF4)
    assert np.array_equal(m, rm), _diff(m, rm)
    assert np.array_equal(c, rc), _diff(c, rc)


@pytest.mark.parametrize("mode,tau,r_s", [(rfq.RFQ_FALLBACK_NONE, 0.0, 256), (rfq.RFQ_FALLBACK_AMAX, 20.0, 128),
                                          (rfq.RFQ_FALLBACK_AMAX, 10.0, 64), (rfq.RFQ_FALLBACK_AMAX, 20.0, 256)])
def test_phi_modes(orc, mode, tau, r_s):
    """AMAX on 128 x 256 tiles runs the fused kernel (phi computed in the
    quantizer's pass); other tile widths the separate phi pass."""
    xb = make_activation(ActSpec(300, 1024, "laplace", body_scale=0.3, chan_count=5, chan_scale=50.0, seed=3))
    _compare(orc, xb, rfq.RFQ_SCALE_MMA, mode=mode, tau=tau, r_s=r_s)


@pytest.mark.parametrize("layout", [rfq.RFQ_SCALE_MMA, rfq.RFQ_SCALE_ROWMAJOR])
@pytest.mark.parametrize("M,K", [(1, 256), (200, 768)])
def test_phi_amax_fused_tiles(orc, layout, M, K):
    """The fused AMAX quantizer on ragged rows, tau set to tile (0, 0)'s own
    max |x| (phi is strict: that tile keeps no residual)."""
    xb = make_activation(ActSpec(M, K, "laplace", body_scale=0.3, chan_count=4, chan_scale=50.0, seed=M + K))
    x = (xb.astype(np.uint32) << 16).view(np.float32)
    tau = float(np.abs(x[:128, :256]).max())
    _compare(orc, xb, layout, mode=rfq.RFQ_FALLBACK_AMAX, tau=tau, r_s=256)
    _, _, phi = _quant(xb, layout, rfq.RFQ_FALLBACK_AMAX, tau, 128, 256)
    assert phi[0].item() == 0


@pytest.mark.parametrize("K,N", [(64, 16), (640, 272), (12288, 64)])
def test_weight_quant(orc, K, N):
    wb = make_weight(K, N, seed=K + N)
    for layout in (rfq.RFQ_SCALE_ROWMAJOR, rfq.RFQ_SCALE_MMA):
        wq = rfq.empty_qtensor(H, layout, N, K)
        rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
        torch.cuda.synchronize()
        c, m = qtensor_host(wq)
        rc, rm = orc.quantize_weight(wb, orc.FMT_HIF4)
        assert np.array_equal(m, rm), _diff(m, rm)
        assert np.array_equal(c, rc), _diff(c, rc)


def test_dequant_fp32_and_bf16_exact(orc):
    xb = make_activation(ActSpec(130, 640, "laplace", body_scale=0.3, chan_count=3, chan_scale=50.0, seed=7))
    for layout in (rfq.RFQ_SCALE_ROWMAJOR, rfq.RFQ_SCALE_MMA):
        xq, xr, _ = _quant(xb, layout)
        for q in (xq, xr):
            c, m = qtensor_host(q)
            ref = orc.dequant(orc.FMT_HIF4, c, m, 130, 640)
            for dt in (torch.float32, torch.bfloat16):
                out = torch.empty(130, 640, dtype=dt, device=DEV)
                rfq.rfq_dequant(q, out)
                torch.cuda.synchronize()
                assert np.array_equal(out.double().cpu().numpy(), ref)


@pytest.mark.parametrize("mode,tau,r_s,layout", [
    (rfq.RFQ_FALLBACK_ALL, 0.0, 256, rfq.RFQ_SCALE_MMA), (rfq.RFQ_FALLBACK_ALL, 0.0, 256, rfq.RFQ_SCALE_ROWMAJOR),
    (rfq.RFQ_FALLBACK_NONE, 0.0, 256, rfq.RFQ_SCALE_MMA), (rfq.RFQ_FALLBACK_AMAX, 10.0, 128, rfq.RFQ_SCALE_MMA),
    (rfq.RFQ_FALLBACK_AMAX, 10.0, 256, rfq.RFQ_SCALE_MMA), (rfq.RFQ_FALLBACK_AMAX, 10.0, 256, rfq.RFQ_SCALE_ROWMAJOR)])
def test_quantize_act_expand(orc, mode, tau, r_s, layout):
    """The quantizer's own bf16 values of X~ and X^ are bit for bit the
    oracle's dequantization of its codes (Sec. 3.3 decoder), with X^ zero on
    phi = 0 tiles; the codes and metadata are those of rfq_quantize_act."""
    M, K = 300, 1024
    xb = make_activation(ActSpec(M, K, "laplace", body_scale=0.3, chan_count=5, chan_scale=50.0, seed=13))
    xb[7, :64] = 0                                   # an all-zero block
    xb[9, 64] = 0x8000                               # a negative zero
    x = to_dev_bf16(xb)
    res = mode != rfq.RFQ_FALLBACK_NONE
    xq = rfq.empty_qtensor(H, layout, M, K)
    xr = rfq.empty_qtensor(H, layout, M, K) if res else None
    xq16 = rfq.empty_bf16_operand(M, K)
    xr16 = rfq.empty_bf16_operand(M, K) if res else None
    for t in (xq16, xr16):
        if t is not None:
            t.codes.fill_(float("nan"))
    phi = torch.empty(((M + 127) // 128) * ((K + r_s - 1) // r_s), dtype=torch.uint8, device=DEV)
    rfq.rfq_quantize_act_expand(x, xq, xr, xq16, xr16, phi, mode=mode, tau=tau, p_s=128, r_s=r_s)
    torch.cuda.synchronize()
    ref = orc.quantize_act(xb, orc.FMT_HIF4, mode, tau, 128, r_s)
    mc, mm = qtensor_host(xq)
    assert np.array_equal(mc, ref["main_codes"]) and np.array_equal(mm, ref["main_scales"])
    pairs = [(xq16, ref["main_codes"], ref["main_scales"])]
    if res:
        rc, rm = qtensor_host(xr)
        assert np.array_equal(rc, ref["res_codes"]) and np.array_equal(rm, ref["res_scales"])
        pairs.append((xr16, ref["res_codes"], ref["res_scales"]))
    for t, c, m in pairs:
        want = orc.dequant(orc.FMT_HIF4, c, m, M, K)
        got = t.codes.view(torch.int16).cpu().numpy().view(np.uint16)
        assert np.array_equal(got, f32_to_bf16_bits(want.astype(np.float32))), "bf16 values differ"
        assert np.array_equal(np.signbit(got.view(np.int16)), np.signbit(want)), "signs of zero differ"


def _expand(q):
    t = rfq.empty_bf16_operand(q.rows, q.k)
    rfq.rfq_dequant(q, t.codes)
    return t


def _linear(xb, wb, out=rfq.RFQ_OUT_F32, mode=rfq.RFQ_FALLBACK_ALL, tau=0.0, r_s=256, use_phi=False,
            expand=False):
    M, K = xb.shape
    N = wb.shape[1]
    wq = rfq.empty_qtensor(H, rfq.RFQ_SCALE_ROWMAJOR, N, K)
    rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
    w16 = rfq.empty_bf16_operand(N, K)
    rfq.rfq_dequant(wq, w16.codes)
    xq, xr, phi = _quant(xb, rfq.RFQ_SCALE_MMA, mode, tau, 128, r_s)
    y = guarded_full((M, N), float("nan"), torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16)
    ws = torch.zeros(64, dtype=torch.int32, device=DEV)
    a, r = (_expand(xq), _expand(xr) if xr is not None else None) if expand else (xq, xr)
    rfq.rfq_linear(a, r, phi if use_phi else None, r_s, w16, y, out, ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    return xq, xr, wq, y.double().cpu().numpy()


def _ref(orc, xq, xr, wq, M, K, N):
    mc, mm = qtensor_host(xq)
    wc, wm = qtensor_host(wq)
    rc, rm = qtensor_host(xr) if xr is not None else (None, None)
    return orc.linear(orc.FMT_HIF4, mc, mm, rc, rm, wc, wm, M, K, N)


@pytest.mark.parametrize("expand", [False, True])
@pytest.mark.parametrize("M,K,N", [(1, 64, 16), (128, 512, 256), (129, 640, 272), (300, 1024, 528)])
def test_linear_shapes(orc, M, K, N, expand):
    xb = make_activation(ActSpec(M, K, "laplace", body_scale=0.3, chan_count=2, chan_scale=50.0, seed=M + N))
    wb = make_weight(K, N, seed=K)
    xq, xr, wq, y = _linear(xb, wb, expand=expand)
    check_y(y, _ref(orc, xq, xr, wq, M, K, N))


@pytest.mark.parametrize("expand", [False, True])
def test_linear_no_residual_and_phi(orc, expand):
    M, K, N = 256, 1024, 256
    xb = make_activation(ActSpec(M, K, "laplace", body_scale=0.3, chan_count=3, chan_scale=50.0, seed=5))
    wb = make_weight(K, N, seed=5)
    xq, xr, wq, y = _linear(xb, wb, mode=rfq.RFQ_FALLBACK_NONE, expand=expand)
    check_y(y, _ref(orc, xq, None, wq, M, K, N))
    xq, xr, wq, y = _linear(xb, wb, mode=rfq.RFQ_FALLBACK_AMAX, tau=10.0, r_s=128, use_phi=True, expand=expand)
    check_y(y, _ref(orc, xq, xr, wq, M, K, N))
    xq, xr, wq, y = _linear(xb, wb, mode=rfq.RFQ_FALLBACK_AMAX, tau=10.0, r_s=256, use_phi=True, expand=expand)
    check_y(y, _ref(orc, xq, xr, wq, M, K, N))


@pytest.mark.parametrize("expand", [False, True])
def test_phi_records_wrap(orc, expand):
    """320 output tiles (several per CTA, so the per-tile phi records wrap
    their two buffers) with a mixed phi pattern at r_s = 64."""
    M, K, N = 640, 1024, 16384
    xb = make_activation(ActSpec(M, K, "laplace", body_scale=0.3, chan_count=24, chan_scale=50.0, seed=21))
    wb = make_weight(K, N, seed=21)
    xq, xr, wq, y = _linear(xb, wb, mode=rfq.RFQ_FALLBACK_AMAX, tau=10.0, r_s=64, use_phi=True, expand=expand)
    q = orc.quantize_act(xb, orc.FMT_HIF4, orc.PHI_AMAX, 10.0, 128, 64)
    assert 0.1 < q["phi"].mean() < 0.9
    check_y(y, _ref(orc, xq, xr, wq, M, K, N))


@pytest.mark.parametrize("out,expand", [(rfq.RFQ_OUT_BF16, True), (rfq.RFQ_OUT_F32, True), (rfq.RFQ_OUT_BF16, False)])
def test_full_size_qwen_down_hif4(orc, out, expand):
    spec = WORKLOADS["qwen_down_hif4"]
    M, K, N = spec.act.M, spec.act.K, spec.N
    xb = make_activation(spec.act)
    wb = make_weight(K, N, seed=spec.act.seed)
    xq, xr, wq, y = _linear(xb, wb, out=out, expand=expand)
    wc, wm = qtensor_host(wq)
    rwc, rwm = orc.quantize_weight(wb, orc.FMT_HIF4)
    assert np.array_equal(wc, rwc) and np.array_equal(wm, rwm)
    rng = np.random.default_rng(1)
    rows = np.unique(np.concatenate([rng.choice(M, 10, replace=False), [0, M - 1]]))
    q = orc.quantize_act(xb[rows], orc.FMT_HIF4)
    mc, mm = qtensor_host(xq)
    rc, rm = qtensor_host(xr)
    assert np.array_equal(mc[rows], q["main_codes"]) and np.array_equal(mm[rows], q["main_scales"])
    assert np.array_equal(rc[rows], q["res_codes"]) and np.array_equal(rm[rows], q["res_scales"])
    ref = orc.linear(orc.FMT_HIF4, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"], rwc, rwm,
                     len(rows), K, N)
    check_y(y[rows], ref, bf16=(out == rfq.RFQ_OUT_BF16))
