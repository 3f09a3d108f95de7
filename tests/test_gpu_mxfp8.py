"""GPU parity of the MXFP8 (E4M3) path against the CPU oracle: the MXFP8
quantizers, the FP4-to-FP8 residual pathway (Sec. 4.2, Sec. 4.3), the exact
MXFP4 -> MXFP8 re-encoding and the kind::mxf8f6f4 GEMM (W8A8, W4A8 and
RFQ with an FP8 residual).  Codes and scale bytes bit for bit; Y within the
GEMM tolerance of check_y."""
import numpy as np
import pytest
import torch

from gpu_util import DEV, check_y, qtensor_host, to_dev_bf16, guarded_full
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import WORKLOADS, ActSpec, f32_to_bf16_bits, make_activation, make_weight

pytestmark = pytest.mark.gpu
F4, F8 = rfq.RFQ_FMT_MXFP4, rfq.RFQ_FMT_MXFP8
MMA, ROW = rfq.RFQ_SCALE_MMA, rfq.RFQ_SCALE_ROWMAJOR


def _poison(*qs):
    for q in qs:
        if q is not None:
            q.codes.fill_(0xAB)
            q.scales.fill_(0xAB)


def _diff(a, b):
    idx = np.argwhere(a != b)
    return f"{len(idx)} mismatches, first at {idx[:5].tolist()}: gpu {a[tuple(idx[0])]} ref {b[tuple(idx[0])]}"


def _all_bf16_patterns(k=256):
    """Every finite bf16 pattern once, in blocks of 32 sharing a range."""
    bits = np.arange(65536, dtype=np.uint32)
    x = (bits << 16).view(np.float32)
    fin = bits[np.isfinite(x)].astype(np.uint16)
    rng = np.random.default_rng(0)
    fin = rng.permutation(fin)
    n = -(-len(fin) // k) * k
    return np.concatenate([fin, np.zeros(n - len(fin), np.uint16)]).reshape(-1, k)


def _sweep_blocks():
    """Blocks whose leading element fixes the block exponent e (448 x 2^e
    ... 511.9 x 2^e) while the others walk every bf16 significand through
    the E4M3 grid, across the whole exponent range."""
    ys = []
    for ex in range(-12, 9):
        for mant in range(128):
            ys.append((1 + mant / 128.0) * 2.0 ** ex)
    ys = np.array(ys)
    ys = np.concatenate([ys, -ys, [0.0, -0.0]])
    per = 31
    nb = -(-len(ys) // per)
    ys = np.concatenate([ys, np.zeros(nb * per - len(ys))]).reshape(nb, per)
    blocks = []
    for e in list(range(-133, -124)) + list(range(-40, 41, 9)) + list(range(112, 120)):
        lead = np.full((nb, 1), 510.0 * 2.0 ** e)
        blocks.append(np.concatenate([lead, ys * 2.0 ** e], axis=1))
    x = np.concatenate(blocks).astype(np.float32)
    x = x[np.isfinite(x).all(axis=1)]
    x = np.concatenate([x, np.zeros((-len(x) % 8, 32), np.float32)])   # whole 256-element rows
    return f32_to_bf16_bits(x.reshape(-1, 256))


@pytest.mark.parametrize("layout", [ROW, MMA])
@pytest.mark.parametrize("src", ["all_patterns", "sweep"])
def test_act_quant_mxfp8_bit_exact(orc, layout, src):
    xb = _all_bf16_patterns() if src == "all_patterns" else _sweep_blocks()
    M, K = xb.shape
    xq = rfq.empty_qtensor(F8, layout, M, K)
    _poison(xq)
    rfq.rfq_quantize_act(to_dev_bf16(xb), xq, None, None, mode=rfq.RFQ_FALLBACK_NONE)
    ref = orc.quantize_act(xb, orc.FMT_MXFP8, orc.PHI_NONE)
    mc, ms = qtensor_host(xq)
    assert np.array_equal(ms, ref["main_scales"]), _diff(ms, ref["main_scales"])
    assert np.array_equal(mc, ref["main_codes"]), _diff(mc, ref["main_codes"])


@pytest.mark.parametrize("layout", [ROW, MMA])
@pytest.mark.parametrize("mode,tau,r_s", [(rfq.RFQ_FALLBACK_ALL, 0.0, 256), (rfq.RFQ_FALLBACK_AMAX, 30.0, 128),
                                          (rfq.RFQ_FALLBACK_AMAX, 30.0, 256)])
def test_act_quant_fp8_residual_bit_exact(orc, layout, mode, tau, r_s):
    """X~ = Q_MXFP4(X) and X^ = Q_MXFP8(X - X~) in one pass (with phi; on
    128 x 256 tiles phi is computed in the same pass)."""
    for xb in (_all_bf16_patterns(), make_activation(ActSpec(300, 1024, "normal", chan_count=3, chan_scale=64.0,
                                                             tok_count=2, tok_scale=200.0, seed=7))):
        M, K = xb.shape
        xq = rfq.empty_qtensor(F4, layout, M, K)
        xr = rfq.empty_qtensor(F8, layout, M, K)
        phi = torch.empty(((M + 127) // 128) * ((K + r_s - 1) // r_s), dtype=torch.uint8, device=DEV)
        _poison(xq, xr)
        rfq.rfq_quantize_act(to_dev_bf16(xb), xq, xr, phi, mode=mode, tau=tau, p_s=128, r_s=r_s)
        ref = orc.quantize_act(xb, orc.FMT_MXFP4, mode, tau, 128, r_s, res_fmt=orc.FMT_MXFP8)
        mc, ms = qtensor_host(xq)
        rc, rs = qtensor_host(xr)
        assert np.array_equal(mc, ref["main_codes"]) and np.array_equal(ms, ref["main_scales"])
        assert np.array_equal(rs, ref["res_scales"]), _diff(rs, ref["res_scales"])
        assert np.array_equal(rc, ref["res_codes"]), _diff(rc, ref["res_codes"])
        assert np.array_equal(phi.cpu().numpy().reshape(ref["phi"].shape), ref["phi"])


@pytest.mark.parametrize("layout", [ROW, MMA])
def test_weight_quant_mxfp8_and_dequant(orc, layout):
    K, N = 512, 272
    wb = make_weight(K, N, seed=3)
    wb[:, 7] = f32_to_bf16_bits(np.linspace(-3e4, 3e4, K).astype(np.float32))   # one wide-range column
    wq = rfq.empty_qtensor(F8, layout, N, K)
    _poison(wq)
    rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
    rc, rs = orc.quantize_weight(wb, orc.FMT_MXFP8)
    wc, ws = qtensor_host(wq)
    assert np.array_equal(ws, rs) and np.array_equal(wc, rc), _diff(wc, rc)
    out = torch.empty(N, K, dtype=torch.float32, device=DEV)
    rfq.rfq_dequant(wq, out)
    assert np.array_equal(out.cpu().numpy().astype(np.float64), orc.dequant(orc.FMT_MXFP8, rc, rs, N, K))


@pytest.mark.parametrize("layout", [ROW, MMA])
def test_convert_mxfp4_to_mxfp8_is_exact(orc, layout):
    xb = _all_bf16_patterns()
    M, K = xb.shape
    x4 = rfq.empty_qtensor(F4, layout, M, K)
    rfq.rfq_quantize_act(to_dev_bf16(xb), x4, None, None, mode=rfq.RFQ_FALLBACK_NONE)
    x8 = rfq.empty_qtensor(F8, layout, M, K)
    _poison(x8)
    rfq.rfq_convert(x4, x8)
    c4, s4 = qtensor_host(x4)
    c8, s8 = qtensor_host(x8)
    assert np.array_equal(s8, s4)
    # every E4M3 code is the oracle's E4M3 encoding of the E2M1 code's value
    e4 = np.array([orc.e4m3_encode(orc.e2m1_decode(c)) for c in range(16)], np.uint8)
    lo, hi = c4 & 0xF, c4 >> 4
    want = np.stack([e4[lo], e4[hi]], axis=2).reshape(M, K)
    assert np.array_equal(c8, want)
    assert np.array_equal(orc.dequant(orc.FMT_MXFP8, c8, s8, M, K), orc.dequant(orc.FMT_MXFP4, c4, s4, M, K))


@pytest.mark.parametrize("layout,mode,tau", [(MMA, rfq.RFQ_FALLBACK_ALL, 0.0), (ROW, rfq.RFQ_FALLBACK_ALL, 0.0),
                                             (MMA, rfq.RFQ_FALLBACK_AMAX, 30.0)])
def test_quantize_act_expand_fp8_residual(orc, layout, mode, tau):
    """The FP4-to-FP8 quantizer writing X~ re-encoded as MXFP8 in the same
    pass: the E4M3 codes are the oracle's E4M3 encoding of each E2M1 value,
    the scale bytes those of X~, and X~ and X^ are the oracle's bit for bit.
    Every finite bf16 pattern (255 rows of 256: M % 128 != 0)."""
    xb = _all_bf16_patterns()
    M, K = xb.shape
    x4 = rfq.empty_qtensor(F4, layout, M, K)
    xr = rfq.empty_qtensor(F8, layout, M, K)
    x8 = rfq.empty_qtensor(F8, layout, M, K)
    _poison(x4, xr, x8)
    phi = torch.empty(((M + 127) // 128) * (K // 256), dtype=torch.uint8, device=DEV)
    rfq.rfq_quantize_act_expand(to_dev_bf16(xb), x4, xr, x8, None, phi, mode=mode, tau=tau)
    torch.cuda.synchronize()
    ref = orc.quantize_act(xb, orc.FMT_MXFP4, mode, tau, 128, 256, res_fmt=orc.FMT_MXFP8)
    c4, s4 = qtensor_host(x4)
    cr, sr = qtensor_host(xr)
    assert np.array_equal(c4, ref["main_codes"]), _diff(c4, ref["main_codes"])
    assert np.array_equal(s4, ref["main_scales"]), _diff(s4, ref["main_scales"])
    assert np.array_equal(cr, ref["res_codes"]), _diff(cr, ref["res_codes"])
    assert np.array_equal(sr, ref["res_scales"]), _diff(sr, ref["res_scales"])
    c8, s8 = qtensor_host(x8)
    assert np.array_equal(s8, s4)
    e4 = np.array([orc.e4m3_encode(orc.e2m1_decode(c)) for c in range(16)], np.uint8)
    want = np.stack([e4[c4 & 0xF], e4[c4 >> 4]], axis=2).reshape(M, K)
    assert np.array_equal(c8, want), _diff(c8, want)
    if layout == MMA:   # padding rows of the tensor-core scale layout hold zeros
        from gpu_util import mma_scale_to_rowmajor
        full = mma_scale_to_rowmajor(x8.scales.cpu().numpy(), -(-M // 128) * 128, K)
        assert not full[M:].any()


def _gemm_case(orc, M, K, N, kind, out=rfq.RFQ_OUT_F32, mode=rfq.RFQ_FALLBACK_ALL, tau=0.0, r_s=256, seed=1,
               rows=None, xb=None, wb=None, packed_w=False):
    """kind: 'w8a8', 'w4a8', 'rfq8' (MXFP4 main + MXFP8 residual, both
    products on the FP8 path) or 'rfq8mix' (the same RFQ through
    rfq_linear_mixed: the main product on the FP4 path, the residual on the
    FP8 one).  packed_w (w4a8, rfq8): W~ passed as MXFP4 (multiplied as
    E2M1 from its packed codes) instead of its E4M3 re-encoding."""
    if xb is None:
        xb = make_activation(ActSpec(M, K, "normal", chan_count=3, chan_scale=64.0, tok_count=1, tok_scale=200.0,
                                     seed=seed))
    if wb is None:
        wb = make_weight(K, N, seed=seed + 1)
    x = to_dev_bf16(xb)
    w = to_dev_bf16(wb)
    ws = torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)
    y = guarded_full((M, N), float("nan"), torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16)
    phi = None
    if kind == "w8a8":
        wq = rfq.empty_qtensor(F8, MMA, N, K)
        rfq.rfq_quantize_weight(w, wq)
        wref = orc.quantize_weight(wb, orc.FMT_MXFP8)
        w_fmt = orc.FMT_MXFP8
    else:
        w4 = rfq.empty_qtensor(F4, MMA, N, K)
        rfq.rfq_quantize_weight(w, w4)
        if packed_w:
            wq = w4
        else:
            wq = rfq.empty_qtensor(F8, MMA, N, K)
            rfq.rfq_convert(w4, wq)
        wref = orc.quantize_weight(wb, orc.FMT_MXFP4)
        w_fmt = orc.FMT_MXFP4
    if kind in ("w8a8", "w4a8"):
        xq = rfq.empty_qtensor(F8, MMA, M, K)
        rfq.rfq_quantize_act(x, xq, None, None, mode=rfq.RFQ_FALLBACK_NONE)
        rfq.rfq_linear(xq, None, None, 256, wq, y, out, ws)
        q = orc.quantize_act(xb, orc.FMT_MXFP8, orc.PHI_NONE)
        sel = slice(None) if rows is None else rows
        ref = orc.linear(orc.FMT_MXFP8, q["main_codes"][sel], q["main_scales"][sel], None, None, *wref,
                         len(q["main_codes"][sel]), K, N, w_fmt=w_fmt)
    else:
        x4 = rfq.empty_qtensor(F4, MMA, M, K)
        xr = rfq.empty_qtensor(F8, MMA, M, K)
        phi = torch.empty(((M + 127) // 128) * ((K + r_s - 1) // r_s), dtype=torch.uint8, device=DEV)
        rfq.rfq_quantize_act(x, x4, xr, phi, mode=mode, tau=tau, p_s=128, r_s=r_s)
        if kind == "rfq8mix":
            rfq.rfq_linear_mixed(x4, xr, phi if mode == rfq.RFQ_FALLBACK_AMAX else None, r_s, w4, y, out, ws)
        else:
            xq = rfq.empty_qtensor(F8, MMA, M, K)
            rfq.rfq_convert(x4, xq)
            rfq.rfq_linear(xq, xr, phi if mode == rfq.RFQ_FALLBACK_AMAX else None, r_s, wq, y, out, ws)
        q = orc.quantize_act(xb, orc.FMT_MXFP4, mode, tau, 128, r_s, res_fmt=orc.FMT_MXFP8)
        sel = slice(None) if rows is None else rows
        ref = orc.linear(orc.FMT_MXFP4, q["main_codes"][sel], q["main_scales"][sel], q["res_codes"][sel],
                         q["res_scales"][sel], *wref, len(q["main_codes"][sel]), K, N, res_fmt=orc.FMT_MXFP8,
                         w_fmt=w_fmt)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    yh = y.float().cpu().numpy()
    check_y(yh if rows is None else yh[rows], ref, bf16=(out == rfq.RFQ_OUT_BF16))
    return yh


@pytest.mark.parametrize("kind", ["w8a8", "w4a8", "rfq8", "rfq8mix"])
@pytest.mark.parametrize("M,K,N", [(1, 128, 16), (128, 512, 256), (129, 384, 272), (300, 640, 528),
                                   (513, 1024, 784)])
def test_linear_mxfp8_shapes(orc, kind, M, K, N):
    _gemm_case(orc, M, K, N, kind, seed=M + N)


@pytest.mark.parametrize("kind", ["w4a8", "rfq8"])
@pytest.mark.parametrize("M,K,N", [(1, 128, 16), (129, 384, 272), (300, 640, 528), (513, 1024, 784)])
def test_linear_packed_mxfp4_weight(orc, kind, M, K, N):
    """MXFP8 activations times an MXFP4 W~ multiplied as E2M1 from its
    packed codes (the padded 4-bit copy), against the oracle."""
    _gemm_case(orc, M, K, N, kind, seed=M + N + 7, packed_w=True)


@pytest.mark.parametrize("kind", ["rfq8", "rfq8mix", "rfq8w4"])
@pytest.mark.parametrize("r_s,tau", [(128, 30.0), (256, 30.0), (256, 1e30)])
def test_linear_fp8_residual_selective_phi(orc, kind, r_s, tau):
    _gemm_case(orc, 384, 1152, 512, kind.replace("w4", ""), mode=rfq.RFQ_FALLBACK_AMAX, tau=tau, r_s=r_s, seed=11,
               packed_w=kind.endswith("w4"))


@pytest.mark.parametrize("kind", ["rfq8", "rfq8mix"])
def test_linear_mxfp8_bf16_output(orc, kind):
    _gemm_case(orc, 256, 1024, 512, kind, out=rfq.RFQ_OUT_BF16, seed=5)


def test_mixed_rate_matches_all_e4m3_path(orc):
    """The ways of multiplying the FP4-to-FP8 RFQ give the same Y up to fp32
    accumulation order: every product is exact in each (E2M1 values are E4M3
    values), so all match the oracle and each other within the tolerance,
    on ragged shapes with more tiles than CTA pairs.  (W~ as E2M1 or as
    E4M3 gives the same exact products, but the tensor core's summation
    inside one MMA differs between the operand types, so Y is not
    bit-identical.)"""
    M, K, N = 1000, 1280, 1040
    y8 = _gemm_case(orc, M, K, N, "rfq8", seed=21)
    y8w4 = _gemm_case(orc, M, K, N, "rfq8", seed=21, packed_w=True)
    ym = _gemm_case(orc, M, K, N, "rfq8mix", seed=21)
    check_y(ym, y8)
    check_y(y8w4, y8)


def test_mixed_rate_host_checks():
    """rfq_linear_mixed wants MXFP4 X~ and W~, an MXFP8 X^ and one K; W~'s
    codes need only the 16-byte alignment of every operand (its padded copy
    is made in shared memory), so a 16-byte offset computes as the aligned
    tensor does."""
    M, K, N = 256, 256, 256
    x4, w4 = rfq.empty_qtensor(F4, MMA, M, K), rfq.empty_qtensor(F4, MMA, N, K)
    x8, w8 = rfq.empty_qtensor(F8, MMA, M, K), rfq.empty_qtensor(F8, MMA, N, K)
    y = torch.empty(M, N, device=DEV)
    ws = torch.zeros(64, dtype=torch.int32, device=DEV)
    for args in ((x8, x8, w4), (x4, x4, w4), (x4, x8, w8)):
        with pytest.raises(rfq.RFQError) as e:
            rfq.rfq_linear_mixed(args[0], args[1], None, 256, args[2], y, rfq.RFQ_OUT_F32, ws)
        assert e.value.status == rfq.RFQ_ERR_INVALID_ARG
    with pytest.raises(rfq.RFQError) as e:
        rfq.rfq_linear_mixed(x4, x8, None, 256, rfq.empty_qtensor(F4, MMA, N, 512), y, rfq.RFQ_OUT_F32, ws)
    assert e.value.status == rfq.RFQ_ERR_SHAPE
    # the same W~ codes 16 bytes off a 32-byte boundary give the same Y
    x = to_dev_bf16(make_activation(ActSpec(M, K, "normal", seed=3)))
    rfq.rfq_quantize_weight(to_dev_bf16(make_weight(K, N, seed=4)), w4)
    rfq.rfq_quantize_act(x, x4, x8, None)
    buf = torch.zeros(w4.codes.numel() + 16, dtype=torch.uint8, device=DEV)
    assert buf.data_ptr() % 32 == 0
    buf[16:].copy_(w4.codes)
    w_off = rfq.QTensor(w4.fmt, w4.scale_layout, N, K, buf[16:], w4.scales)
    y0, y1 = torch.empty(M, N, device=DEV), torch.empty(M, N, device=DEV)
    rfq.rfq_linear_mixed(x4, x8, None, 256, w4, y0, rfq.RFQ_OUT_F32, ws)
    rfq.rfq_linear_mixed(x4, x8, None, 256, w_off, y1, rfq.RFQ_OUT_F32, ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    assert torch.equal(y0, y1)


def test_fp8_residual_is_closer_than_fp4_residual(orc):
    """The point of the FP4-to-FP8 pathway: on the same X and W, the RFQ
    product with an MXFP8 residual is closer to X W (in fp64) than the one
    with an MXFP4 residual, which is closer than plain W4A4."""
    M, K, N = 256, 1024, 256
    xb = make_activation(ActSpec(M, K, "normal", chan_count=3, chan_scale=64.0, seed=13))
    wb = make_weight(K, N, seed=13)
    xf = orc.bf16_bits_to_f64(xb)
    wc, wsf = orc.quantize_weight(wb, orc.FMT_MXFP4)
    w = orc.dequant(orc.FMT_MXFP4, wc, wsf, N, K)
    exact = xf @ w.T
    y8 = _gemm_case(orc, M, K, N, "rfq8", xb=xb, wb=wb)
    # the same activation through the MXFP4 pathways, from the oracle
    q4 = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_ALL)
    y4 = orc.linear(orc.FMT_MXFP4, q4["main_codes"], q4["main_scales"], q4["res_codes"], q4["res_scales"], wc, wsf,
                    M, K, N)
    y0 = orc.linear(orc.FMT_MXFP4, q4["main_codes"], q4["main_scales"], None, None, wc, wsf, M, K, N)
    e8, e4, e0 = (np.linalg.norm(v - exact) for v in (y8, y4, y0))
    assert e8 < e4 < e0, (e8, e4, e0)


@pytest.mark.parametrize("kind", ["w4a8", "rfq8", "rfq8mix"])
def test_full_size_wan_ffn_up_mxfp8(orc, kind):
    spec = WORKLOADS["wan_ffn_up"]
    M, K, N = spec.act.M, spec.act.K, spec.N
    rows = np.unique(np.concatenate([np.random.default_rng(2).choice(M, 6, replace=False), [0, M - 1]]))
    # the activation generator of the workload, through the same helper
    xb = make_activation(spec.act)
    wb = make_weight(K, N, seed=spec.act.seed)
    x, w = to_dev_bf16(xb), to_dev_bf16(wb)
    ws = torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)
    y = torch.empty(M, N, dtype=torch.bfloat16, device=DEV)
    w4 = rfq.empty_qtensor(F4, MMA, N, K)
    rfq.rfq_quantize_weight(w, w4)
    w8 = rfq.empty_qtensor(F8, MMA, N, K)
    rfq.rfq_convert(w4, w8)
    wref = orc.quantize_weight(wb, orc.FMT_MXFP4)
    if kind == "w4a8":
        xq = rfq.empty_qtensor(F8, MMA, M, K)
        rfq.rfq_quantize_act(x, xq, None, None, mode=rfq.RFQ_FALLBACK_NONE)
        rfq.rfq_linear(xq, None, None, 256, w8, y, rfq.RFQ_OUT_BF16, ws)
        q = orc.quantize_act(xb[rows], orc.FMT_MXFP8, orc.PHI_NONE)
        ref = orc.linear(orc.FMT_MXFP8, q["main_codes"], q["main_scales"], None, None, *wref, len(rows), K, N,
                         w_fmt=orc.FMT_MXFP4)
    else:
        x4 = rfq.empty_qtensor(F4, MMA, M, K)
        xr = rfq.empty_qtensor(F8, MMA, M, K)
        rfq.rfq_quantize_act(x, x4, xr, None)
        if kind == "rfq8mix":
            rfq.rfq_linear_mixed(x4, xr, None, 256, w4, y, rfq.RFQ_OUT_BF16, ws)
        else:
            xq = rfq.empty_qtensor(F8, MMA, M, K)
            rfq.rfq_convert(x4, xq)
            rfq.rfq_linear(xq, xr, None, 256, w8, y, rfq.RFQ_OUT_BF16, ws)
        q = orc.quantize_act(xb[rows], orc.FMT_MXFP4, orc.PHI_ALL, res_fmt=orc.FMT_MXFP8)
        ref = orc.linear(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"], *wref,
                         len(rows), K, N, res_fmt=orc.FMT_MXFP8, w_fmt=orc.FMT_MXFP4)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    check_y(y.float().cpu().numpy()[rows], ref, bf16=True)
