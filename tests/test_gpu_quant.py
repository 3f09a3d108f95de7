"""GPU parity of the quantization kernels against the CPU oracle: every code
and scale byte must match bit for bit (Sec. 3.2 Eq. 3-4, Sec. 4.3)."""
import numpy as np
import pytest
import torch

from gpu_util import DEV, qtensor_host, to_dev_bf16
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import WORKLOADS, ActSpec, f32_to_bf16_bits, make_activation, make_weight

pytestmark = pytest.mark.gpu


def _act_quant(xb, layout, mode=rfq.RFQ_FALLBACK_ALL, tau=0.0, p_s=128, r_s=256):
    M, K = xb.shape
    x = to_dev_bf16(xb)
    xq = rfq.empty_qtensor(rfq.RFQ_FMT_MXFP4, layout, M, K)
    xr = rfq.empty_qtensor(rfq.RFQ_FMT_MXFP4, layout, M, K) if mode != rfq.RFQ_FALLBACK_NONE else None
    phi = torch.empty(((M + p_s - 1) // p_s) * ((K + r_s - 1) // r_s), dtype=torch.uint8, device=DEV)
    # poison the outputs so unwritten bytes show up
    xq.codes.fill_(0xAB); xq.scales.fill_(0xAB)
    if xr is not None:
        xr.codes.fill_(0xAB); xr.scales.fill_(0xAB)
    rfq.rfq_quantize_act(x, xq, xr, phi, mode=mode, tau=tau, p_s=p_s, r_s=r_s)
    torch.cuda.synchronize()
    return xq, xr, phi


def _compare(orc, xb, layout, mode=rfq.RFQ_FALLBACK_ALL, tau=0.0, p_s=128, r_s=256):
    xq, xr, phi = _act_quant(xb, layout, mode, tau, p_s, r_s)
    ref = orc.quantize_act(xb, orc.FMT_MXFP4, mode, tau, p_s, r_s)
    mc, ms = qtensor_host(xq)
    assert np.array_equal(mc, ref["main_codes"]), _diff(mc, ref["main_codes"])
    assert np.array_equal(ms, ref["main_scales"]), _diff(ms, ref["main_scales"])
    if xr is not None:
        rc, rs = qtensor_host(xr)
        assert np.array_equal(rs, ref["res_scales"]), _diff(rs, ref["res_scales"])
        assert np.array_equal(rc, ref["res_codes"]), _diff(rc, ref["res_codes"])
        assert np.array_equal(phi.cpu().numpy().reshape(ref["phi"].shape), ref["phi"])
    if layout == rfq.RFQ_SCALE_MMA:
        M, K = xb.shape
        pad = xq.scales.cpu().numpy()
        rows_pad = ((M + 127) // 128) * 128
        if rows_pad > M:   # padding rows of the tensor-core layout hold zeros
            from gpu_util import mma_scale_to_rowmajor
            full = mma_scale_to_rowmajor(pad, rows_pad, K)
            assert not full[M:].any()
    return xq, xr


def _diff(a, b):
    idx = np.argwhere(a != b)
    return f"{len(idx)} mismatches, first at {idx[:5].tolist()}: gpu {a[tuple(idx[0])]} ref {b[tuple(idx[0])]}"


def _sweep_blocks():
    """Blocks that walk every bf16 significand through the E2M1 grid at
    every scale exponent: element 0 of a block is 7.96875 * 2^e (so the
    block exponent is e), the rest are +-y * 2^e for all bf16 y < 8."""
    ys = []
    for ex in range(-10, 3):
        for mant in range(128):
            ys.append((1 + mant / 128.0) * 2.0 ** ex)
    ys = np.array(ys)
    ys = np.concatenate([ys, -ys, [0.0, -0.0]])
    per = 31
    nb = -(-len(ys) // per)
    ys = np.concatenate([ys, np.zeros(nb * per - len(ys))]).reshape(nb, per)
    blocks = []
    for e in list(range(-127, -118)) + list(range(-40, 41, 7)) + list(range(117, 126)):
        lead = np.full((nb, 1), 7.96875 * 2.0 ** e)
        blocks.append(np.concatenate([lead, ys * 2.0 ** e], axis=1))
    x = np.concatenate(blocks).astype(np.float32)
    return f32_to_bf16_bits(x.reshape(-1, 256))


def test_rounding_sweep_all_significands_all_scales(orc):
    xb = _sweep_blocks()
    _compare(orc, xb, rfq.RFQ_SCALE_ROWMAJOR)


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
    _compare(orc, xs, rfq.RFQ_SCALE_MMA)


@pytest.mark.parametrize("M,K", [(1, 32), (3, 96), (127, 128), (129, 384), (300, 640), (64, 5120)])
def test_ragged_shapes_rowmajor(orc, M, K):
    xb = make_activation(ActSpec(M, K, "student_t3", chan_count=max(1, K // 200), chan_scale=100.0, seed=M + K))
    _compare(orc, xb, rfq.RFQ_SCALE_ROWMAJOR)


@pytest.mark.parametrize("M,K", [(1, 128), (127, 128), (129, 384), (300, 640), (257, 5120)])
def test_ragged_shapes_mma_layout(orc, M, K):
    xb = make_activation(ActSpec(M, K, "normal", chan_count=3, chan_scale=64.0, tok_count=2, tok_scale=200.0,
                                 seed=M * 7 + K))
    _compare(orc, xb, rfq.RFQ_SCALE_MMA)


def test_zero_and_degenerate_blocks(orc):
    M, K = 8, 256
    x = np.zeros((M, K), np.float32)
    x[1] = -0.0                                   # negative zeros
    x[2, :32] = 3.0                               # all-equal block
    x[3] = np.float32(3.3895314e38)               # max bf16 everywhere
    x[4, 0] = 3.3895314e38; x[4, 1] = 1e-40       # extreme range in one block
    x[5] = 2.0 ** -133                            # smallest subnormal
    x[6, ::2] = 0.25; x[6, 1::2] = -0.75          # ties
    x[7] = np.linspace(-6, 6, K)
    xb = f32_to_bf16_bits(x)
    _compare(orc, xb, rfq.RFQ_SCALE_ROWMAJOR)
    _compare(orc, xb, rfq.RFQ_SCALE_MMA)


def test_no_residual_mode(orc):
    xb = make_activation(ActSpec(130, 256, "normal", chan_count=2, chan_scale=64.0, seed=5))
    _compare(orc, xb, rfq.RFQ_SCALE_MMA, mode=rfq.RFQ_FALLBACK_NONE)


@pytest.mark.parametrize("p_s,r_s,tau", [(128, 256, 30.0), (128, 128, 10.0), (16, 64, 20.0), (128, 512, 1e30)])
def test_phi_amax_mode(orc, p_s, r_s, tau):
    xb = make_activation(ActSpec(300, 1024, "normal", chan_count=5, chan_scale=64.0, seed=11))
    _compare(orc, xb, rfq.RFQ_SCALE_MMA, mode=rfq.RFQ_FALLBACK_AMAX, tau=tau, p_s=p_s, r_s=r_s)


@pytest.mark.parametrize("layout", [rfq.RFQ_SCALE_MMA, rfq.RFQ_SCALE_ROWMAJOR])
@pytest.mark.parametrize("M,K", [(1, 256), (200, 768), (385, 1024)])
def test_phi_amax_fused_tiles(orc, layout, M, K):
    """128 x 256 phi tiles (the GEMMs' granularity, K % 256 == 0) take the
    fused quantizer, which reduces each tile's max |x| and quantizes it in
    one pass.  tau is set to tile (0, 0)'s own max |x|: phi is a strict
    comparison (Sec. 4.3), so that tile falls back to no residual."""
    xb = make_activation(ActSpec(M, K, "student_t3", chan_count=4, chan_scale=80.0, seed=M + K))
    x = (xb.astype(np.uint32) << 16).view(np.float32)
    tau = float(np.abs(x[:128, :256]).max())
    xq, xr = _compare(orc, xb, layout, mode=rfq.RFQ_FALLBACK_AMAX, tau=tau, p_s=128, r_s=256)
    _, _, phi = _act_quant(xb, layout, rfq.RFQ_FALLBACK_AMAX, tau, 128, 256)
    assert phi[0].item() == 0


@pytest.mark.parametrize("r_s", [256, 128])
def test_phi_amax_nan_dropped_inf_kept(orc, r_s):
    """A NaN element does not count towards a tile's max |x| (the maximum
    skips it, as the oracle's comparison does) and an Inf does, both in the
    fused 128 x 256 quantizer (r_s = 256) and in the separate phi pass
    (r_s = 128).  Only phi is compared: the codes of NaN elements are not
    specified."""
    M, K, tau = 256, 512, 50.0
    xb = make_activation(ActSpec(M, K, "normal", seed=21))   # |x| < 6 here
    xb[5, 7] = 0x7FC0       # NaN in tile (0, 0)
    xb[200, 10] = 0xFFC1    # negative NaN with a payload in tile (1, 0)
    xb[130, 300] = 0x7F80   # +Inf in tile (1, 300 // r_s)
    _, _, phi = _act_quant(xb, rfq.RFQ_SCALE_MMA, rfq.RFQ_FALLBACK_AMAX, tau, 128, r_s)
    ref = orc.quantize_act(xb, orc.FMT_MXFP4, rfq.RFQ_FALLBACK_AMAX, tau, 128, r_s)["phi"]
    got = phi.cpu().numpy().reshape(ref.shape)
    assert np.array_equal(got, ref)
    want = np.zeros_like(ref)
    want[1, 300 // r_s] = 1
    assert np.array_equal(got, want)


def test_tiny_workload_both_layouts(orc):
    spec = WORKLOADS["tiny"]
    xb = make_activation(spec.act)
    _compare(orc, xb, rfq.RFQ_SCALE_ROWMAJOR)
    _compare(orc, xb, rfq.RFQ_SCALE_MMA)


@pytest.mark.parametrize("K,N", [(512, 512), (128, 16), (384, 300), (5120, 272)])
def test_weight_quant(orc, K, N):
    wb = make_weight(K, N, seed=K + N)
    w = to_dev_bf16(wb)
    for layout in (rfq.RFQ_SCALE_ROWMAJOR, rfq.RFQ_SCALE_MMA):
        if layout == rfq.RFQ_SCALE_MMA and K % 128:
            continue
        wq = rfq.empty_qtensor(rfq.RFQ_FMT_MXFP4, layout, N, K)
        wq.codes.fill_(0xAB); wq.scales.fill_(0xAB)
        rfq.rfq_quantize_weight(w, wq)
        torch.cuda.synchronize()
        c, s = qtensor_host(wq)
        rc, rs = orc.quantize_weight(wb, orc.FMT_MXFP4)
        assert np.array_equal(c, rc), _diff(c, rc)
        assert np.array_equal(s, rs), _diff(s, rs)


def test_dequant_matches_oracle(orc):
    xb = make_activation(ActSpec(200, 512, "student_t3", chan_count=3, chan_scale=100.0, seed=3))
    for layout in (rfq.RFQ_SCALE_ROWMAJOR, rfq.RFQ_SCALE_MMA):
        xq, xr, _ = _act_quant(xb, layout)
        for q in (xq, xr):
            out = torch.empty(200, 512, dtype=torch.float32, device=DEV)
            rfq.rfq_dequant(q, out)
            torch.cuda.synchronize()
            c, s = qtensor_host(q)
            ref = orc.dequant(orc.FMT_MXFP4, c, s, 200, 512)
            assert np.array_equal(out.cpu().numpy().astype(np.float64), ref)
            out16 = torch.empty(200, 512, dtype=torch.bfloat16, device=DEV)
            rfq.rfq_dequant(q, out16)
            torch.cuda.synchronize()
            assert np.array_equal(out16.double().cpu().numpy(), ref)   # in bf16's normal range: exact


def test_check_finite_flags_inf_and_nan():
    """Checked mode: rfq_check_finite records RFQ_ERR_NONFINITE for any Inf or
    NaN in X (every position class: first, last, interior element of a
    16-byte chunk), nothing for finite X (including max bf16 and -0), and a
    GEMM given that workspace computes nothing until the record is cleared."""
    M, K = 300, 640
    xb = make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, seed=12))
    xb[3, 5] = 0x7F7F      # the largest finite bf16
    xb[4, 6] = 0x8000      # -0
    ws = torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)
    rfq.rfq_check_finite(to_dev_bf16(xb), ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    for (r, c, bits) in [(0, 0, 0x7F80), (M - 1, K - 1, 0xFF80), (150, 333, 0x7FC0), (7, 1, 0xFFC1)]:
        bad = xb.copy()
        bad[r, c] = bits
        rfq.rfq_check_finite(to_dev_bf16(bad), ws)
        assert rfq.rfq_workspace_status(ws) == rfq.RFQ_ERR_NONFINITE, (r, c, hex(bits))
        # a GEMM with the flagged workspace leaves Y untouched
        N = 256
        wq = rfq.empty_qtensor(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, N, K)
        rfq.rfq_quantize_weight(to_dev_bf16(make_weight(K, N, seed=1)), wq)
        xq = rfq.empty_qtensor(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, M, K)
        rfq.rfq_quantize_act(to_dev_bf16(xb), xq, None, None, mode=rfq.RFQ_FALLBACK_NONE)
        y = torch.full((M, N), 7.0, dtype=torch.float32, device=DEV)
        rfq.rfq_linear(xq, None, None, 256, wq, y, rfq.RFQ_OUT_F32, ws)
        assert rfq.rfq_workspace_status(ws, clear=True) == rfq.RFQ_ERR_NONFINITE
        assert (y == 7.0).all()
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
