"""GPU parity of the RFQ GEMM (Algorithm 1, Eq. rfq) against the fp64 CPU
oracle.  fp32 output: relative Frobenius error <= 1e-5 and max abs error
<= 1e-3 max|Y|; bf16 output adds its own final rounding (see check_y)."""
import numpy as np
import pytest
import torch

from gpu_util import DEV, check_y, qtensor_host, to_dev_bf16, guarded_full
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import WORKLOADS, ActSpec, make_activation, make_weight

pytestmark = pytest.mark.gpu
MMA = rfq.RFQ_SCALE_MMA
FMT = rfq.RFQ_FMT_MXFP4


def _workspace():
    return torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)


def _run(xb, wb, mode=rfq.RFQ_FALLBACK_ALL, out=rfq.RFQ_OUT_F32, tau=0.0, r_s=256, use_phi=False):
    M, K = xb.shape
    N = wb.shape[1]
    x, w = to_dev_bf16(xb), to_dev_bf16(wb)
    wq = rfq.empty_qtensor(FMT, MMA, N, K)
    rfq.rfq_quantize_weight(w, wq)
    xq = rfq.empty_qtensor(FMT, MMA, M, K)
    xr = rfq.empty_qtensor(FMT, MMA, M, K) if mode != rfq.RFQ_FALLBACK_NONE else None
    phi = torch.empty(((M + 127) // 128) * ((K + r_s - 1) // r_s), dtype=torch.uint8, device=DEV)
    rfq.rfq_quantize_act(x, xq, xr, phi, mode=mode, tau=tau, p_s=128, r_s=r_s)
    y = guarded_full((M, N), float("nan"), torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16)
    ws = _workspace()
    rfq.rfq_linear(xq, xr, phi if use_phi else None, r_s, wq, y, out, ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    return xq, xr, wq, y.float().cpu().numpy(), phi


def _ref(orc, xq, xr, wq, M, K, N):
    mc, ms = qtensor_host(xq)
    wc, wsf = qtensor_host(wq)
    rc, rs = qtensor_host(xr) if xr is not None else (None, None)
    return orc.linear(orc.FMT_MXFP4, mc, ms, rc, rs, wc, wsf, M, K, N)


def test_tiny_workload_fp32(orc):
    spec = WORKLOADS["tiny"]
    xb = make_activation(spec.act)
    wb = make_weight(spec.act.K, spec.N, seed=spec.act.seed)
    xq, xr, wq, y, _ = _run(xb, wb)
    # the device codes are the oracle's (checked in test_gpu_quant); here the
    # product of the device codes must match the oracle's GEMM
    ref = _ref(orc, xq, xr, wq, 128, 512, 512)
    check_y(y, ref)
    # and the whole chain from X and W must match the oracle end to end
    q = orc.quantize_act(xb)
    wc, ws = orc.quantize_weight(wb)
    ref2 = orc.linear(0, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"], wc, ws, 128, 512, 512)
    check_y(y, ref2)


@pytest.mark.parametrize("M,K,N", [(1, 128, 16), (127, 256, 256), (129, 384, 272), (300, 640, 528),
                                   (256, 1024, 512), (513, 2048, 784)])
def test_ragged_shapes(orc, M, K, N):
    xb = make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, tok_count=1, tok_scale=200.0,
                                 seed=M + N))
    wb = make_weight(K, N, seed=K)
    xq, xr, wq, y, _ = _run(xb, wb)
    check_y(y, _ref(orc, xq, xr, wq, M, K, N))


def test_plain_w4a4_without_residual(orc):
    M, K, N = 200, 512, 256
    xb = make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, seed=2))
    wb = make_weight(K, N, seed=2)
    xq, xr, wq, y, _ = _run(xb, wb, mode=rfq.RFQ_FALLBACK_NONE)
    assert xr is None
    check_y(y, _ref(orc, xq, None, wq, M, K, N))


@pytest.mark.parametrize("M,K,r_s,tau", [(384, 1024, 256, 30.0), (384, 1024, 128, 20.0), (384, 1024, 512, 1e30),
                                         (384, 1024, 256, 0.0), (100, 1152, 128, 20.0), (300, 1152, 256, 20.0)])
def test_phi_amax_skips_residual_tiles(orc, M, K, r_s, tau):
    N = 256
    xb = make_activation(ActSpec(M, K, "normal", chan_count=3, chan_scale=64.0, seed=9))
    wb = make_weight(K, N, seed=9)
    xq, xr, wq, y, phi = _run(xb, wb, mode=rfq.RFQ_FALLBACK_AMAX, tau=tau, r_s=r_s, use_phi=True)
    check_y(y, _ref(orc, xq, xr, wq, M, K, N))
    q = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_AMAX, tau, 128, r_s)
    assert np.array_equal(phi.cpu().numpy().reshape(q["phi"].shape), q["phi"])


@pytest.mark.parametrize("M", [100, 256])
def test_phi_amax_many_stage_blocks(orc, M):
    """K = 135168: one output tile of 528 k-stages, so its CTA(s) walk more
    than two blocks of 256 per-stage residual masks; about half the 128 x 256
    tiles have phi = 1.  Y is checked on sampled rows."""
    K, N, r_s, tau = 135168, 256, 256, 30.0
    xb = make_activation(ActSpec(M, K, "normal", chan_count=360, chan_scale=64.0, seed=11))
    wb = make_weight(K, N, seed=11)
    xq, xr, wq, y, phi = _run(xb, wb, mode=rfq.RFQ_FALLBACK_AMAX, tau=tau, r_s=r_s, use_phi=True)
    q = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_AMAX, tau, 128, r_s)
    assert np.array_equal(phi.cpu().numpy().reshape(q["phi"].shape), q["phi"])
    assert 0.2 < q["phi"].mean() < 0.8
    rwc, rws = orc.quantize_weight(wb)
    wc, ws = qtensor_host(wq)
    assert np.array_equal(wc, rwc) and np.array_equal(ws, rws)
    rows = np.unique(np.concatenate([np.random.default_rng(1).choice(M, 10, replace=False), [0, M - 1]]))
    ref = orc.linear(0, q["main_codes"][rows], q["main_scales"][rows], q["res_codes"][rows], q["res_scales"][rows],
                     rwc, rws, len(rows), K, N)
    check_y(y[rows], ref)


def test_phi_amax_records_wrap(orc):
    """180 output tiles of 256 x 256 (up to three per CTA pair, so the
    per-tile phi records wrap their two buffers), a ragged last row pair, an
    odd number of 128-element chunks and a mixed phi pattern at r_s = 128."""
    M, K, N, r_s, tau = 600, 640, 15360, 128, 30.0
    xb = make_activation(ActSpec(M, K, "normal", chan_count=3, chan_scale=64.0, seed=31))
    wb = make_weight(K, N, seed=31)
    xq, xr, wq, y, phi = _run(xb, wb, mode=rfq.RFQ_FALLBACK_AMAX, tau=tau, r_s=r_s, use_phi=True)
    q = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_AMAX, tau, 128, r_s)
    assert np.array_equal(phi.cpu().numpy().reshape(q["phi"].shape), q["phi"])
    assert 0.1 < q["phi"].mean() < 0.9
    check_y(y, _ref(orc, xq, xr, wq, M, K, N))


def test_bf16_output(orc):
    M, K, N = 256, 1024, 512
    xb = make_activation(ActSpec(M, K, "normal", chan_count=4, chan_scale=64.0, seed=4))
    wb = make_weight(K, N, seed=4)
    xq, xr, wq, y, _ = _run(xb, wb, out=rfq.RFQ_OUT_BF16)
    check_y(y, _ref(orc, xq, xr, wq, M, K, N), bf16=True)


def test_repeated_calls_are_deterministic(orc):
    M, K, N = 256, 512, 256
    xb = make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, seed=8))
    wb = make_weight(K, N, seed=8)
    y1 = _run(xb, wb)[3]
    y2 = _run(xb, wb)[3]
    assert np.array_equal(y1, y2)


def _full_size(orc, name, out, n_rows=24):
    """Full-size workload through the launch configuration the benchmark
    times; the oracle checks the weight codes in full and Y on sampled rows
    (rows are independent in both the quantizer and the GEMM)."""
    spec = WORKLOADS[name]
    M, K, N = spec.act.M, spec.act.K, spec.N
    xb = make_activation(spec.act)
    wb = make_weight(K, N, seed=spec.act.seed)
    xq, xr, wq, y, _ = _run(xb, wb, out=out)
    wc, ws = qtensor_host(wq)
    rwc, rws = orc.quantize_weight(wb)
    assert np.array_equal(wc, rwc) and np.array_equal(ws, rws)
    rng = np.random.default_rng(0)
    rows = np.unique(np.concatenate([rng.choice(M, n_rows - 2, replace=False), [0, M - 1]]))
    q = orc.quantize_act(xb[rows])
    mc, ms = qtensor_host(xq)
    rc, rs = qtensor_host(xr)
    assert np.array_equal(mc[rows], q["main_codes"]) and np.array_equal(ms[rows], q["main_scales"])
    assert np.array_equal(rc[rows], q["res_codes"]) and np.array_equal(rs[rows], q["res_scales"])
    ref = orc.linear(0, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"], rwc, rws,
                     len(rows), K, N)
    check_y(y[rows], ref, bf16=(out == rfq.RFQ_OUT_BF16))
    assert np.isfinite(y).all()


def test_full_size_wan_ffn_up_bf16(orc):
    _full_size(orc, "wan_ffn_up", rfq.RFQ_OUT_BF16)


def test_full_size_wan_ffn_up_fp32(orc):
    _full_size(orc, "wan_ffn_up", rfq.RFQ_OUT_F32, n_rows=12)


def test_full_size_qwen_gate_up_bf16(orc):
    _full_size(orc, "qwen_gate_up", rfq.RFQ_OUT_BF16, n_rows=12)


@pytest.mark.parametrize("M", [100, 130])
def test_phi_beyond_record_capacity_falls_back_exactly(orc, M):
    """K / 256 = 2049 full k-stages: more than a phi record holds, so the GEMM
    issues every residual product (exact, since phi = 0 residuals are stored
    as zero) -- on the single-CTA (M <= 128) and the CTA-pair path."""
    K, N, r_s = 524544, 16, 256
    xb = make_activation(ActSpec(M, K, "normal", chan_count=400, chan_scale=64.0, seed=17))
    wb = make_weight(K, N, seed=17)
    xq, xr, wq, y, phi = _run(xb, wb, mode=rfq.RFQ_FALLBACK_AMAX, tau=30.0, r_s=r_s, use_phi=True)
    q = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_AMAX, 30.0, 128, r_s)
    assert np.array_equal(phi.cpu().numpy().reshape(q["phi"].shape), q["phi"])
    assert 0.0 < q["phi"].mean() < 1.0
    rwc, rws = orc.quantize_weight(wb)
    ref = orc.linear(0, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"], rwc, rws, M, K, N)
    check_y(y, ref)


def test_profile_build_computes_y_and_counts_its_stages(orc):
    """rfq_linear_profile: the CTA-pair kernel's measuring build gives the
    same Y (oracle parity) and counters that add up: every tile and stage of
    the grid counted once, waits within the measured cycles, a plausible SM
    clock."""
    M, K, N = 1000, 1280, 784
    xb = make_activation(ActSpec(M, K, "normal", chan_count=4, chan_scale=64.0, tok_count=2, tok_scale=200.0,
                                 seed=77))
    wb = make_weight(K, N, seed=77)
    x, w = to_dev_bf16(xb), to_dev_bf16(wb)
    wq = rfq.empty_qtensor(FMT, MMA, N, K)
    rfq.rfq_quantize_weight(w, wq)
    xq, xr = rfq.empty_qtensor(FMT, MMA, M, K), rfq.empty_qtensor(FMT, MMA, M, K)
    rfq.rfq_quantize_act(x, xq, xr)
    y = guarded_full((M, N), float("nan"), torch.float32)
    ws = _workspace()
    c = rfq.rfq_linear_profile(xq, xr, wq, y, rfq.RFQ_OUT_F32, ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    check_y(y.double().cpu().numpy(), _ref(orc, xq, xr, wq, M, K, N))
    tiles = -(-N // 256) * -(-M // 256)
    assert c["tiles"] == tiles
    assert c["stages"] == tiles * (K // 256) + (tiles if (K // 128) % 2 else 0)
    assert 0 < c["pairs"] <= 80
    assert c["cycles"] > 0 and c["ns"] > 0
    for k in ("wait_acc_cycles", "wait_copies_cycles", "wait_scales_cycles"):
        assert 0 <= c[k] <= c["cycles"], k
    mhz = c["cycles"] / c["ns"] * 1e3
    assert 500 < mhz < 3000, mhz
    # the measuring build is the CTA-pair kernel's: 128 rows or fewer are refused
    small = rfq.empty_qtensor(FMT, MMA, 64, K)
    with pytest.raises(rfq.RFQError) as e:
        rfq.rfq_linear_profile(small, small, wq, torch.empty(64, N, device=DEV), rfq.RFQ_OUT_F32, ws)
    assert e.value.status == rfq.RFQ_ERR_UNSUPPORTED
