"""The GEMMs' bounded waits, made to run out on purpose.

Every mbarrier wait in the GEMM kernels gives up after a limit and records
RFQ_ERR_TIMEOUT in the caller's workspace; the kernel then drains what it has
in flight, frees its tensor memory and returns.  The workspace's held start
(word 2 set, word 3 left zero) makes each copy producer wait for a gate that
nothing opens, before its first copy, with a 20 ms limit (word 1): the wait
runs out with no copy or MMA in flight, every other role of the kernel gives
up on the recorded status, and the device stays usable.  Each case checks
that the timeout is reported, that Y is left unwritten, that the record is
sticky (a later call with that workspace computes nothing), that an opened
gate lets the call compute, and that after the workspace is cleared the same
buffers give the oracle's result."""
import numpy as np
import pytest
import torch

from conftest import ROOT
from gpu_util import DEV, check_y, qtensor_host, to_dev_bf16
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import ActSpec, make_activation, make_weight

pytestmark = pytest.mark.gpu
F4, F8, H, MMA = rfq.RFQ_FMT_MXFP4, rfq.RFQ_FMT_MXFP8, rfq.RFQ_FMT_HIF4, rfq.RFQ_SCALE_MMA
LIMIT_US = 20000


def _ws():
    return torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)


def _held_then_recovered(launch, y, ref, bf16=False, ws=None):
    # the gate stays shut: the producers' wait runs out
    ws = _ws() if ws is None else ws
    ws[1] = LIMIT_US
    ws[2] = 1
    launch(ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_ERR_TIMEOUT
    assert torch.isnan(y.float()).all(), "a timed-out call wrote Y"
    # the record is sticky: with the gate open, the same workspace still computes nothing
    ws[3] = 1
    launch(ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_ERR_TIMEOUT
    assert torch.isnan(y.float()).all(), "a call after a recorded timeout wrote Y"
    # a held start whose gate is open computes normally
    ws.zero_()
    ws[1] = LIMIT_US
    ws[2] = 1
    ws[3] = 1
    launch(ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    check_y(y.double().cpu().numpy(), ref, bf16=bf16)
    # cleared workspace, same buffers: the oracle's result
    y.fill_(float("nan"))
    ws.zero_()
    launch(ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    check_y(y.double().cpu().numpy(), ref, bf16=bf16)


def _mx_operands(M, K, N, seed, res_fmt=F4):
    xb = make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, tok_count=1, tok_scale=100.0,
                                 seed=seed))
    wb = make_weight(K, N, seed=seed + 1)
    wq = rfq.empty_qtensor(F4, MMA, N, K)
    rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
    xq = rfq.empty_qtensor(F4, MMA, M, K)
    xr = rfq.empty_qtensor(res_fmt, MMA, M, K)
    phi = torch.empty(((M + 127) // 128) * ((K + 255) // 256), dtype=torch.uint8, device=DEV)
    rfq.rfq_quantize_act(to_dev_bf16(xb), xq, xr, phi, mode=rfq.RFQ_FALLBACK_AMAX, tau=150.0, p_s=128, r_s=256)
    return xb, wb, wq, xq, xr, phi


def _mx_ref(orc, xq, xr, wq, M, K, N, res_fmt=None):
    mc, ms = qtensor_host(xq)
    rc, rs = qtensor_host(xr)
    wc, wsf = qtensor_host(wq)
    if res_fmt is None:
        return orc.linear(orc.FMT_MXFP4, mc, ms, rc, rs, wc, wsf, M, K, N)
    return orc.linear(orc.FMT_MXFP4, mc, ms, rc, rs, wc, wsf, M, K, N, res_fmt=res_fmt)


@pytest.mark.parametrize("M,out,use_phi", [(100, rfq.RFQ_OUT_F32, False),     # single CTA
                                           (100, rfq.RFQ_OUT_BF16, True),     # single CTA, phi reader
                                           (600, rfq.RFQ_OUT_F32, False),     # CTA pairs
                                           (600, rfq.RFQ_OUT_BF16, True)])    # CTA pairs, phi reader
def test_mxfp4_gemm_timeout(orc, M, out, use_phi):
    K, N = 1024, 512
    _, _, wq, xq, xr, phi = _mx_operands(M, K, N, seed=M + out)
    y = torch.full((M, N), float("nan"), dtype=torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16,
                   device=DEV)
    launch = lambda ws: rfq.rfq_linear(xq, xr, phi if use_phi else None, 256, wq, y, out, ws)
    _held_then_recovered(launch, y, _mx_ref(orc, xq, xr, wq, M, K, N), bf16=out == rfq.RFQ_OUT_BF16)


def test_e4m3_pair_gemm_timeout(orc):
    """The FP4-to-FP8 residual on the E4M3 instantiation of the pair GEMM."""
    M, K, N = 384, 512, 256
    _, _, wq, x4, xr, _ = _mx_operands(M, K, N, seed=5, res_fmt=F8)
    w8 = rfq.empty_qtensor(F8, MMA, N, K)
    rfq.rfq_convert(wq, w8)
    x8 = rfq.empty_qtensor(F8, MMA, M, K)
    rfq.rfq_convert(x4, x8)
    y = torch.full((M, N), float("nan"), dtype=torch.float32, device=DEV)
    launch = lambda ws: rfq.rfq_linear(x8, xr, None, 256, w8, y, rfq.RFQ_OUT_F32, ws)
    _held_then_recovered(launch, y, _mx_ref(orc, x4, xr, wq, M, K, N, res_fmt=orc.FMT_MXFP8))


def test_hif4_gemm_timeout(orc):
    M, K, N = 256, 512, 256
    xb = make_activation(ActSpec(M, K, "laplace", body_scale=0.3, chan_count=3, chan_scale=50.0, seed=21))
    wb = make_weight(K, N, seed=22)
    wq = rfq.empty_qtensor(H, rfq.RFQ_SCALE_ROWMAJOR, N, K)
    rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
    w16 = rfq.empty_bf16_operand(N, K)
    rfq.rfq_dequant(wq, w16.codes)
    xq = rfq.empty_qtensor(H, MMA, M, K)
    xr = rfq.empty_qtensor(H, MMA, M, K)
    xq16, xr16 = rfq.empty_bf16_operand(M, K), rfq.empty_bf16_operand(M, K)
    rfq.rfq_quantize_act_expand(to_dev_bf16(xb), xq, xr, xq16, xr16, None)
    y = torch.full((M, N), float("nan"), dtype=torch.float32, device=DEV)
    launch = lambda ws: rfq.rfq_linear(xq16, xr16, None, 256, w16, y, rfq.RFQ_OUT_F32, ws)
    mc, mm = qtensor_host(xq)
    rc, rm = qtensor_host(xr)
    wc, wm = qtensor_host(wq)
    _held_then_recovered(launch, y, orc.linear(orc.FMT_HIF4, mc, mm, rc, rm, wc, wm, M, K, N))


@pytest.mark.parametrize("M", [100, 300])   # single CTA; CTA pairs quantizing into the workspace
def test_fused_gemm_timeout(orc, M):
    K, N = 512, 256
    xb = make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, seed=31))
    wb = make_weight(K, N, seed=32)
    wq = rfq.empty_qtensor(F4, MMA, N, K)
    rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
    x = to_dev_bf16(xb)
    y = torch.full((M, N), float("nan"), dtype=torch.float32, device=DEV)
    launch = lambda ws: rfq.rfq_linear_fused(x, wq, y, rfq.RFQ_OUT_F32, ws)
    q = orc.quantize_act(xb)
    wc, wsf = qtensor_host(wq)
    ref = orc.linear(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"], wc, wsf,
                     M, K, N)
    _held_then_recovered(launch, y, ref, ws=rfq.fused_workspace(M, K))


@pytest.mark.parametrize("counts", [[100, 300, 0, 50], [2100, 2500]])   # single-CTA and CTA-pair forms
def test_grouped_gemm_timeout(orc, counts):
    K, N = 512, 256
    starts, pos = [], 0
    for c in counts:
        starts.append(pos)
        pos = -(-(pos + c) // 128) * 128
    ends = [s + c for s, c in zip(starts, counts)]
    total = max(pos, 128)
    xb = np.zeros((total, K), np.uint16)
    for g, c in enumerate(counts):
        if c:
            xb[starts[g]:ends[g]] = make_activation(ActSpec(c, K, "normal", chan_count=2, chan_scale=64.0,
                                                            seed=40 + g))
    G = len(counts)
    wb = np.concatenate([make_weight(K, N, seed=50 + g) for g in range(G)], axis=1)
    wq = rfq.empty_qtensor(F4, MMA, G * N, K)
    rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
    xq = rfq.empty_qtensor(F4, MMA, total, K)
    xr = rfq.empty_qtensor(F4, MMA, total, K)
    rfq.rfq_quantize_act(to_dev_bf16(xb), xq, xr)
    off = torch.from_numpy(np.array(starts + [ends[-1]], np.int32)).to(DEV)
    y = torch.full((total, N), float("nan"), dtype=torch.float32, device=DEV)
    launch = lambda ws: rfq.rfq_linear_grouped(xq, xr, None, 256, off, wq, N, y, rfq.RFQ_OUT_F32, ws)
    mc, ms = qtensor_host(xq)
    rc, rs = qtensor_host(xr)
    wc, wsf = qtensor_host(wq)
    ref = np.full((total, N), np.nan)
    for g in range(G):
        a, b = starts[g], -(-ends[g] // 128) * 128 if g + 1 < G else ends[g]
        if b > a:
            ref[a:b] = orc.linear(orc.FMT_MXFP4, mc[a:b], ms[a:b], rc[a:b], rs[a:b], wc[g * N:(g + 1) * N],
                                  wsf[g * N:(g + 1) * N], b - a, K, N)
    rows = ~np.isnan(ref[:, 0])

    def check(yg, r, bf16=False):
        check_y(yg[rows], r[rows], bf16=bf16)

    # rows outside every group stay NaN; compare the computed rows only
    ws = _ws()
    ws[1], ws[2] = LIMIT_US, 1
    launch(ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_ERR_TIMEOUT
    assert torch.isnan(y).all()
    ws.zero_()
    launch(ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    check(y.double().cpu().numpy(), ref)


def test_debug_sync_reports_the_timeout_at_the_call():
    """With RFQ_DEBUG_SYNC set, rfq_linear synchronizes and returns the
    workspace's status: a held start that runs out raises RFQ_ERR_TIMEOUT
    from the call itself (a child process: the variable is read once)."""
    import os
    import subprocess
    import sys
    code = """
import sys, torch
sys.path.insert(0, %r)
sys.path.insert(0, %r)
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import ActSpec, make_activation, make_weight
from gpu_util import to_dev_bf16
M, K, N = 600, 512, 256
F, L = rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA
wq = rfq.empty_qtensor(F, L, N, K); rfq.rfq_quantize_weight(to_dev_bf16(make_weight(K, N, seed=1)), wq)
xq, xr = rfq.empty_qtensor(F, L, M, K), rfq.empty_qtensor(F, L, M, K)
rfq.rfq_quantize_act(to_dev_bf16(make_activation(ActSpec(M, K, "normal", seed=2))), xq, xr)
y = torch.empty(M, N, device="cuda")
ws = torch.zeros(64, dtype=torch.int32, device="cuda")
rfq.rfq_linear(xq, xr, None, 256, wq, y, rfq.RFQ_OUT_F32, ws)   # computes: RFQ_OK
ws[1], ws[2] = 20000, 1
try:
    rfq.rfq_linear(xq, xr, None, 256, wq, y, rfq.RFQ_OUT_F32, ws)
except rfq.RFQError as e:
    print("STATUS", e.status)
""" % (ROOT, os.path.join(ROOT, "tests"))
    env = dict(os.environ, RFQ_DEBUG_SYNC="1")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert f"STATUS {rfq.RFQ_ERR_TIMEOUT}" in r.stdout, r.stdout + r.stderr[-2000:]
