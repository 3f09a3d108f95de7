"""GPU parity of rfq_linear_host: the RFQ linear layer (Algorithm 1,
Eq. rfq) from host memory, in row chunks on copy streams.  Its Y equals
rfq_linear's on the device-resident operands bit for bit (row chunks do not
change any output element's accumulation) and matches the oracle end to end
from X and W within the GEMM tolerance."""
import numpy as np
import pytest
import torch

from gpu_util import DEV, check_y, to_dev_bf16
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import ActSpec, make_activation, make_weight

pytestmark = pytest.mark.gpu
MMA, F4 = rfq.RFQ_SCALE_MMA, rfq.RFQ_FMT_MXFP4


def _case(orc, M, K, N, chunk, mode=rfq.RFQ_FALLBACK_ALL, tau=0.0, out=rfq.RFQ_OUT_F32, pinned=True, seed=0):
    xb = make_activation(ActSpec(M, K, "normal", chan_count=3, chan_scale=64.0, seed=seed))
    wb = make_weight(K, N, seed=seed + 1)
    wq = rfq.empty_qtensor(F4, MMA, N, K)
    rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
    x_host = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16)
    if pinned:
        x_host = x_host.pin_memory()
    ydt = torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16
    y_host = torch.full((M, N), float("nan"), dtype=ydt)
    if pinned:
        y_host = y_host.pin_memory()
    res = mode != rfq.RFQ_FALLBACK_NONE
    x_dev = torch.empty(M, K, dtype=torch.bfloat16, device=DEV)
    xq = rfq.empty_qtensor(F4, MMA, M, K)
    xr = rfq.empty_qtensor(F4, MMA, M, K) if res else None
    phi = torch.empty(max(((M + 127) // 128) * ((K + 255) // 256), 1), dtype=torch.uint8, device=DEV)
    y_dev = torch.empty(M, N, dtype=ydt, device=DEV)
    ws = torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)
    rfq.rfq_linear_host(x_host, wq, y_host, out, x_dev, xq, xr, phi, y_dev, ws, mode=mode, tau=tau,
                        chunk_rows=chunk)
    torch.cuda.synchronize()
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    # the same operands through the device entry points, whole matrices at once
    x2 = to_dev_bf16(xb)
    q2 = rfq.empty_qtensor(F4, MMA, M, K)
    r2 = rfq.empty_qtensor(F4, MMA, M, K) if res else None
    phi2 = torch.empty_like(phi)
    rfq.rfq_quantize_act(x2, q2, r2, phi2, mode=mode, tau=tau, p_s=128, r_s=256)
    y2 = torch.empty(M, N, dtype=ydt, device=DEV)
    rfq.rfq_linear(q2, r2, phi2 if mode == rfq.RFQ_FALLBACK_AMAX else None, 256, wq, y2, out, ws)
    assert torch.equal(y_host, y2.cpu())
    # and the oracle from X and W
    omode = {rfq.RFQ_FALLBACK_ALL: orc.PHI_ALL, rfq.RFQ_FALLBACK_NONE: orc.PHI_NONE,
             rfq.RFQ_FALLBACK_AMAX: orc.PHI_AMAX}[mode]
    q = orc.quantize_act(xb, orc.FMT_MXFP4, omode, tau, 128, 256)
    wc, wsf = orc.quantize_weight(wb)
    ref = orc.linear(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], q["res_codes"] if res else None,
                     q["res_scales"] if res else None, wc, wsf, M, K, N)
    check_y(y_host.float().numpy(), ref, bf16=(out == rfq.RFQ_OUT_BF16))


@pytest.mark.parametrize("M,chunk", [(1000, 256), (300, 0), (128, 128), (1, 128)])
def test_host_path_chunks(orc, M, chunk):
    _case(orc, M, 512, 272, chunk, seed=M)


def test_host_path_bf16_no_residual_and_amax(orc):
    _case(orc, 700, 768, 528, 256, mode=rfq.RFQ_FALLBACK_NONE, out=rfq.RFQ_OUT_BF16, seed=3)
    _case(orc, 700, 768, 528, 384, mode=rfq.RFQ_FALLBACK_AMAX, tau=30.0, seed=4)


def test_host_path_pageable_memory(orc):
    _case(orc, 513, 512, 256, 256, pinned=False, seed=5)


def test_host_path_empty():
    K, N = 256, 256
    wq = rfq.empty_qtensor(F4, MMA, N, K)
    ws = torch.zeros(64, dtype=torch.int32, device=DEV)
    x_host = torch.empty(0, K, dtype=torch.bfloat16)
    y_host = torch.empty(0, N)
    # (the empty host tensors have no storage: NULL pointers, allowed at M = 0)
    rfq.rfq_linear_host(x_host, wq, y_host, rfq.RFQ_OUT_F32, torch.empty(0, K, dtype=torch.bfloat16, device=DEV),
                        rfq.empty_qtensor(F4, MMA, 0, K), rfq.empty_qtensor(F4, MMA, 0, K), None,
                        torch.empty(0, N, device=DEV), ws)
    torch.cuda.synchronize()
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
