"""The allocation-free RFQ GEMM entry point (rfq_linear_noalloc).

Callers that cannot allocate device memory (no cudaMalloc in their serving
loop, or a host program that owns every device buffer) call this variant; it
keeps the GEMM's workspace in a fixed array inside the library instead of a
caller buffer.  Its output must match rfq_linear's within the Y tolerance of
the other tests, on two calls in a row (the second call reuses the array the
first one left behind), and the oracle's product of the same codes.  This
file is collected last on purpose.
"""
import numpy as np
import pytest
import torch

from gpu_util import DEV, check_y, qtensor_host, to_dev_bf16
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import ActSpec, make_activation, make_weight

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("out", [rfq.RFQ_OUT_F32, rfq.RFQ_OUT_BF16])
def test_noalloc_matches_rfq_linear_twice(orc, out):
    M, K, N = 300, 1024, 528
    xb = make_activation(ActSpec(M, K, "normal", chan_count=3, chan_scale=64.0, tok_count=1, tok_scale=200.0,
                                 seed=21))
    wb = make_weight(K, N, seed=21)
    x, w = to_dev_bf16(xb), to_dev_bf16(wb)
    F, L = rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA
    wq = rfq.empty_qtensor(F, L, N, K)
    xq = rfq.empty_qtensor(F, L, M, K)
    xr = rfq.empty_qtensor(F, L, M, K)
    rfq.rfq_quantize_weight(w, wq)
    rfq.rfq_quantize_act(x, xq, xr)
    dt = torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16
    y_ref = torch.empty(M, N, dtype=dt, device=DEV)
    ws = torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)
    rfq.rfq_linear(xq, xr, None, 256, wq, y_ref, out, ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    ref = y_ref.double().cpu().numpy()
    mc, ms = qtensor_host(xq)
    rc, rs = qtensor_host(xr)
    wc, wsf = qtensor_host(wq)
    y_orc = orc.linear(orc.FMT_MXFP4, mc, ms, rc, rs, wc, wsf, M, K, N)
    for _ in range(2):
        y = torch.full((M, N), float("nan"), dtype=dt, device=DEV)
        rfq.rfq_linear_noalloc(xq, xr, None, 256, wq, y, out)
        torch.cuda.synchronize()
        got = y.double().cpu().numpy()
        assert np.isfinite(got).all()
        check_y(got, ref, bf16=(out == rfq.RFQ_OUT_BF16))
        check_y(got, y_orc, bf16=(out == rfq.RFQ_OUT_BF16))
