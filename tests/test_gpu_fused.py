"""GPU parity of rfq_linear_fused (the quantizer inside the GEMM, Sec. 4.3's
on-the-fly residual) against the fp64 CPU oracle: Y = Q(X) W~ + Q(X - Q(X)) W~
with the oracle's own quantization of X, and against the two-kernel path
(rfq_quantize_act + rfq_linear), whose codes are bit-exact."""
import numpy as np
import pytest
import torch

from gpu_util import DEV, check_y, to_dev_bf16
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import WORKLOADS, ActSpec, make_activation, make_weight

pytestmark = pytest.mark.gpu
MMA = rfq.RFQ_SCALE_MMA
FMT = rfq.RFQ_FMT_MXFP4


def _ws():
    return torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)


def _weight(wb):
    K, N = wb.shape
    wq = rfq.empty_qtensor(FMT, MMA, N, K)
    rfq.rfq_quantize_weight(to_dev_bf16(wb), wq)
    return wq


def _fused(xb, wq, out=rfq.RFQ_OUT_F32, mode=rfq.RFQ_FALLBACK_ALL):
    M, K = xb.shape
    y = torch.full((M, wq.rows), float("nan"), device=DEV,
                   dtype=torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16)
    ws = _ws()
    rfq.rfq_linear_fused(to_dev_bf16(xb), wq, y, out, ws, mode=mode)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    return y.float().cpu().numpy()


def _two_kernel(xb, wq, out=rfq.RFQ_OUT_F32, mode=rfq.RFQ_FALLBACK_ALL):
    M, K = xb.shape
    xq = rfq.empty_qtensor(FMT, MMA, M, K)
    xr = rfq.empty_qtensor(FMT, MMA, M, K) if mode != rfq.RFQ_FALLBACK_NONE else None
    rfq.rfq_quantize_act(to_dev_bf16(xb), xq, xr, None, mode=mode)
    y = torch.empty((M, wq.rows), device=DEV, dtype=torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16)
    ws = _ws()
    rfq.rfq_linear(xq, xr, None, 256, wq, y, out, ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    return y.float().cpu().numpy()


def _oracle(orc, xb, wb, residual=True):
    M, K = xb.shape
    N = wb.shape[1]
    q = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_ALL if residual else orc.PHI_NONE)
    wc, ws = orc.quantize_weight(wb)
    return orc.linear(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], q["res_codes"] if residual else None,
                      q["res_scales"] if residual else None, wc, ws, M, K, N)


def test_tiny_workload(orc):
    spec = WORKLOADS["tiny"]
    xb = make_activation(spec.act)
    wb = make_weight(spec.act.K, spec.N, seed=spec.act.seed)
    wq = _weight(wb)
    y = _fused(xb, wq)
    check_y(y, _oracle(orc, xb, wb))
    # same codes, same MMAs as the two-kernel path
    assert np.allclose(y, _two_kernel(xb, wq), rtol=0, atol=1e-6 * np.abs(y).max())


@pytest.mark.parametrize("M,K,N", [(1, 128, 16), (127, 256, 256), (129, 384, 272), (300, 640, 528),
                                   (513, 2048, 784)])
def test_ragged_shapes(orc, M, K, N):
    xb = make_activation(ActSpec(M, K, "student_t3", chan_count=2, chan_scale=64.0, tok_count=1, tok_scale=200.0,
                                 seed=M + N))
    wb = make_weight(K, N, seed=K)
    y = _fused(xb, _weight(wb))
    check_y(y, _oracle(orc, xb, wb))


def test_plain_w4a4_mode_none(orc):
    M, K, N = 200, 512, 256
    xb = make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, seed=2))
    wb = make_weight(K, N, seed=2)
    y = _fused(xb, _weight(wb), mode=rfq.RFQ_FALLBACK_NONE)
    check_y(y, _oracle(orc, xb, wb, residual=False))


def test_bf16_output_matches_two_kernel_path(orc):
    M, K, N = 384, 1024, 512
    xb = make_activation(ActSpec(M, K, "normal", chan_count=4, chan_scale=64.0, seed=4))
    wb = make_weight(K, N, seed=4)
    wq = _weight(wb)
    y = _fused(xb, wq, out=rfq.RFQ_OUT_BF16)
    check_y(y, _oracle(orc, xb, wb), bf16=True)
    y2 = _two_kernel(xb, wq, out=rfq.RFQ_OUT_BF16)
    # accumulation order may differ between the kernels by one bf16 rounding
    assert np.abs(y - y2).max() <= 2.0 ** -7 * np.abs(y2).max()


def test_full_size_wan_ffn_up_sampled_rows(orc):
    """The bench's Wan2.2 FFN up shape; Y checked on sampled rows."""
    spec = WORKLOADS["wan_ffn_up"]
    M, K, N = spec.act.M, spec.act.K, spec.N
    xb = make_activation(spec.act)
    wb = make_weight(K, N, seed=spec.act.seed)
    y = _fused(xb, _weight(wb), out=rfq.RFQ_OUT_BF16)
    rng = np.random.default_rng(1)
    rows = np.unique(np.concatenate([rng.choice(M, 10, replace=False), [0, M - 1]]))
    check_y(y[rows], _oracle(orc, xb[rows], wb), bf16=True)
    assert np.isfinite(y).all()
