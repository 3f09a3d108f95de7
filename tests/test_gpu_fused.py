"""GPU parity of rfq_linear_fused (the quantizer inside the GEMM, Sec. 4.3's
on-the-fly residual) against the fp64 CPU oracle: Y = Q(X) W~ + Q(X - Q(X)) W~
with the oracle's own quantization of X, and against the two-kernel path
(rfq_quantize_act + rfq_linear), whose codes are bit-exact.  Beyond 128 rows
the GEMM's own warps quantize X into the workspace's scratch: those codes and
scale bytes must be the oracle's bit for bit, and the unit counters must be
left zero for the next call."""
import numpy as np
import pytest
import torch

from gpu_util import DEV, check_y, guarded_full, mma_scale_to_rowmajor, to_dev_bf16
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


def _layout(M, K, res):
    """Byte offsets inside the fused workspace (M > 128), as include/rfq.h
    states them: the 256-byte GEMM workspace, the counters, then the scratch
    ring of R = min(12, ceil(M / 256)) slots of 256 rows -- codes of X~ and
    X^ and their MMA-layout scales -- each 1024-byte aligned."""
    up = lambda v: (v + 1023) // 1024 * 1024
    tiles, stages, pairs = -(-M // 128), (K // 128 + 1) // 2, -(-M // 256)
    ring = min(12, pairs)
    rows = ring * 256
    codes, sf = rows * K // 2, rows * (K // 32)
    ctr = 256
    n_ctr = 2 + tiles + tiles * stages + pairs
    mc = up(ctr + 4 * n_ctr)
    rc = up(mc + codes)
    ms = up(rc + (codes if res else 0))
    rs = up(ms + sf)
    total = up(rs + (sf if res else 0))
    return dict(ctr=ctr, n_ctr=n_ctr, mc=mc, rc=rc, ms=ms, rs=rs, total=total, codes=codes, sf=sf, ring=ring,
                pairs=pairs, rows=rows)


def _fused(xb, wq, out=rfq.RFQ_OUT_F32, mode=rfq.RFQ_FALLBACK_ALL, ws=None, calls=1):
    M, K = xb.shape
    y = guarded_full((M, wq.rows), float("nan"), torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16)
    if ws is None:
        ws = rfq.fused_workspace(M, K, mode)
    x = to_dev_bf16(xb)
    for _ in range(calls):
        rfq.rfq_linear_fused(x, wq, y, out, ws, mode=mode)
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


def test_workspace_size():
    for M, K, mode in [(1, 128, rfq.RFQ_FALLBACK_ALL), (128, 4096, rfq.RFQ_FALLBACK_NONE),
                       (129, 384, rfq.RFQ_FALLBACK_ALL), (32760, 5120, rfq.RFQ_FALLBACK_ALL),
                       (1000, 640, rfq.RFQ_FALLBACK_NONE)]:
        want = rfq.rfq_linear_workspace_bytes() if M <= 128 else _layout(M, K, mode != rfq.RFQ_FALLBACK_NONE)["total"]
        assert rfq.rfq_linear_fused_workspace_bytes(M, K, mode) == want
    assert rfq.rfq_linear_fused_workspace_bytes(300, 96) == 0
    small = torch.zeros(64, dtype=torch.int32, device=DEV)
    with pytest.raises(ValueError):
        rfq.rfq_linear_fused(torch.zeros(300, 256, dtype=torch.bfloat16, device=DEV), rfq.empty_qtensor(FMT, MMA, 16, 256),
                             torch.zeros(300, 16, device=DEV), rfq.RFQ_OUT_F32, small)


@pytest.mark.parametrize("M,K,mode", [(129, 384, rfq.RFQ_FALLBACK_ALL), (300, 640, rfq.RFQ_FALLBACK_ALL),
                                      (1000, 2048, rfq.RFQ_FALLBACK_ALL), (777, 1024, rfq.RFQ_FALLBACK_NONE),
                                      (4000, 512, rfq.RFQ_FALLBACK_ALL)])   # 16 row blocks: the ring wraps
def test_in_gemm_quantizer_codes_are_the_oracles(orc, M, K, mode):
    """The codes and E8M0 bytes the GEMM's warps leave in the workspace's
    ring (slot s holds the last 256-row block b with b % R == s) are the
    oracle's quantization of X (main and residual, every byte; rows past M
    zero); the counters are zero after each of three calls on the same
    workspace, and Y matches the oracle each time."""
    N = 256
    res = mode != rfq.RFQ_FALLBACK_NONE
    xb = make_activation(ActSpec(M, K, "student_t3", chan_count=3, chan_scale=100.0, tok_count=2, tok_scale=200.0,
                                 seed=M + K))
    xb[3, :32] = 0                     # an all-zero block
    xb[5, 40] = 0x8000                 # a negative zero
    wb = make_weight(K, N, seed=M)
    wq = _weight(wb)
    ws = rfq.fused_workspace(M, K, mode)
    L = _layout(M, K, res)
    assert ws.numel() * 4 == L["total"]
    q = orc.quantize_act(xb, orc.FMT_MXFP4, orc.PHI_ALL if res else orc.PHI_NONE)
    wc, wsf = orc.quantize_weight(wb)
    ref = orc.linear(orc.FMT_MXFP4, q["main_codes"], q["main_scales"], q["res_codes"] if res else None,
                     q["res_scales"] if res else None, wc, wsf, M, K, N)
    # what the ring must hold: per slot, the last block written to it, zero
    # past M; a 128-row half of a slot wholly past M is never written (the
    # GEMM loads a zero-filled box for it), so only written rows are compared
    rows_pad = L["pairs"] * 256
    tiles = -(-M // 128)
    written = np.zeros(L["rows"], bool)
    for s_ in range(L["ring"]):
        b_ = max(p for p in range(L["pairs"]) if p % L["ring"] == s_)
        for h in range(2):
            written[s_ * 256 + h * 128:s_ * 256 + (h + 1) * 128] = 2 * b_ + h < tiles
    want = {}
    for key in ("main", "res") if res else ("main",):
        c = np.zeros((rows_pad, K // 2), np.uint8)
        c[:M] = q[key + "_codes"]
        sc = np.zeros((rows_pad, K // 32), np.uint8)
        sc[:M] = q[key + "_scales"]
        wc_, ws_ = np.zeros((L["rows"], K // 2), np.uint8), np.zeros((L["rows"], K // 32), np.uint8)
        for s in range(L["ring"]):
            b = max(p for p in range(L["pairs"]) if p % L["ring"] == s)
            wc_[s * 256:(s + 1) * 256] = c[b * 256:(b + 1) * 256]
            ws_[s * 256:(s + 1) * 256] = sc[b * 256:(b + 1) * 256]
        want[key] = (wc_, ws_)
    for call in range(3):
        y = _fused(xb, wq, mode=mode, ws=ws)
        check_y(y, ref)
        b = ws.view(torch.uint8).cpu().numpy()
        assert not b[L["ctr"]:L["ctr"] + 4 * L["n_ctr"]].any(), "counters left non-zero"
        for key, (co, so) in (("main", (L["mc"], L["ms"])), ("res", (L["rc"], L["rs"]))):
            if key not in want:
                continue
            got_c = b[co:co + L["codes"]].reshape(L["rows"], K // 2)
            assert np.array_equal(got_c[written], want[key][0][written]), f"call {call}: {key} codes differ"
            got_s = mma_scale_to_rowmajor(b[so:so + L["sf"]], L["rows"], K)
            assert np.array_equal(got_s[written], want[key][1][written]), f"call {call}: {key} scale bytes differ"
        if call == 0:
            # stale bytes in the scratch must not matter: every one is rewritten
            ws.view(torch.uint8)[L["mc"]:].fill_(0x77)


def test_many_tiles_per_pair(orc):
    """More output tiles than CTA pairs (tiles walk in row-block order while
    the quantizer runs ahead): rows sampled across the whole M."""
    M, K, N = 4096, 1024, 4096
    xb = make_activation(ActSpec(M, K, "normal", chan_count=8, chan_scale=64.0, tok_count=4, tok_scale=200.0, seed=7))
    wb = make_weight(K, N, seed=7)
    wq = _weight(wb)
    y = _fused(xb, wq, out=rfq.RFQ_OUT_BF16, calls=2)
    rng = np.random.default_rng(3)
    rows = np.unique(np.concatenate([rng.choice(M, 24, replace=False), [0, 127, 128, 255, 256, M - 1]]))
    check_y(y[rows], _oracle(orc, xb[rows], wb), bf16=True)
    assert np.isfinite(y).all()
