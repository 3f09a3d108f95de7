"""GPU parity of the grouped (mixture-of-experts) RFQ GEMM: one launch over
groups of token rows, group g against its own weight W~_g (Algorithm 1,
Eq. rfq per expert).  Each group's rows of Y must match the oracle's RFQ
GEMM of that group's rows and weight; the zero rows padding a group to the
next 128-row start give zero rows; rows past the last group stay untouched;
offsets that break the contract are reported, not computed."""
import numpy as np
import pytest
import torch

from gpu_util import DEV, check_y, qtensor_host, to_dev_bf16, guarded_full
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import ActSpec, make_activation, make_weight

pytestmark = pytest.mark.gpu
F4, F8, MMA = rfq.RFQ_FMT_MXFP4, rfq.RFQ_FMT_MXFP8, rfq.RFQ_SCALE_MMA


def _case(orc, counts, K, N, fmt="rfq4", mode=rfq.RFQ_FALLBACK_ALL, tau=0.0, r_s=256, out=rfq.RFQ_OUT_F32, seed=0,
          packed_w=False):
    G = len(counts)
    starts = []
    pos = 0
    for c in counts:
        starts.append(pos)
        pos = -(-(pos + c) // 128) * 128
    ends = [s + c for s, c in zip(starts, counts)]
    total = max(pos, 128)
    off = np.array(starts + [ends[-1]], np.int32)
    # group g's rows sit at [starts[g], ends[g]); padding rows are zero
    xb = np.zeros((total, K), np.uint16)
    for g in range(G):
        if counts[g]:
            xb[starts[g]:ends[g]] = make_activation(ActSpec(counts[g], K, "normal", chan_count=2, chan_scale=64.0,
                                                            tok_count=1, tok_scale=100.0, seed=seed + g))
    wbs = [make_weight(K, N, seed=seed + 100 + g) for g in range(G)]
    wb = np.concatenate(wbs, axis=1)                  # W for all groups: [K, G N]
    x, w = to_dev_bf16(xb), to_dev_bf16(wb)
    ws = torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)
    y = guarded_full((total, N), float("nan"), torch.float32 if out == rfq.RFQ_OUT_F32 else torch.bfloat16)
    phi = None
    f8 = fmt != "rfq4"
    wq = rfq.empty_qtensor(F4, MMA, G * N, K)
    rfq.rfq_quantize_weight(w, wq)
    if f8 and packed_w:
        w8 = wq          # MXFP8 activations x the MXFP4 W~, multiplied as E2M1
    elif f8:
        w8 = rfq.empty_qtensor(F8, MMA, G * N, K)
        rfq.rfq_convert(wq, w8)
    if fmt == "rfq4":
        xq = rfq.empty_qtensor(F4, MMA, total, K)
        xr = rfq.empty_qtensor(F4, MMA, total, K)
        phi = torch.empty(((total + 127) // 128) * ((K + r_s - 1) // r_s), dtype=torch.uint8, device=DEV)
        rfq.rfq_quantize_act(x, xq, xr, phi, mode=mode, tau=tau, p_s=128, r_s=r_s)
        rfq.rfq_linear_grouped(xq, xr, phi if mode == rfq.RFQ_FALLBACK_AMAX else None, r_s,
                               torch.from_numpy(off).to(DEV), wq, N, y, out, ws)
    elif fmt == "w4a8":
        xq = rfq.empty_qtensor(F8, MMA, total, K)
        rfq.rfq_quantize_act(x, xq, None, None, mode=rfq.RFQ_FALLBACK_NONE)
        rfq.rfq_linear_grouped(xq, None, None, 256, torch.from_numpy(off).to(DEV), w8, N, y, out, ws)
    else:  # rfq8
        x4 = rfq.empty_qtensor(F4, MMA, total, K)
        xr = rfq.empty_qtensor(F8, MMA, total, K)
        rfq.rfq_quantize_act(x, x4, xr, None)
        xq = rfq.empty_qtensor(F8, MMA, total, K)
        rfq.rfq_convert(x4, xq)
        rfq.rfq_linear_grouped(xq, xr, None, 256, torch.from_numpy(off).to(DEV), w8, N, y, out, ws)
    assert rfq.rfq_workspace_status(ws) == rfq.RFQ_OK
    yh = y.float().cpu().numpy()
    # the oracle, group by group (phi tiles are 128-row tiles of the stacked X)
    res_fmt = {"rfq4": orc.FMT_MXFP4, "rfq8": orc.FMT_MXFP8, "w4a8": None}[fmt]
    if fmt == "w4a8":
        q = orc.quantize_act(xb, orc.FMT_MXFP8, orc.PHI_NONE)
    else:
        q = orc.quantize_act(xb, orc.FMT_MXFP4, mode, tau, 128, r_s, res_fmt=res_fmt)
    for g in range(G):
        if counts[g] == 0:
            continue
        rows = slice(starts[g], ends[g])
        wc, wsf = orc.quantize_weight(wbs[g], orc.FMT_MXFP4)
        if fmt == "w4a8":
            ref = orc.linear(orc.FMT_MXFP8, q["main_codes"][rows], q["main_scales"][rows], None, None, wc, wsf,
                             counts[g], K, N, w_fmt=orc.FMT_MXFP4)
        else:
            ref = orc.linear(orc.FMT_MXFP4, q["main_codes"][rows], q["main_scales"][rows], q["res_codes"][rows],
                             q["res_scales"][rows], wc, wsf, counts[g], K, N, res_fmt=res_fmt,
                             w_fmt=orc.FMT_MXFP4)
        check_y(yh[rows], ref, bf16=(out == rfq.RFQ_OUT_BF16))
    # group g spans rows [off[g], off[g+1]): its zero padding rows give zero
    # rows of Y; rows from off[G] on belong to no group and are not written
    real = np.zeros(total, bool)
    for s_, e_ in zip(starts, ends):
        real[s_:e_] = True
    pad = ~real
    pad[ends[-1]:] = False
    assert (yh[pad] == 0).all()
    assert np.isnan(yh[ends[-1]:]).all()
    return yh


@pytest.mark.parametrize("counts,K,N", [([300, 0, 1, 128, 257], 512, 256), ([5, 130, 64], 640, 384),
                                         ([128] * 3, 256, 128)])
def test_grouped_rfq_mxfp4(orc, counts, K, N):
    _case(orc, counts, K, N)


def test_grouped_many_groups_many_tiles(orc):
    """48 groups of 1..400 rows, 3 column tiles each: more tiles than CTA
    pairs, so every pair walks several groups."""
    rng = np.random.default_rng(3)
    counts = [int(c) for c in rng.integers(1, 400, size=48)]
    _case(orc, counts, 256, 768, out=rfq.RFQ_OUT_BF16, seed=7)


def test_grouped_long_groups_on_cta_pairs(orc):
    """Groups averaging 2048 stacked rows or more run on 256-row CTA pairs
    (shorter ones on 128-row tiles of single CTAs): both forms are checked,
    with a group ending inside a 32-row output box."""
    _case(orc, [2100, 2500], 256, 256, seed=13)
    _case(orc, [2100, 2500], 256, 256, out=rfq.RFQ_OUT_BF16, seed=14)


def test_grouped_selective_phi(orc):
    _case(orc, [200, 333, 70], 1152, 256, mode=rfq.RFQ_FALLBACK_AMAX, tau=30.0, r_s=128, seed=9)


@pytest.mark.parametrize("packed_w", [False, True])
@pytest.mark.parametrize("fmt", ["w4a8", "rfq8"])
def test_grouped_mxfp8(orc, fmt, packed_w):
    _case(orc, [150, 0, 260, 9], 512, 256, fmt=fmt, seed=11, packed_w=packed_w)


def test_grouped_bad_offsets_are_reported(orc):
    K, N, G = 256, 128, 2
    total = 256
    x = to_dev_bf16(make_activation(ActSpec(total, K, "normal", seed=1)))
    w = to_dev_bf16(make_weight(K, G * N, seed=2))
    xq = rfq.empty_qtensor(F4, MMA, total, K)
    rfq.rfq_quantize_act(x, xq, None, None, mode=rfq.RFQ_FALLBACK_NONE)
    wq = rfq.empty_qtensor(F4, MMA, G * N, K)
    rfq.rfq_quantize_weight(w, wq)
    ws = torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=DEV)
    for bad in ([0, 100, 256], [0, 256, 128], [0, 128, 300]):   # unaligned start, decreasing, past the rows
        y = guarded_full((total, N), float("nan"), torch.float32)
        off = torch.tensor(bad, dtype=torch.int32, device=DEV)
        rfq.rfq_linear_grouped(xq, None, None, 256, off, wq, N, y, rfq.RFQ_OUT_F32, ws)
        assert rfq.rfq_workspace_status(ws, clear=True) == rfq.RFQ_ERR_SHAPE
        assert torch.isnan(y).all()
