"""The debug build (librfq_debug.so, -DRFQ_DEBUG_BOUNDS): every direct
global store of the quantizers and the CTA-pair GEMM is checked against its
buffer's extent.  On cases that exercise those stores -- ragged rows in both
scale layouts, the fused quantizer's ring, a grouped GEMM whose group ends
inside a 32-row output box -- the debug build must record no out-of-range
store and give the normal build's bytes exactly."""
import os
import subprocess
import sys

import pytest

from conftest import ROOT

pytestmark = pytest.mark.gpu

_CASES = r'''
import sys, numpy as np, torch
sys.path.insert(0, ROOT); sys.path.insert(0, ROOT + "/tests")
from paper_2608_26581_gb300 import rfq
from paper_2608_26581_gb300.synth import ActSpec, make_activation, make_weight
from gpu_util import to_dev_bf16
F, MMA, ROW = rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, rfq.RFQ_SCALE_ROWMAJOR
out = []
def keep(*ts):
    for t in ts:
        out.append(t.view(torch.uint8).reshape(-1).cpu().numpy().copy())
# quantizers: ragged rows, both layouts, the fused AMAX form
for M, K, lay in ((300, 1024, MMA), (129, 640, ROW), (1, 256, MMA)):
    x = to_dev_bf16(make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, seed=M)))
    xq, xr = rfq.empty_qtensor(F, lay, M, K), rfq.empty_qtensor(F, lay, M, K)
    rfq.rfq_quantize_act(x, xq, xr)
    keep(xq.codes, xq.scales, xr.codes, xr.scales)
x = to_dev_bf16(make_activation(ActSpec(385, 1024, "normal", chan_count=2, chan_scale=64.0, seed=5)))
xq, xr = rfq.empty_qtensor(F, MMA, 385, 1024), rfq.empty_qtensor(F, MMA, 385, 1024)
phi = torch.empty(4 * 4, dtype=torch.uint8, device="cuda")
rfq.rfq_quantize_act(x, xq, xr, phi, mode=rfq.RFQ_FALLBACK_AMAX, tau=100.0, p_s=128, r_s=256)
keep(xq.codes, xq.scales, xr.codes, xr.scales, phi)
# weights, CTA-pair GEMM, fused quantizer ring
M, K, N = 700, 512, 272
wq = rfq.empty_qtensor(F, MMA, N, K)
rfq.rfq_quantize_weight(to_dev_bf16(make_weight(K, N, seed=7)), wq)
keep(wq.codes, wq.scales)
x = to_dev_bf16(make_activation(ActSpec(M, K, "normal", chan_count=2, chan_scale=64.0, seed=8)))
xq, xr = rfq.empty_qtensor(F, MMA, M, K), rfq.empty_qtensor(F, MMA, M, K)
rfq.rfq_quantize_act(x, xq, xr)
y = torch.zeros(M, N, dtype=torch.bfloat16, device="cuda")
ws = torch.zeros(64, dtype=torch.int32, device="cuda")
rfq.rfq_linear(xq, xr, None, 256, wq, y, rfq.RFQ_OUT_BF16, ws)
yf = torch.zeros(M, N, dtype=torch.float32, device="cuda")
rfq.rfq_linear_fused(x, wq, yf, rfq.RFQ_OUT_F32, rfq.fused_workspace(M, K))
keep(y, yf)
# grouped, long groups on CTA pairs, one ending inside a 32-row box
counts = [2100, 2500]
starts = [0, 2176]
total = 2176 + 2560
xs = np.zeros((total, K), np.uint16)
xs[0:2100] = make_activation(ActSpec(2100, K, "normal", seed=9))
xs[2176:2176 + 2500] = make_activation(ActSpec(2500, K, "normal", seed=10))
NG = 256   # the grouped GEMM's per-group N is a multiple of 128
wg = rfq.empty_qtensor(F, MMA, 2 * NG, K)
rfq.rfq_quantize_weight(to_dev_bf16(np.concatenate([make_weight(K, NG, seed=11), make_weight(K, NG, seed=12)], 1)), wg)
gq, gr = rfq.empty_qtensor(F, MMA, total, K), rfq.empty_qtensor(F, MMA, total, K)
rfq.rfq_quantize_act(to_dev_bf16(xs), gq, gr)
off = torch.tensor([0, 2176, 2176 + 2500], dtype=torch.int32, device="cuda")
yg = torch.zeros(total, NG, dtype=torch.float32, device="cuda")
rfq.rfq_linear_grouped(gq, gr, None, 256, off, wg, NG, yg, rfq.RFQ_OUT_F32, ws)
keep(yg)
torch.cuda.synchronize()
st, line = rfq.rfq_debug_bounds()
np.savez(OUT, *out, status=np.array([st, line]))
'''


def _run(lib, out_path):
    code = f"ROOT = {ROOT!r}\nOUT = {out_path!r}\n" + _CASES
    env = dict(os.environ, RFQ_LIBRARY=lib)
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=600)
    assert r.returncode == 0, r.stderr[-3000:]


def test_debug_build_records_no_out_of_range_store_and_matches(tmp_path):
    import numpy as np
    from paper_2608_26581_gb300 import _build, rfq
    debug_lib = _build.build(debug=True)
    _run(debug_lib, str(tmp_path / "debug.npz"))
    _run(_build.LIB, str(tmp_path / "normal.npz"))
    d, n = np.load(tmp_path / "debug.npz"), np.load(tmp_path / "normal.npz")
    assert list(d["status"]) == [rfq.RFQ_OK, 0], f"out-of-range store recorded at line {d['status'][1]}"
    assert list(n["status"])[0] == rfq.RFQ_ERR_UNSUPPORTED
    keys = [k for k in d.files if k.startswith("arr_")]
    assert len(keys) == len([k for k in n.files if k.startswith("arr_")]) and keys
    for k in keys:
        assert np.array_equal(d[k], n[k]), k
