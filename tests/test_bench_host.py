"""Host-side logic of bench.py that needs no GPU: the clock-sample
summary over the loaded window, the launch count it claims per step, the
oracle baseline's units and its multi-process timing (on a tiny workload)."""
import datetime
import os
import sys
import tempfile

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _sampler_with(lines):
    cs = bench.ClockSampler(0)
    cs.proc = object()            # as if nvidia-smi had started
    cs.f = tempfile.TemporaryFile(mode="w+")
    cs.f.write("\n".join(lines) + "\n")
    return cs


def _ts(t):
    return datetime.datetime.fromtimestamp(t).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]


def test_clock_summary_keeps_the_loaded_window():
    t0 = 1_800_000_000.0
    lines = [f"{_ts(t0 - 1.0)}, 2070, 2070, 200.0, Not Active, Not Active, Not Active, Not Active",
             f"{_ts(t0 + 0.10)}, 1500, 2070, 1390.0, Not Active, Not Active, Not Active, Active",
             f"{_ts(t0 + 0.12)}, 1600, 2070, 1395.0, Not Active, Not Active, Not Active, Active",
             f"{_ts(t0 + 0.14)}, 1700, 2070, 1380.0, Not Active, Not Active, Not Active, Not Active",
             f"{_ts(t0 + 2.0)}, 2070, 2070, 150.0, Not Active, Active, Not Active, Not Active",
             "garbage line"]
    s = _sampler_with(lines).summary(t0, t0 + 0.5)
    assert s["samples"] == 3 and s["sm_mhz"] == 1600 and s["sm_max_mhz"] == 2070
    assert s["reasons"] == ["sw_power_cap"] and s["window"].startswith("timed")
    # no sample inside the window: every sample counts
    s = _sampler_with(lines).summary(t0 + 10, t0 + 11)
    assert s["samples"] == 5 and "hw_thermal_slowdown" in s["reasons"] and s["window"] == "whole run"


def test_launches_per_step():
    L = bench._launches_per_step
    assert L(True, False, False, False, "rfq4", False) == 1          # quantizer alone
    assert L(False, True, False, False, "rfq4", False) == 1          # fused linear
    assert L(False, False, False, False, "rfq4", False) == 2         # quantizer + GEMM
    assert L(False, False, True, False, "rfq4", False) == 2          # HiF4: the quantizer writes the bf16 operands
    assert L(False, False, False, False, "rfq8", False) == 2         # rfq8: the quantizer writes X~ as E4M3
    assert L(False, False, False, False, "rfq4", True, True) == 2    # phi in the quantizer's pass
    assert L(False, False, False, False, "rfq4", True, False) == 3   # separate phi pass


def test_oracle_units():
    spec = bench._workload(0, "wan_ffn_up")
    work, unit, div = bench._oracle_units(spec, 8)
    assert unit == bench.UNIT and div == 1e12 and work == 2 * 2 * 8 * 13824 * 5120
    spec = bench._workload(0, "act_quant")
    work, unit, div = bench._oracle_units(spec, 64)
    assert unit == "GB/s" and work == 64 * 4096 * 3.0625


def test_oracle_timed_on_host_cores():
    """Spawned oracle processes on the tiny workload: one timing per
    repetition, a positive rate, the worker count in the sample text."""
    n, unit, sample, reps = bench.cpu_oracle_timed("tiny", 2, 1, 2, workers=2)
    assert n == 2 and unit == bench.UNIT and len(reps) == 2
    assert all(v > 0 and dt > 0 for v, dt in reps)
    assert "2 processes on 2 host cores" in sample
    n, _, sample, reps = bench.cpu_oracle_timed("act_quant", 64, 1, 1, workers=1)
    assert n == 1 and reps[0][0] > 0 and "processes" not in sample


def test_act_quant_algorithmic_bytes():
    """The per-launch byte counts the roofline divides by (X read once,
    every output written once)."""
    B = bench._act_quant_bytes
    # Wan FFN, MXFP4 main + residual: 3.0625 B per element + the 128-row scale padding
    assert B(32760, 5120, "mxfp4", True) == 32760 * 5120 * 2 + 2 * (32760 * 5120 // 2 + 32768 * 160)
    assert B(32760, 5120, "mxfp4", True) == 513_679_360
    assert B(16384, 4096, "mxfp4", True) == 205_520_896          # the act-quant workload
    assert B(16384, 4096, "mxfp4", False) == 16384 * 4096 * 2 + 16384 * 4096 // 2 + 16384 * 128
    # HiF4 (Qwen down): codes, metadata and the bf16 values of X~ and X^
    hif4 = B(4096, 12288, "hif4", True, operand=True)
    assert hif4 == 4096 * 12288 * (2 + 2 * 0.5 + 2 * 2) + 2 * 4096 * 192 * 4
    # FP4-to-FP8 residual with X~ as E4M3: 2 + 0.5 + 1 + 1 bytes per element + three scale planes
    assert B(32760, 5120, "rfq8", True, operand=True) == 32760 * 5120 * 9 // 2 + 3 * 32768 * 160
    assert B(4096, 4096, "mxfp8", False) == 4096 * 4096 * 3 + 4096 * 128
