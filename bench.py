"""Benchmark of the RFQ W4A4 linear layer on GB300.

One step = one pass of the hot path over one batch: the one-pass activation
quantizer (main + residual MXFP4 codes and scales) followed by the RFQ GEMM
(main and residual MMAs into one accumulator, bf16 Y).  The weight is
quantized once before timing (an offline step).  Workload: the Wan2.2-14B
DiT FFN up projection, X [32760 x 5120] bf16, W [5120 x 13824], synthetic.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl rfq|reference]

Prints one JSON line (rank 0).  `value` is executed tensor throughput in
TFLOP/s summed over ranks (2*M*N*K for the main product plus the same again
for the residual product on phi = 1 tiles).  Under torchrun every rank runs
the full workload on its own GPU (token rows shard across GPUs with no
exchange): weak scaling.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)

WORKLOAD = "wan_ffn_up"
METRIC = "RFQ W4A4 linear TFLOP/s & % FP4 MMA peak; act-quant HBM GB/s (1xGB300)"
UNIT = "TFLOP/s"
FP4_OVER_BF16 = 13.5 / 2.25   # nominal dense FP4 : BF16 tensor rate of GB300


def _peaks():
    p = os.path.join(HERE, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16_burst=d["bf16_tflops"], bf16_sust=d["bf16_tflops_sustained"],
                    src="measured")
    return dict(hbm=6800.0, bf16_burst=1900.0, bf16_sust=1700.0, src="fallback")


def _kernel_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current kernel sources (matching hash); else None."""
    path = os.path.join(HERE, "profiles", "dram_traffic.txt")
    if not os.path.exists(path):
        return None
    h = _src_hash()
    for line in open(path):
        f = line.split()
        if len(f) >= 4 and not line.startswith("#") and f[0] == kernel and f[1] == workload and f[2] == h:
            return float(f[3])
    return None


def _src_hash():
    d = os.path.join(HERE, "paper_2608_26581_gb300", "csrc")
    m = hashlib.sha256()
    for n in sorted(os.listdir(d)):
        m.update(open(os.path.join(d, n), "rb").read())
    return m.hexdigest()[:16]


class ClockSampler:
    """Samples SM clocks and throttle reasons with nvidia-smi while running."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.f = None

    def __enter__(self):
        self.f = tempfile.TemporaryFile(mode="w+")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            self.proc.wait()

    def summary(self):
        if self.proc is None:
            return None
        self.f.seek(0)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.f:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 7:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _workload(rows: int = 0):
    """The benchmark workload; rows > 0 keeps only the first `rows` token
    rows (a smaller case of the same kernels, for profiler captures)."""
    import dataclasses
    from paper_2608_26581_gb300.synth import WORKLOADS
    spec = WORKLOADS[WORKLOAD]
    if rows and rows < spec.act.M:
        spec = dataclasses.replace(spec, name=f"{spec.name}_first{rows}rows",
                                   act=dataclasses.replace(spec.act, M=rows))
    return spec


def _config(spec, extra=None):
    c = {"workload": spec.name, "M": spec.act.M, "K": spec.act.K, "N": spec.N, "main_format": "mxfp4",
         "residual_format": "mxfp4", "phi": "all tiles (phi = 1)", "y_dtype": "bf16",
         "inputs": "synthetic: X N(0,1), 1% outlier channels x64, 0.1% tokens x200; W N(0,0.02)",
         "l2": "inputs larger than L2 (X 335 MB, Y 906 MB per step), no flush"}
    if extra:
        c.update(extra)
    return c


def cpu_oracle_sample(rows_per_call: int = 8, calls: int = 2):
    """Times the CPU oracle (single thread, fp64) on a bounded sample of the
    workload: `calls` x (quantize + RFQ GEMM of `rows_per_call` token rows
    against the full quantized weight).  Returns (TFLOP/s, seconds, sample)."""
    import oracle
    from paper_2608_26581_gb300.synth import ActSpec, make_activation, make_weight
    spec = _workload()
    K, N = spec.act.K, spec.N
    a = spec.act
    xb = make_activation(ActSpec(rows_per_call * calls, K, a.body, a.body_scale, a.chan_frac, a.chan_count,
                                 a.chan_scale, 0.0, None, 1.0, a.seed))
    wb = make_weight(K, N, seed=a.seed)
    wc, ws = oracle.quantize_weight(wb)
    t0 = time.perf_counter()
    for i in range(calls):
        x = xb[i * rows_per_call:(i + 1) * rows_per_call]
        q = oracle.quantize_act(x)
        oracle.linear(0, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"], wc, ws,
                      rows_per_call, K, N)
    dt = time.perf_counter() - t0
    flop = 2.0 * 2.0 * rows_per_call * calls * N * K
    sample = (f"{calls} x (quantize_act + RFQ linear) of {rows_per_call} rows of X [.., {K}] "
              f"against the full W~ [{N} x {K}] (weight quantization untimed)")
    return flop / dt / 1e12, dt, sample


def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return
    spec = _workload()
    for _ in range(args.warmup):
        cpu_oracle_sample(rows_per_call=2, calls=1)
    vals, times = [], []
    sample = ""
    for _ in range(args.steps):
        v, dt, sample = cpu_oracle_sample(rows_per_call=2, calls=1)
        vals.append(v)
        times.append(dt)
    value = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * statistics.median(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": _config(spec, {"sample": sample}),
            "cpu_baseline": {"kind": "oracle", "cores": 1, "sample": sample, "value": value, "unit": UNIT},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)


def run_rfq(args):
    import torch
    import torch.distributed as dist

    from paper_2608_26581_gb300 import rfq
    from paper_2608_26581_gb300.synth import make_activation, make_weight

    ws, rank, local = _dist()
    if ws > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    spec = _workload(args.rows)
    M, K, N = spec.act.M, spec.act.K, spec.N
    F, L = rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA

    xb = make_activation(spec.act)
    wb = make_weight(K, N, seed=spec.act.seed)
    x_host = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).pin_memory()
    w = torch.from_numpy(wb.view(np.int16)).to(dev).view(torch.bfloat16)
    x = x_host.to(dev)
    wq = rfq.empty_qtensor(F, L, N, K, device=dev)
    rfq.rfq_quantize_weight(w, wq)                         # offline weight step, untimed
    xq = rfq.empty_qtensor(F, L, M, K, device=dev)
    xr = rfq.empty_qtensor(F, L, M, K, device=dev)
    y = torch.empty(M, N, dtype=torch.bfloat16, device=dev)
    y_host = torch.empty(M, N, dtype=torch.bfloat16).pin_memory()
    wsp = torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)

    ev = lambda: torch.cuda.Event(enable_timing=True)
    per_step = [(ev(), ev(), ev()) for _ in range(args.steps)]

    def step(i=None):
        if i is not None:
            per_step[i][0].record(stream)
        rfq.rfq_quantize_act(x, xq, xr, None, stream=stream)
        if i is not None:
            per_step[i][1].record(stream)
        rfq.rfq_linear(xq, xr, None, 256, wq, y, rfq.RFQ_OUT_BF16, wsp, stream=stream)
        if i is not None:
            per_step[i][2].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if rfq.rfq_workspace_status(wsp) != rfq.RFQ_OK:
        raise RuntimeError("rfq_linear reported a device timeout")

    def barrier():
        if ws > 1:
            dist.barrier()

    t_start, t_end = ev(), ev()
    with ClockSampler(local) as clk:
        barrier()
        torch.cuda.synchronize()
        t_start.record(stream)
        for i in range(args.steps):
            step(i)
        t_end.record(stream)
        torch.cuda.synchronize()
        barrier()
    ms = t_start.elapsed_time(t_end) / args.steps
    q_ms = statistics.mean(a.elapsed_time(b) for a, b, _ in per_step)
    g_ms = statistics.mean(b.elapsed_time(c) for _, b, c in per_step)
    if ws > 1:
        t = torch.tensor([ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())

    # end to end through the public API with host buffers
    e2e_ms = None
    for i in range(0 if args.no_e2e else args.warmup + args.steps):
        if i == args.warmup:
            barrier()
            torch.cuda.synchronize()
            e0, e1 = ev(), ev()
            e0.record(stream)
        x.copy_(x_host, non_blocking=True)
        step()
        y_host.copy_(y, non_blocking=True)
    if not args.no_e2e:
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        e2e_ms = e0.elapsed_time(e1) / args.steps
    if ws > 1 and e2e_ms is not None:
        t = torch.tensor([e2e_ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        e2e_ms = float(t.item())
    if rfq.rfq_workspace_status(wsp) != rfq.RFQ_OK:
        raise RuntimeError("rfq_linear reported a device timeout")

    flop = 2.0 * 2.0 * M * N * K                 # main + residual product, phi = 1 everywhere
    value = ws * flop / (ms * 1e-3) / 1e12
    pk = _peaks()
    fp4_peak = pk["bf16_sust"] * FP4_OVER_BF16
    gemm_tflops = flop / (g_ms * 1e-3) / 1e12
    aq_bytes = M * K * 2 + 2 * (M * K // 2) + 2 * (((M + 127) // 128) * 128 * K // 32)
    aq_gbs = aq_bytes / (q_ms * 1e-3) / 1e9
    clocks = clk.summary()

    if rank == 0:
        cpu = None
        if ws == 1 and not args.no_cpu_baseline:
            v, dt, sample = cpu_oracle_sample()
            cpu = {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample,
                   "seconds": round(dt, 2)}
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "mxfp4 (e2m1 x e2m1, fp32 accumulate)", "data": "synthetic",
            "config": _config(spec, {"parallelism": f"dp{ws} over token rows" if ws > 1 else "single GPU"}),
            "effective_tflops_2mnk": ws * flop / 2 / (ms * 1e-3) / 1e12,
            "roofline": {"bound": "tensor", "kernel": "gemm_mxf4_kernel", "achieved": gemm_tflops,
                         "peak": fp4_peak, "unit": "TFLOP/s", "frac": gemm_tflops / fp4_peak,
                         "traffic": _kernel_traffic("gemm_mxf4_kernel", spec.name),
                         "flop_per_launch": flop, "ms_per_launch": g_ms,
                         "peak_source": f"{pk['src']} bf16 sustained {pk['bf16_sust']} TFLOP/s x "
                                        f"{FP4_OVER_BF16:g} (nominal dense FP4/BF16 ratio), of {pk['src']}"},
            "act_quant": {"bound": "hbm", "kernel": "act_quant_mxfp4_kernel", "achieved": aq_gbs,
                          "peak": pk["hbm"], "unit": "GB/s", "frac": aq_gbs / pk["hbm"],
                          "bytes_per_launch": aq_bytes, "ms_per_launch": q_ms,
                          "traffic": _kernel_traffic("act_quant_mxfp4_kernel", spec.name)},
            "e2e": None if e2e_ms is None else {
                "value": ws * flop / (e2e_ms * 1e-3) / 1e12, "unit": UNIT, "ms_per_step": e2e_ms,
                "h2d_bytes_per_step": M * K * 2, "d2h_bytes_per_step": M * N * 2},
            "gpu_launches": 2 * args.steps,
            "clocks": clocks,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if ws > 1:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="rfq", choices=["rfq", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end (host buffer) timing")
    ap.add_argument("--rows", type=int, default=0, help="profile a smaller case: the first ROWS token rows")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_rfq(args)


if __name__ == "__main__":
    main()
