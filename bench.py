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
import datetime
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

WORKLOAD = "wan_ffn_up"   # default; --workload picks another of synth.WORKLOADS
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


# source file of each timed kernel: its DRAM counters hold only for the
# sources they were taken on (the kernel's file plus the shared headers)
_KERNEL_SRC = {"gemm_mxf4_kernel": "gemm_mxf4.cu", "gemm_mxf4_pair_kernel": "gemm_mxf4_pair.cu",
               "act_quant8_kernel": "quant_mxfp8.cu", "act_quant_rfq8_amax_kernel": "quant_mxfp8.cu",
               "act_quant_rfq8_kernel": "quant_mxfp8.cu",
               "gemm_mxf4_fused_kernel": "gemm_mxf4_fused.cu",
               "act_quant_mxfp4_kernel": "quant_mxfp4.cu", "act_quant_mxfp4_amax_kernel": "quant_mxfp4.cu",
               "gemm_hif4_kernel": "gemm_hif4.cu", "act_quant_hif4_kernel": "quant_hif4.cu",
               "act_quant_hif4_amax_kernel": "quant_hif4.cu"}


def _kernel_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from profiles/dram_traffic.txt (an ncu capture of
    that kernel on that workload), if the kernel's sources still hash to the
    value recorded there; else None."""
    path = os.path.join(HERE, "profiles", "dram_traffic.txt")
    if not os.path.exists(path) or kernel not in _KERNEL_SRC:
        return None
    h = _src_hash(kernel)
    for line in open(path):
        f = line.split()
        if len(f) >= 4 and not line.startswith("#") and f[0] == kernel and f[1] == workload and f[2] == h:
            return float(f[3])
    return None


def _act_quant_bytes(rows: int, K: int, kind: str, residual: bool, operand: bool = False) -> int:
    """Algorithmic DRAM bytes of one activation-quantizer launch: X (bf16)
    read once and every output written once.  kind: "mxfp4" (E2M1 codes,
    E8M0 scales per 32, scale rows padded to 128), "hif4" (codes, a 32-bit
    metadata word per 64, rows padded to 128; operand: the bf16 values of X~
    and X^ too), "rfq8" (MXFP4 X~ and an MXFP8 residual; operand: X~ as
    E4M3 with its scales too), "mxfp8" (E4M3 codes and scales)."""
    rows_pad = (rows + 127) // 128 * 128
    x = rows * K * 2
    sf = rows_pad * (K // 32)
    paths = 2 if residual else 1
    if kind == "mxfp4":
        return x + paths * (rows * K // 2 + sf)
    if kind == "hif4":
        return x + paths * (rows * K // 2 + rows_pad * (K // 64) * 4) + (paths * rows * K * 2 if operand else 0)
    if kind == "rfq8":
        return x + (rows * K // 2 + sf) + (rows * K + sf) + ((rows * K + sf) if operand else 0)
    if kind == "mxfp8":
        return x + rows * K + sf
    raise ValueError(kind)


def _launches_per_step(quant_only, fused, hif4, no_res, scheme, amax_phi, amax_fused=False):
    """This library's kernel launches in one timed step."""
    if quant_only or fused:
        return 1
    n = 1 + (1 if amax_phi and not amax_fused else 0)   # quantizer (+ the phi amax kernel; the
                                                        # HiF4 quantizer also writes the bf16 values)
    return n + 1                            # GEMM


def _src_hash(kernel: str):
    d = os.path.join(HERE, "paper_2608_26581_gb300", "csrc")
    m = hashlib.sha256()
    extra = ("mxfp4_math.cuh",) if kernel in ("act_quant_mxfp4_kernel", "act_quant_mxfp4_amax_kernel",
                                              "gemm_mxf4_fused_kernel", "act_quant8_kernel", "act_quant_rfq8_kernel",
                                              "act_quant_rfq8_amax_kernel", "gemm_mxf4_pair_kernel") else ()
    for n in (_KERNEL_SRC[kernel], "ptx.cuh", "internal.h") + extra:
        m.update(open(os.path.join(d, n), "rb").read())
    return m.hexdigest()[:16]


class ClockSampler:
    """Samples SM clocks and throttle reasons with nvidia-smi (every 20 ms,
    each sample time-stamped) while running; `summary` keeps the samples
    inside a host-time window (the GPU's loaded interval)."""
    Q = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
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
                 "-lms", "20"], stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.1)
            self.proc.terminate()
            self.proc.wait()

    def summary(self, t0=None, t1=None, label="timed and warm-up replays"):
        """Median SM clock, max clock and the throttle reasons of the samples
        taken in [t0, t1] (host seconds, time.time()); all samples when no
        window is given or none falls inside it."""
        if self.proc is None:
            return None
        self.f.seek(0)
        rows = []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.f:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 8:
                continue
            try:
                ts = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                rows.append((ts, float(f[1]), float(f[2]), f[4:8]))
            except ValueError:
                continue
        if not rows:
            return None
        inside = [r for r in rows if t0 is not None and t0 <= r[0] <= t1]
        use = inside or rows
        reasons = sorted({n for r in use for n, v in zip(names, r[3]) if v.lower().startswith("active")})
        return {"sm_mhz": statistics.median(r[1] for r in use), "sm_max_mhz": max(r[2] for r in use),
                "samples": len(use), "window": label if inside else "whole run",
                "reasons": reasons}


class _Nvtx:
    """An NVTX range around a phase of the run (visible in a profiler's
    timeline; no cost otherwise)."""

    def __init__(self, name: str):
        self.name = name

    def __enter__(self):
        import torch
        torch.cuda.nvtx.range_push(self.name)

    def __exit__(self, *a):
        import torch
        torch.cuda.nvtx.range_pop()


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _max_over_ranks(value: float, ws: int, dist, device) -> float:
    """The largest `value` over all ranks (the job's time is its slowest
    rank's); `dist` is torch.distributed with an initialised group."""
    if ws == 1:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _job_rate(units_per_rank: float, ws: int, ms: float) -> float:
    """Whole-job throughput in units per second: every rank processes its own
    copy of the workload (weak scaling), the job takes the slowest rank's
    time."""
    return ws * units_per_rank / (ms * 1e-3)


def _workload(rows: int = 0, name: str = WORKLOAD, seed=None):
    """The benchmark workload; rows > 0 keeps only the first `rows` token
    rows (a smaller case of the same kernels, for profiler captures); seed
    replaces its input seed."""
    import dataclasses
    from paper_2608_26581_gb300.synth import WORKLOADS
    spec = WORKLOADS[name]
    if seed is not None:
        spec = dataclasses.replace(spec, act=dataclasses.replace(spec.act, seed=seed))
    if rows and rows < spec.act.M:
        spec = dataclasses.replace(spec, name=f"{spec.name}_first{rows}rows",
                                   act=dataclasses.replace(spec.act, M=rows))
    return spec


def _inputs_desc(a):
    body = {"normal": "N(0,1)", "student_t3": "Student-t(3)", "laplace": f"Laplace(0,{a.body_scale:g})"}[a.body]
    d = f"synthetic: X {body}"
    if a.chan_count or a.chan_frac:
        d += f", {a.chan_count if a.chan_count is not None else f'{100 * a.chan_frac:g}%'} outlier channels x{a.chan_scale:g}"
    if a.tok_count or a.tok_frac:
        d += f", {a.tok_count if a.tok_count is not None else f'{100 * a.tok_frac:g}%'} tokens x{a.tok_scale:g}"
    return d + "; W N(0,0.02)"


def _config(spec, extra=None):
    M, K, N = spec.act.M, spec.act.K, spec.N
    x_mb, y_mb = M * K * 2 / 1e6, M * N * 2 / 1e6
    c = {"workload": spec.name, "M": M, "K": K, "N": N, "seed": spec.act.seed, "main_format": spec.fmt,
         "residual_format": spec.fmt, "phi": "all tiles (phi = 1)", "y_dtype": "bf16",
         "inputs": _inputs_desc(spec.act),
         "l2": (f"inputs larger than L2 (X {x_mb:.0f} MB, Y {y_mb:.0f} MB per step; two buffer sets "
                f"alternate between steps), no flush" if x_mb + y_mb > 129 else
                "working set below L2 size (two buffer sets alternate between steps)")}
    if extra:
        c.update(extra)
    return c


_ORACLE_W = {}


def _oracle_weight(spec):
    """The oracle's quantized weight of a workload (computed once per process:
    weight quantization is an offline step, not part of the timed sample)."""
    import oracle
    from paper_2608_26581_gb300.synth import make_weight
    if spec.name not in _ORACLE_W:
        fmt = oracle.FMT_HIF4 if spec.fmt == "hif4" else oracle.FMT_MXFP4
        _ORACLE_W[spec.name] = oracle.quantize_weight(make_weight(spec.act.K, spec.N, seed=spec.act.seed), fmt)
    return _ORACLE_W[spec.name]


def _oracle_rows(spec, rows: int, part: int = 0):
    """Synthetic token rows for the CPU oracle sample (the workload's
    distribution; `part` selects a distinct seeded draw per worker)."""
    from paper_2608_26581_gb300.synth import ActSpec, make_activation
    a = spec.act
    return make_activation(ActSpec(rows, a.K, a.body, a.body_scale, a.chan_frac, a.chan_count,
                                   a.chan_scale, 0.0, None, 1.0, a.seed + 1000 * part))


def _oracle_run(spec, xb, rows_per_call: int, calls: int, wq):
    """The timed oracle work: `calls` x (quantize + RFQ GEMM of
    `rows_per_call` rows against the full quantized weight), or quantization
    alone for the quantizer-only workload."""
    import oracle
    fmt = oracle.FMT_HIF4 if spec.fmt == "hif4" else oracle.FMT_MXFP4
    K, N = spec.act.K, spec.N
    for i in range(calls):
        x = xb[i * rows_per_call:(i + 1) * rows_per_call]
        q = oracle.quantize_act(x, fmt)
        if N:
            oracle.linear(fmt, q["main_codes"], q["main_scales"], q["res_codes"], q["res_scales"], wq[0], wq[1],
                          rows_per_call, K, N)


def _oracle_units(spec, rows: int):
    """(work, unit, divisor) of `rows` oracle rows in the bench's metric:
    TFLOP of the main + residual product, or GB of the quantizer's bytes."""
    if spec.N:
        return 2.0 * 2.0 * rows * spec.N * spec.act.K, UNIT, 1e12
    per_elem = 3.125 if spec.fmt == "hif4" else 3.0625
    return rows * spec.act.K * per_elem, "GB/s", 1e9


def _oracle_sample_desc(spec, rows_per_call: int, calls: int, workers: int):
    K, N = spec.act.K, spec.N
    per = (f"{calls} x (quantize_act + RFQ linear) of {rows_per_call} rows of X [.., {K}] against the full "
           f"W~ [{N} x {K}] (weight quantization untimed)" if N else
           f"{calls} x quantize_act (main + residual) of {rows_per_call} rows of X [.., {K}]")
    return (f"{workers} processes on {workers} host cores, each: {per}; wall time from a common start"
            if workers > 1 else per)


def _oracle_workers(spec) -> int:
    """Processes for the CPU baseline: one per host core while the free
    memory holds each one's copy of the quantized weight and the oracle's
    fp64 expansion of it (plus headroom)."""
    n = min(os.cpu_count() or 1, 64)
    need = (spec.N * spec.act.K * 12 + (1 << 30)) if spec.N else (1 << 30)
    try:
        with open("/proc/meminfo") as f:
            avail = next(int(l.split()[1]) * 1024 for l in f if l.startswith("MemAvailable:"))
        n = min(n, max(1, avail // 2 // need))
    except (OSError, StopIteration, ValueError):
        n = 1
    return int(max(1, n))


def _oracle_proc(key, rows_per_call, calls, reps, part, barrier, q):
    """One worker of the multi-core CPU baseline: its own rows, the same
    bounded sample as the others, every repetition started together at a
    barrier (spawned process: no CUDA in it)."""
    try:
        spec = _workload(0, key)
        wq = _oracle_weight(spec) if spec.N else None
        xb = _oracle_rows(spec, rows_per_call * calls, part)
        for r in range(reps):
            barrier.wait(timeout=1800)
            t0 = time.monotonic()
            _oracle_run(spec, xb, rows_per_call, calls, wq)
            q.put((r, t0, time.monotonic()))
    except Exception as e:  # reported to the parent, which raises
        q.put(("error", repr(e), 0.0))


def cpu_oracle_timed(key: str, rows_per_call: int, calls: int, reps: int, workers: int = 0):
    """Times the CPU oracle (fp64, as it stands) on a bounded sample of the
    workload `key` (of synth.WORKLOADS) on the host cores: one spawned
    process per core (up to 64, as memory allows; or `workers`), each
    running `calls` x `rows_per_call` rows, `reps` times, all starting
    together.  Returns (workers, unit, sample, [(value, seconds)] per
    repetition), the value being the whole sample's work over the
    repetition's wall time in the bench's metric."""
    import multiprocessing
    spec = _workload(0, key)
    n = workers if workers > 0 else _oracle_workers(spec)
    ctx = multiprocessing.get_context("spawn")
    barrier, q = ctx.Barrier(n), ctx.Queue()
    procs = [ctx.Process(target=_oracle_proc, args=(key, rows_per_call, calls, reps, i, barrier, q),
                         daemon=True) for i in range(n)]
    for p_ in procs:
        p_.start()
    got = []
    try:
        for _ in range(n * reps):
            r = q.get(timeout=3600)
            if r[0] == "error":
                raise RuntimeError(f"CPU oracle worker failed: {r[1]}")
            got.append(r)
    finally:
        for p_ in procs:
            p_.join(timeout=60)
    work, unit, div = _oracle_units(spec, n * rows_per_call * calls)
    out = []
    for rep in range(reps):
        t = [(t0, t1) for r_, t0, t1 in got if r_ == rep]
        wall = max(b for _, b in t) - min(a for a, _ in t)
        out.append((work / wall / div, wall))
    return n, unit, _oracle_sample_desc(spec, rows_per_call, calls, n), out


def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return
    spec = _workload(0, args.workload, args.seed)
    rows = 8 if spec.N else 64   # 8 rows share each call's fp64 expansion of W~
    n, unit, sample, reps = cpu_oracle_timed(args.workload, rows, 1, args.warmup + args.steps)
    timed = reps[args.warmup:]
    value = statistics.median(v for v, _ in timed)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": unit, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * statistics.median(t for _, t in timed),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": _config(spec, {"sample": sample}),
            "cpu_baseline": {"kind": "oracle", "cores": n, "sample": sample, "value": value, "unit": unit},
            "e2e": {"value": value, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
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
    spec = _workload(args.rows, args.workload, args.seed)
    M, K, N = spec.act.M, spec.act.K, spec.N
    hif4 = spec.fmt == "hif4"
    quant_only = N == 0
    fused = args.variant == "fused"
    if fused and (hif4 or quant_only):
        raise SystemExit("--variant fused applies to the MXFP4 linear workloads")
    # selective fallback: phi(p, r) = [max |x| over the 128 x 256 tile > tau]
    # (Sec. 4.3); the GEMMs skip the residual loads and MMAs of phi = 0 tiles
    amax_phi = args.phi_tau is not None
    if amax_phi and (fused or quant_only):
        raise SystemExit("--phi-tau applies to the two-kernel linear workloads")
    # plain W4A4 (no residual pathway): the baseline RFQ's correction adds to
    no_res = args.no_residual
    if no_res and (fused or quant_only or amax_phi):
        raise SystemExit("--no-residual applies to the two-kernel linear workloads without --phi-tau")
    # MXFP8 schemes (Table 1 baselines and the FP4-to-FP8 residual of Sec. 4.2):
    #   rfq8: MXFP4 main + MXFP8 residual, both on the FP8 path (X~
    #         re-encoded exactly as E4M3 by the quantizer in the same pass,
    #         W~ multiplied as E2M1 from its packed codes); w4a8: MXFP8 X x
    #         MXFP4 W (E2M1); w8a8: MXFP8 X x MXFP8 W.  All on kind::mxf8f6f4.
    #   rfq8mix: the rfq8 RFQ through rfq_linear_mixed -- the main product
    #         on kind::mxf4 (X~ and W~ packed), the residual on
    #         kind::mxf8f6f4 (X^ as E4M3, W~ expanded from its packed codes
    #         by the copy engine); no E4M3 copy of X~ or W~.
    scheme = args.scheme
    mixed = scheme == "rfq8mix"
    f8 = scheme != "rfq4"
    if f8 and (hif4 or quant_only or fused or no_res):
        raise SystemExit("--scheme applies to the MXFP4 linear workloads (two-kernel, with residual flags unset)")
    if amax_phi and scheme in ("w4a8", "w8a8"):
        raise SystemExit("--phi-tau needs a residual pathway")
    if mixed and spec.groups > 0:
        raise SystemExit("--scheme rfq8mix runs the plain (ungrouped) GEMM")
    F = rfq.RFQ_FMT_HIF4 if hif4 else rfq.RFQ_FMT_MXFP4
    amax_fused = amax_phi and K % 256 == 0   # phi computed in the quantizer's pass
    L = rfq.RFQ_SCALE_MMA

    xb = make_activation(spec.act)
    # grouped (mixture-of-experts) workload: the routed rows of each expert,
    # stacked with every expert starting on a 128-row boundary (zero rows
    # between); one launch multiplies each expert's rows by its own W~
    grouped = spec.groups > 0
    Mb = M   # rows of the stacked buffers
    if grouped:
        if hif4 or fused or quant_only:
            raise SystemExit("grouped workloads run the MXFP4 / MXFP8 two-kernel path")
        from paper_2608_26581_gb300.synth import group_layout, make_group_counts
        counts = make_group_counts(M, spec.groups, seed=spec.act.seed)
        starts, ends, Mb = group_layout(counts)
        xs = np.zeros((Mb, K), np.uint16)
        cum = np.concatenate([[0], np.cumsum(counts)])
        for g in range(spec.groups):
            xs[starts[g]:ends[g]] = xb[cum[g]:cum[g + 1]]
        xb = xs
        group_off = torch.tensor(np.concatenate([starts, ends[-1:]]).astype(np.int32), device=dev)
    x_host = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).pin_memory()
    x = x_host.to(dev)
    wop = None
    NW = N * (spec.groups if grouped else 1)   # weight rows (every expert's W~ stacked)
    if not quant_only:
        wb = make_weight(K, NW, seed=spec.act.seed)
        w = torch.from_numpy(wb.view(np.int16)).to(dev).view(torch.bfloat16)
        wq = rfq.empty_qtensor(rfq.RFQ_FMT_MXFP8 if scheme == "w8a8" else F, L, NW, K, device=dev)
        rfq.rfq_quantize_weight(w, wq)                     # offline weight step, untimed
        if hif4:
            wop = rfq.empty_bf16_operand(N, K, device=dev)  # exact bf16 expansion of W~ (offline)
            rfq.rfq_dequant(wq, wop.codes)
        else:
            wop = wq
        del w
    no_res = no_res or scheme in ("w4a8", "w8a8")

    def buffer_set(xd):
        """The device buffers of one step: X and everything the step writes."""
        b = {"x": xd,
             "xq": rfq.empty_qtensor(rfq.RFQ_FMT_MXFP8 if scheme in ("w4a8", "w8a8") else F, L, Mb, K, device=dev),
             "xr": None if no_res else
                   rfq.empty_qtensor(rfq.RFQ_FMT_MXFP8 if scheme in ("rfq8", "rfq8mix") else F, L, Mb, K,
                                     device=dev),
             # rfq8: the E4M3 re-encoding of X~ that the GEMM multiplies
             "xq8": rfq.empty_qtensor(rfq.RFQ_FMT_MXFP8, L, Mb, K, device=dev) if scheme == "rfq8" else None,
             "phi": (torch.empty(((Mb + 127) // 128) * ((K + 255) // 256), dtype=torch.uint8, device=dev)
                     if amax_phi else None),
             # HiF4: the GEMM takes the exact bf16 expansions of X~ and X^
             # (expanding once per activation, not once per output tile)
             "xq16": rfq.empty_bf16_operand(M, K, device=dev) if hif4 and not quant_only else None,
             "xr16": rfq.empty_bf16_operand(M, K, device=dev) if hif4 and not quant_only and not no_res else None,
             "y": torch.empty(Mb, max(N, 16), dtype=torch.bfloat16, device=dev)}
        return b

    # Two buffer sets, used by alternate steps: no step finds in L2 what the
    # step before it read or wrote (each set's X plus its outputs exceeds
    # L2 for every workload but the tiny parity case).
    bufs = [buffer_set(x), buffer_set(x.clone())]
    y_host = torch.empty(Mb, max(N, 16), dtype=torch.bfloat16).pin_memory()
    # the GEMM workspace; the fused variant's also holds the in-GEMM quantizer's
    # unit counters and scratch codes (one workspace: the steps never overlap)
    wsp = (rfq.fused_workspace(Mb, K, rfq.RFQ_FALLBACK_ALL, device=dev) if fused else
           torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=dev))
    stream = torch.cuda.current_stream(dev)
    # quantizer-only workload: its result (both pathways' codes and scales) is read back
    q_out = lambda b: [b["xq"].codes, b["xq"].scales, b["xr"].codes, b["xr"].scales]
    host_q = [torch.empty_like(t, device="cpu").pin_memory() for t in q_out(bufs[0])] if quant_only else []
    q_bytes = sum(t.numel() for t in host_q)

    ev = lambda: torch.cuda.Event(enable_timing=True)

    # Events between the step's phases, recorded inside the captured graph
    # (event-record nodes): q = the quantizer (for HiF4 it also writes the
    # bf16 values of X~ and X^, for rfq8 X~ as E4M3), g = the GEMM (events 2
    # and 3; event 1 = event 2 marks the end of the quantizer).
    per_step = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(4)]
                for _ in range(args.steps)]

    def step(i=None, r=0):
        """One step on buffer set r; with i, events mark its phases."""
        bs = bufs[r]
        x_, xq, xr, xq8, ph, y_ = bs["x"], bs["xq"], bs["xr"], bs["xq8"], bs["phi"], bs["y"]
        # (recorded on the current stream: the capture stream inside the graph)
        mark = ((lambda j: per_step[i][j].record(torch.cuda.current_stream(dev))) if i is not None
                else (lambda j: None))
        if fused:
            # the quantizer runs inside the GEMM: one kernel per step
            for j in range(3):
                mark(j)
            rfq.rfq_linear_fused(x_, wop, y_, rfq.RFQ_OUT_BF16, wsp, stream=None)
            mark(3)
            return
        mark(0)
        mode = rfq.RFQ_FALLBACK_AMAX if amax_phi else (rfq.RFQ_FALLBACK_NONE if no_res else rfq.RFQ_FALLBACK_ALL)
        tau = args.phi_tau if amax_phi else 0.0
        if hif4 and not quant_only:
            # HiF4: the quantizer also writes the exact bf16 values of X~ and
            # X^ that the bf16 GEMM multiplies (no separate expansion pass)
            rfq.rfq_quantize_act_expand(x_, xq, xr, bs["xq16"], bs["xr16"], ph, mode=mode, tau=tau,
                                        p_s=128, r_s=256, stream=None)
        elif xq8 is not None:
            # rfq8: the quantizer also writes X~ re-encoded as MXFP8 (E4M3)
            rfq.rfq_quantize_act_expand(x_, xq, xr, xq8, None, ph, mode=mode, tau=tau, p_s=128, r_s=256,
                                        stream=None)
        else:
            rfq.rfq_quantize_act(x_, xq, xr, ph, mode=mode, tau=tau, p_s=128, r_s=256, stream=None)
        mark(1)
        mark(2)
        if quant_only:
            pass
        elif hif4:
            rfq.rfq_linear(bs["xq16"], bs["xr16"], ph, 256, wop, y_, rfq.RFQ_OUT_BF16, wsp, stream=None)
        elif grouped:
            rfq.rfq_linear_grouped(xq8 if xq8 is not None else xq, xr, ph, 256, group_off,
                                   wop, N, y_, rfq.RFQ_OUT_BF16, wsp, stream=None)
        elif mixed:
            rfq.rfq_linear_mixed(xq, xr, ph, 256, wq, y_, rfq.RFQ_OUT_BF16, wsp, stream=None)
        else:
            rfq.rfq_linear(xq8 if xq8 is not None else xq, xr, ph, 256, wop, y_, rfq.RFQ_OUT_BF16, wsp,
                           stream=None)
        mark(3)

    with _Nvtx("rfq warm-up steps (eager)"):
        for i in range(args.warmup):
            step(None, i & 1)
        torch.cuda.synchronize()
    if rfq.rfq_workspace_status(wsp) != rfq.RFQ_OK:
        raise RuntimeError("rfq_linear reported a device timeout")

    def barrier():
        if ws > 1:
            dist.barrier()

    def capture(instrumented):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for i in range(args.steps):
                step(i if instrumented else None, i & 1)
        g.replay()          # the first replay uploads the graph
        torch.cuda.synchronize()
        return g

    # The timed loop: the K steps captured once in a CUDA graph and replayed
    # between CUDA events, so that the steps run back to back at the device's
    # rate and not at that of the Python code calling the library (tens of
    # microseconds per call).  Per-kernel times: a second graph of the same
    # steps with event-record nodes between the phases, replayed right before
    # the timed replay (the same power and clock history).  Each event node
    # costs a few microseconds, so a step of one kernel (the quantizer alone,
    # the fused linear) takes the timed loop's own step time.
    # The clock samples kept are those of the loaded interval: the warm-up
    # replays, the instrumented one and the timed one, back to back.
    with _Nvtx("rfq graph capture"):
        graph = capture(False)
        graph_ev = capture(True)
    t_start, t_end = ev(), ev()
    with ClockSampler(local) as clk:
        barrier()
        torch.cuda.synchronize()
        h0 = time.time()
        with _Nvtx("rfq warm-up replays + instrumented replay"):
            for _ in range(args.warmup):
                graph.replay()
            graph_ev.replay()
        with _Nvtx("rfq timed replay"):
            t_start.record(stream)
            graph.replay()
            t_end.record(stream)
            torch.cuda.synchronize()
        h1 = time.time()
        barrier()
        # the dense FP4 tensor rate with MMAs alone (both MMA forms), timed
        # right after the step under the same sampler
        mma_peak = None
        if not args.no_mma_peak and ws == 1 and not (quant_only or hif4 or f8):
            h2 = time.time()
            with _Nvtx("rfq MMA-only FP4 rate"):
                mma_peak = _fp4_mma_peak(rfq, wsp, stream, ev)
            mma_peak["clocks"] = clk.summary(h2, time.time(), "the MMA-only launches")
            if mma_peak["clocks"]:
                mma_peak["flop_per_sm_clock"] = (mma_peak["tflops"] * 1e12 / mma_peak["sms"]
                                                 / (mma_peak["clocks"]["sm_mhz"] * 1e6))
        # where the CTA-pair GEMM's tensor pipe idles: one untimed launch of
        # its measuring build (rfq_linear_profile) on the same operands
        mma_prof = None
        if (ws == 1 and not (quant_only or hif4 or f8 or fused or grouped or amax_phi or no_res) and M > 128):
            with _Nvtx("rfq GEMM measuring build"):
                mma_prof = _mma_profile(rfq, bufs[0], wop, K)
    ms = t_start.elapsed_time(t_end) / args.steps
    q_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in per_step)
    g_ms = statistics.mean(e[2].elapsed_time(e[3]) for e in per_step)
    if quant_only:
        q_ms = ms
    elif fused:
        g_ms = ms
    del graph, graph_ev
    ms = _max_over_ranks(ms, ws, dist, dev)

    # End to end through the public API with host buffers: every step copies
    # its X from pinned host memory and its result back to pinned host
    # memory.  The copies run on their own streams against double-buffered
    # device X / Y, so step i's device work overlaps the copies of steps
    # i - 1 and i + 1 (the copy engines give ~200 GB/s per direction).
    e2e_ms = None
    # the two-kernel MXFP4 linear has a C entry point that takes the host
    # buffers itself (rfq_linear_host: row chunks, copies on its own
    # streams); the other variants run the loop below
    host_api = not (quant_only or hif4 or fused or grouped or f8)
    e2e_api = None
    if not args.no_e2e and host_api:
        _nv = _Nvtx("rfq end-to-end loop (rfq_linear_host)")
        _nv.__enter__()
        bs = bufs[0]
        mode = rfq.RFQ_FALLBACK_AMAX if amax_phi else (rfq.RFQ_FALLBACK_NONE if no_res else rfq.RFQ_FALLBACK_ALL)
        tau = args.phi_tau if amax_phi else 0.0
        yh = y_host[:, :N] if y_host.shape[1] != N else y_host
        total = args.warmup + args.steps
        for i in range(total):
            if i == args.warmup:
                barrier()
                torch.cuda.synchronize()
                e0, e1 = ev(), ev()
                e0.record(stream)
            rfq.rfq_linear_host(x_host, wop, yh, rfq.RFQ_OUT_BF16, bs["x"], bs["xq"], bs["xr"], bs["phi"],
                                bs["y"], wsp, mode=mode, tau=tau, chunk_rows=args.e2e_chunk_rows, stream=stream)
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        e2e_ms = e0.elapsed_time(e1) / args.steps
        e2e_api = f"rfq_linear_host (C ABI, pinned host X and Y, {args.e2e_chunk_rows}-row chunks)"
        _nv.__exit__()
    if not args.no_e2e and not host_api:
        _nv = _Nvtx("rfq end-to-end loop (host buffers)")
        _nv.__enter__()
        h2d, d2h = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        x_ready = [torch.cuda.Event(), torch.cuda.Event()]
        x_free = [torch.cuda.Event(), torch.cuda.Event()]
        y_done = [torch.cuda.Event(), torch.cuda.Event()]
        y_free = [torch.cuda.Event(), torch.cuda.Event()]
        total = args.warmup + args.steps
        for i in range(total):
            sl = i & 1
            if i == args.warmup:
                for st_ in (h2d, d2h):
                    stream.wait_stream(st_)
                barrier()
                torch.cuda.synchronize()
                e0, e1 = ev(), ev()
                e0.record(stream)
                h2d.wait_stream(stream)
                d2h.wait_stream(stream)
            with torch.cuda.stream(h2d):
                if i >= 2:
                    h2d.wait_event(x_free[sl])          # step i - 2 has read this X buffer
                bufs[sl]["x"].copy_(x_host, non_blocking=True)
                x_ready[sl].record(h2d)
            stream.wait_event(x_ready[sl])
            if i >= 2:
                stream.wait_event(y_free[sl])           # step i - 2's result has left this buffer set
            step(None, sl)
            x_free[sl].record(stream)
            y_done[sl].record(stream)
            with torch.cuda.stream(d2h):
                d2h.wait_event(y_done[sl])
                if quant_only:
                    for dst, src in zip(host_q, q_out(bufs[sl])):
                        dst.copy_(src, non_blocking=True)
                else:
                    y_host.copy_(bufs[sl]["y"], non_blocking=True)
                y_free[sl].record(d2h)
        stream.wait_stream(h2d)
        stream.wait_stream(d2h)
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        e2e_ms = e0.elapsed_time(e1) / args.steps
        _nv.__exit__()
    if e2e_ms is not None:
        e2e_ms = _max_over_ranks(e2e_ms, ws, dist, dev)
    if rfq.rfq_workspace_status(wsp) != rfq.RFQ_OK:
        raise RuntimeError("rfq_linear reported a device timeout")

    # executed MMA work: the main product, and the residual product on the phi = 1 tiles
    phi_frac = float(bufs[0]["phi"].float().mean().item()) if amax_phi else (0.0 if no_res else 1.0)
    flop = 2.0 * M * N * K * (1.0 + phi_frac)
    pk = _peaks()
    # The timed loop is short (tens of ms at full clocks), so the kernels are
    # held against the burst figure; the sustained one is reported beside it.
    if hif4:
        # HiF4 runs on the bf16 tensor path (exact bf16 expansion)
        t_peak, t_peak_sust = pk["bf16_burst"], pk["bf16_sust"]
        t_src = f"{pk['src']} bf16 burst {pk['bf16_burst']} TFLOP/s, of {pk['src']}"
        t_kernel = "gemm_hif4_kernel"
    elif mixed:
        # main product at the FP4 rate (6x bf16, nominal), residual at the FP8
        # one (2x): the rate the executed FLOP mix allows
        rate = (1.0 + phi_frac) / (1.0 / FP4_OVER_BF16 + phi_frac / 2.0)
        t_peak, t_peak_sust = pk["bf16_burst"] * rate, pk["bf16_sust"] * rate
        t_src = (f"{pk['src']} bf16 burst {pk['bf16_burst']} TFLOP/s x {rate:.3g} (the main product at the nominal "
                 f"FP4/BF16 ratio {FP4_OVER_BF16:g}, the residual at the FP8 one 2, weighted by their FLOP), "
                 f"of {pk['src']}")
        t_kernel = "gemm_mxf4_pair_kernel"   # its mixed-rate instantiation, at every M
    elif f8:
        # kind::mxf8f6f4: the FP8 tensor rate, nominally twice the bf16 one
        t_peak, t_peak_sust = pk["bf16_burst"] * 2.0, pk["bf16_sust"] * 2.0
        t_src = (f"{pk['src']} bf16 burst {pk['bf16_burst']} TFLOP/s x 2 (nominal dense FP8/BF16 ratio), "
                 f"of {pk['src']}")
        t_kernel = "gemm_mxf4_pair_kernel"   # its E4M3 instantiation, at every M
    else:
        t_peak, t_peak_sust = pk["bf16_burst"] * FP4_OVER_BF16, pk["bf16_sust"] * FP4_OVER_BF16
        t_src = (f"{pk['src']} bf16 burst {pk['bf16_burst']} TFLOP/s x {FP4_OVER_BF16:g} "
                 f"(nominal dense FP4/BF16 ratio), of {pk['src']}")
        # CTA pairs beyond one 128-row tile; grouped launches whose groups
        # average under 2048 stacked rows run 128-row tiles on single CTAs
        grouped_single = grouped and Mb < 2048 * spec.groups
        # (fused: CTA pairs with the quantizer in their epilogue warps beyond 128 rows)
        t_kernel = ("gemm_mxf4_pair_kernel" if M > 128 else "gemm_mxf4_fused_kernel") if fused else (
            "gemm_mxf4_kernel" if M <= 128 or grouped_single else "gemm_mxf4_pair_kernel")
    if hif4:
        aq_bytes = _act_quant_bytes(Mb, K, "hif4", not no_res, operand=not quant_only)
        aq_kernel = "act_quant_hif4_amax_kernel" if amax_fused else "act_quant_hif4_kernel"
    elif f8:
        aq_bytes = _act_quant_bytes(Mb, K, "rfq8" if scheme in ("rfq8", "rfq8mix") else "mxfp8",
                                    scheme in ("rfq8", "rfq8mix"), operand=scheme == "rfq8")
        aq_kernel = ("act_quant_rfq8_amax_kernel" if amax_fused else
                     "act_quant_rfq8_kernel" if scheme == "rfq8mix" else "act_quant8_kernel")
    else:
        aq_bytes = _act_quant_bytes(Mb, K, "mxfp4", not no_res)
        # AMAX phi on 128 x 256 tiles: phi and the quantization in one kernel
        aq_kernel = "act_quant_mxfp4_amax_kernel" if amax_fused else "act_quant_mxfp4_kernel"
    if fused:
        act_quant = None   # quantization happens inside the GEMM
    else:
        aq_gbs = aq_bytes / (q_ms * 1e-3) / 1e9
        act_quant = {"bound": "hbm", "kernel": aq_kernel, "achieved": aq_gbs, "peak": pk["hbm"], "unit": "GB/s",
                     "frac": aq_gbs / pk["hbm"], "bytes_per_launch": aq_bytes, "ms_per_launch": q_ms,
                     "traffic": _kernel_traffic(aq_kernel, spec.name + ("+" + scheme if f8 else "")
                                                + ("+w4a4" if no_res and not f8 else ""))}
    if quant_only:
        value = _job_rate(aq_bytes, ws, ms) / 1e9
        unit = "GB/s"
        roofline = dict(act_quant)
    else:
        value = _job_rate(flop, ws, ms) / 1e12
        unit = UNIT
        gemm_tflops = flop / (g_ms * 1e-3) / 1e12
        roofline = {"bound": "tensor", "kernel": t_kernel, "achieved": gemm_tflops, "peak": t_peak,
                    "unit": "TFLOP/s", "frac": gemm_tflops / t_peak,
                    "traffic": _kernel_traffic(t_kernel, spec.name + ("+fused" if fused else "")
                                               + ("+" + scheme if f8 else "")
                                               + ("+phi" if amax_phi else "")
                                               + ("+w4a4" if no_res and not f8 else "")),
                    "flop_per_launch": flop, "ms_per_launch": g_ms,
                    "peak_source": t_src, "frac_of_sustained_peak": gemm_tflops / t_peak_sust}
        if mma_peak is not None and not (hif4 or f8):
            # against this GPU's measured MMA-only FP4 rate (the nominal 6x ratio is not reached)
            roofline["measured_fp4_mma_tflops"] = mma_peak["tflops"]
            roofline["frac_of_measured_fp4_mma"] = gemm_tflops / mma_peak["tflops"]
        if mma_prof is not None:
            roofline["mma_thread_profile"] = mma_prof
    clocks = clk.summary(h0, h1)
    if e2e_ms is not None:
        e2e = {"value": _job_rate(aq_bytes / 1e9 if quant_only else flop / 1e12, ws, e2e_ms), "unit": unit,
               "ms_per_step": e2e_ms, "api": e2e_api or ("rfq entry points on device buffers, host copies on "
                                                         "copy streams (double-buffered across steps)"),
               "h2d_bytes_per_step": Mb * K * 2,
               "d2h_bytes_per_step": q_bytes if quant_only else Mb * N * 2}
    else:
        e2e = None

    if rank == 0:
        cpu = None
        if ws == 1 and not args.no_cpu_baseline and not args.rows:
            n, u, sample, reps = cpu_oracle_timed(args.workload, 8, 4, 1)
            v, dt = reps[0]
            cpu = {"value": v, "unit": u, "cores": n, "kind": "oracle", "sample": sample,
                   "seconds": round(dt, 2)}
        line = {
            "metric": METRIC, "value": value, "unit": unit, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None,
            "dtype": ("hif4 (exact bf16 x bf16, fp32 accumulate)" if hif4 else
                      "mxfp8 (e4m3 x e4m3, fp32 accumulate)" if f8 else "mxfp4 (e2m1 x e2m1, fp32 accumulate)"),
            "data": "synthetic",
            "config": _config(spec, {"parallelism": f"dp{ws} over token rows" if ws > 1 else "single GPU",
                                     "timing": "the K timed steps captured in one CUDA graph, replayed once "
                                               "between CUDA events (per-kernel times: a second graph with events between the kernels)",
                                     "variant": ("fused prologue: X quantized inside the GEMM" if fused
                                                 else "quantizer kernel + GEMM kernel"),
                                     **({"groups": f"{spec.groups} experts, routed rows {M} (min "
                                                   f"{int(counts.min())}, max {int(counts.max())} per expert), "
                                                   f"stacked on 128-row starts: {Mb} rows",
                                         "weight_rows": NW} if grouped else {}),
                                     **({"residual": "none: plain W4A4 (Q(X) W~ only)"}
                                        if no_res and not f8 else {}),
                                     **({"scheme": {"rfq8mix": "RFQ with an MXFP8 residual: MXFP4 X~ x MXFP4 W~ "
                                                               "on the FP4 path + MXFP8 X^ x W~ as E4M3 on "
                                                               "the FP8 path, one accumulator",
                                                    "rfq8": "RFQ with an MXFP8 residual: MXFP4 X~ + MXFP8 X^, "
                                                            "MXFP4 W~, all multiplied as E4M3",
                                                    "w4a8": "W4A8: MXFP8 X x MXFP4 W~ (as E4M3)",
                                                    "w8a8": "W8A8: MXFP8 X x MXFP8 W~"}[scheme]} if f8 else {}),
                                     **({"phi": f"AMAX: phi = [max |x| over the 128 x 256 tile > {args.phi_tau}], "
                                                f"fraction of phi = 1 tiles f = {phi_frac:.4f}",
                                         "phi_fraction": phi_frac} if amax_phi else {})}),
            "roofline": roofline,
            "act_quant": act_quant,
            "e2e": e2e,
            "gpu_launches": _launches_per_step(quant_only, fused, hif4, no_res, scheme, amax_phi,
                                                amax_fused) * args.steps,
            "clocks": clocks,
            "cpu_baseline": cpu,
        }
        if not quant_only:
            line["effective_tflops_2mnk"] = _job_rate(flop / 2, ws, ms) / 1e12
        if mma_peak is not None:
            line["fp4_mma_peak"] = mma_peak
        if ws == 1 and not args.no_extras and not args.rows:
            line["other_configs"] = _other_configs(args)
        print(json.dumps(line), flush=True)
    if ws > 1:
        dist.destroy_process_group()


def _mma_profile(rfq, bs, wop, K):
    """One launch of the CTA-pair GEMM's measuring build; per CTA pair, its
    MMA thread's effective SM clock and the shares of its time spent waiting
    for a drained accumulator, for operand copies and for scale words, and
    the tensor pipe's busy share (stages x MMA cycles per stage, at the
    32 768 FLOP per SM clock the MMA-only loop measures)."""
    import torch
    wsp = torch.zeros(rfq.rfq_linear_workspace_bytes() // 4, dtype=torch.int32, device=bs["x"].device)
    c = rfq.rfq_linear_profile(bs["xq"], bs["xr"], wop, bs["y"], rfq.RFQ_OUT_BF16, wsp)
    if rfq.rfq_workspace_status(wsp) != rfq.RFQ_OK or c["cycles"] <= 0:
        return None
    mma_cycles = 4.0 * K * c["tiles"]          # main + residual 256x256xK per pair, 2 SMs at 32 768 FLOP/clock
    return {"sm_mhz_effective": c["cycles"] / c["ns"] * 1e3, "tensor_busy": mma_cycles / c["cycles"],
            "wait_accumulator": c["wait_acc_cycles"] / c["cycles"],
            "wait_copies": c["wait_copies_cycles"] / c["cycles"],
            "wait_scales": c["wait_scales_cycles"] / c["cycles"],
            "pairs": c["pairs"], "tiles": c["tiles"], "stages": c["stages"],
            "how": "rfq_linear_profile: clock64 / globaltimer in each pair's MMA thread, one untimed launch"}


def _fp4_mma_peak(rfq, wsp, stream, ev, iters: int = 16384, reps: int = 5):
    """MMA-only FP4 rate (rfq_fp4_mma_peak): per form, 3 untimed launches,
    then `reps` launches each timed with CUDA events on the launching stream;
    TFLOP/s of the mean launch.  `tflops` is the faster form's, and
    flop_per_sm_clock divides it by the SM count and the median SM clock the
    sampler saw (filled in by the caller's clock summary when available)."""
    import torch
    out = {"iters_per_launch": iters, "launches": reps}
    best = 0.0
    for name, pair in (("cta1", False), ("cta_pair", True)):
        for _ in range(3):
            rfq.rfq_fp4_mma_peak(pair, iters, wsp)
        ms = []
        for _ in range(reps):
            a, b = ev(), ev()
            a.record(stream)
            flop = rfq.rfq_fp4_mma_peak(pair, iters, wsp)
            b.record(stream)
            b.synchronize()
            ms.append(a.elapsed_time(b))
        t = flop / (statistics.mean(ms) * 1e-3) / 1e12
        out[f"tflops_{name}"] = t
        out[f"ms_per_launch_{name}"] = statistics.mean(ms)
        best = max(best, t)
    if rfq.rfq_workspace_status(wsp) != rfq.RFQ_OK:
        raise RuntimeError("rfq_fp4_mma_peak reported a device timeout")
    out["tflops"] = best
    out["sms"] = torch.cuda.get_device_properties(0).multi_processor_count
    return out


# The other workloads of the benchmark's configuration list, each timed by a
# child run of this script (its own process, inputs, CUDA graph and clock
# samples) after the headline one: the standalone activation quantizer
# (16384 x 4096, Student-t), the Qwen3-VL-8B gate/up and HiF4 down
# projections, and the Wan2.2 FFN up projection on the fused-prologue variant.
_EXTRAS = (("act_quant_16384x4096", ["--workload", "act_quant"]),
           ("qwen3vl8b_gate_up", ["--workload", "qwen_gate_up"]),
           ("qwen3vl8b_down_hif4", ["--workload", "qwen_down_hif4"]),
           ("wan22_ffn_up_fused", ["--workload", "wan_ffn_up", "--variant", "fused"]))


def _other_configs(args):
    out = {}
    for name, extra in _EXTRAS:
        cmd = [sys.executable, os.path.abspath(__file__), "--steps", str(args.steps), "--warmup", str(args.warmup),
               "--no-cpu-baseline", "--no-e2e", "--no-extras", "--no-mma-peak", *extra]
        try:
            r = subprocess.run(cmd, capture_output=True, text=True, timeout=600)
            line = json.loads([ln for ln in r.stdout.splitlines() if ln.startswith("{")][-1])
        except (subprocess.TimeoutExpired, IndexError, ValueError) as e:
            out[name] = {"error": f"{type(e).__name__}: {str(e)[:200]}"}
            continue
        rl = line.get("roofline") or {}
        out[name] = {"value": line["value"], "unit": line["unit"], "ms_per_step": line["ms_per_step"],
                     "kernel": rl.get("kernel"), "kernel_ms_per_launch": rl.get("ms_per_launch"),
                     "kernel_frac": rl.get("frac"), "peak": rl.get("peak"), "peak_unit": rl.get("unit"),
                     "act_quant_frac": (line.get("act_quant") or {}).get("frac"),
                     "variant": line["config"].get("variant"), "workload": line["config"]["workload"],
                     "clocks": line.get("clocks")}
    return out


# the configuration list's entries, in order
_CONFIGS = {1: "tiny", 2: "act_quant", 3: "qwen_gate_up", 4: "qwen_down_hif4", 5: "wan_ffn_up"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="rfq", choices=["rfq", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end (host buffer) timing")
    ap.add_argument("--e2e-chunk-rows", type=int, default=2048,
                    help="row chunk of rfq_linear_host in the end-to-end timing (a multiple of 128)")
    ap.add_argument("--rows", type=int, default=0, help="profile a smaller case: the first ROWS token rows")
    ap.add_argument("--phi-tau", type=float, default=None,
                    help="selective fallback: residual only on 128 x 256 tiles whose max |x| exceeds TAU")
    ap.add_argument("--no-residual", action="store_true",
                    help="plain W4A4: no residual pathway (the baseline the correction is added to)")
    ap.add_argument("--scheme", default="rfq4", choices=["rfq4", "rfq8", "rfq8mix", "w4a8", "w8a8"],
                    help="rfq4: MXFP4 main + MXFP4 residual (default); rfq8: MXFP8 residual; "
                         "w4a8 / w8a8: MXFP8 activation baselines")
    ap.add_argument("--variant", default="two-kernel", choices=["two-kernel", "fused"],
                    help="fused: rfq_linear_fused, the activation quantizer inside the GEMM")
    ap.add_argument("--workload", default=WORKLOAD,
                    choices=["wan_ffn_up", "qwen_gate_up", "qwen_down_hif4", "act_quant", "tiny", "qwen_moe_gate_up"])
    ap.add_argument("--config", type=int, default=0, choices=[0, 1, 2, 3, 4, 5],
                    help="the configuration list's entry (1 tiny, 2 act-quant, 3 Qwen3-VL gate/up, 4 Qwen3-VL "
                         "HiF4 down, 5 Wan2.2 FFN up); overrides --workload")
    ap.add_argument("--seed", type=int, default=None, help="replace the workload's input seed")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the child runs that time the other workloads of the configuration list")
    ap.add_argument("--no-mma-peak", action="store_true",
                    help="skip the MMA-only FP4 rate measurement")
    args = ap.parse_args()
    if args.config:
        args.workload = _CONFIGS[args.config]
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_rfq(args)


if __name__ == "__main__":
    main()
