"""The multi-process path on CPU: world-size-2 process groups over gloo.

bench.py runs one process per GPU; every rank processes its own copy of the
workload (token rows are independent, so the path shards with no data-path
collective), the job's time is the slowest rank's (a MAX all-reduce of the
timings), the job's throughput counts every rank's units, and only rank 0
prints the result line.  These tests drive that host logic with gloo ranks."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, ws, port, out_dir, values):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    try:
        got = bench._max_over_ranks(values[rank], ws, dist, "cpu")
        dist.barrier()
    finally:
        dist.destroy_process_group()
    with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
        f.write(repr(got))


def test_max_over_ranks_two_gloo_ranks(tmp_path):
    values = [3.25, 7.5]
    mp.start_processes(_rank_main, args=(2, _free_port(), str(tmp_path), values), nprocs=2, join=True,
                       start_method="spawn")
    got = [float(open(tmp_path / f"rank{r}.txt").read()) for r in range(2)]
    assert got == [7.5, 7.5]


def test_single_rank_needs_no_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench._max_over_ranks(1.5, 1, None, "cpu") == 1.5


def test_job_rate_counts_every_rank():
    sys.path.insert(0, ROOT)
    import bench
    # 4 ranks x 2e12 units in the slowest rank's 0.5 ms
    assert bench._job_rate(2e12, 4, 0.5) == pytest.approx(1.6e16)
    assert bench._job_rate(2e12, 1, 0.5) == pytest.approx(4e15)


def test_reference_arm_under_torchrun_two_ranks():
    """`bench.py --impl reference` launched the way the driver launches N > 1:
    rank 0 alone runs the oracle and prints one JSON line, rank 1 exits 0."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference",
           "--gpus", "2", "--workload", "tiny", "--steps", "2", "--warmup", "3"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["unit"] == "TFLOP/s" and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
