"""Builds ``librfq.so`` in-tree from ``csrc/*.cu`` for sm_103a with nvcc.

Each translation unit compiles in parallel; the objects link into one shared
library with the CUDA runtime linked statically.  No fast-math and no
flush-to-zero: the quantizers rely on IEEE fp32 with subnormals.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import platform
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(os.path.dirname(HERE), "_build", platform.machine())
LIB = os.path.join(HERE, "librfq.so")
# the debug build: device-side bounds checks on the kernels' direct stores
BUILD_DEBUG = os.path.join(os.path.dirname(HERE), "_build", platform.machine() + "-debug")
LIB_DEBUG = os.path.join(HERE, "librfq_debug.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
         "--expt-relaxed-constexpr"]


def _nvcc():
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", shutil.which("nvcc")):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _stale(obj, src):
    if not os.path.exists(obj):
        return True
    t = os.path.getmtime(obj)
    deps = [src] + glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(CSRC, "*.h")) + [
        os.path.join(os.path.dirname(HERE), "include", "rfq.h")]
    return any(os.path.getmtime(d) > t for d in deps)


def build(verbose: bool = False, ptxas_v: bool = False, force: bool = False, debug: bool = False) -> str:
    """Builds librfq.so, or with debug=True librfq_debug.so (-DRFQ_DEBUG_BOUNDS,
    its own object directory); returns the library's path."""
    nvcc = _nvcc()
    build_dir, lib = (BUILD_DEBUG, LIB_DEBUG) if debug else (BUILD, LIB)
    os.makedirs(build_dir, exist_ok=True)
    srcs = sorted(glob.glob(os.path.join(CSRC, "*.cu")))
    objs = [os.path.join(build_dir, os.path.basename(s)[:-3] + ".o") for s in srcs]

    def compile_one(so):
        src, obj = so
        if not force and not _stale(obj, src):
            return ""
        cmd = [nvcc, *ARCH, *FLAGS, *(["-DRFQ_DEBUG_BOUNDS"] if debug else []), "-c", src, "-o", obj]
        if ptxas_v:
            cmd.insert(1, "-Xptxas=-v")
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        return r.stdout + r.stderr

    with cf.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 4)) as ex:
        outs = list(ex.map(compile_one, zip(srcs, objs)))
    if verbose:
        for o in outs:
            if o:
                print(o, file=sys.stderr)
    if force or not os.path.exists(lib) or any(os.path.getmtime(o) > os.path.getmtime(lib) for o in objs):
        tmp = lib + f".{os.getpid()}.tmp"
        r = subprocess.run([nvcc, *ARCH, "-shared", "-o", tmp, *objs], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(verbose=True, ptxas_v="-v" in sys.argv, force="-f" in sys.argv))
