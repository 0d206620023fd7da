"""Build the CUDA library (libevo.so) in-tree for sm_103a.

Each .cu file is compiled in parallel with nvcc, then linked into one shared
library next to this file.  No CMake, no torch extension machinery: the
library exports only the C ABI of include/evo.h.  build(debug=True) makes
libevo_debug.so, the same library with device-side index checks
(EVO_DEBUG_CHECKS: a failed check records a status bit and skips the access).
"""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
OUT = os.path.join(HERE, "libevo.so")
OUT_DEBUG = os.path.join(HERE, "libevo_debug.so")
BUILD = os.path.join(ROOT, "_build")
SOURCES = ["evo_api.cu", "evo_job.cu", "evo_loop_s01.cu", "evo_loop_s23.cu", "evo_loop_s45.cu", "evo_loop_f32.cu", "evo_wide.cu", "evo_redundancy.cu", "evo_search.cpp"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2", "-Xcompiler", "-ffp-contract=off",
         "-I", os.path.join(ROOT, "include")]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if cand and (os.path.isabs(cand) and os.path.exists(cand) or not os.path.isabs(cand)):
            return cand
    return "nvcc"


def _stale(target: str, deps: list[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def build(verbose: bool = False, extra: list[str] | None = None, debug: bool = False) -> str:
    build_dir = os.path.join(BUILD, "debug") if debug else BUILD
    out = OUT_DEBUG if debug else OUT
    extra = list(extra or []) + (["-DEVO_DEBUG_CHECKS=1"] if debug else [])
    os.makedirs(build_dir, exist_ok=True)
    nvcc = _nvcc()
    headers = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    headers.append(os.path.join(ROOT, "include", "evo.h"))
    objs = []
    jobs = []
    for src in SOURCES:
        s = os.path.join(CSRC, src)
        o = os.path.join(build_dir, os.path.splitext(src)[0] + ".o")
        objs.append(o)
        if _stale(o, [s] + headers):
            jobs.append([nvcc, *ARCH, *FLAGS, *extra, "-c", s, "-o", o])

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        if verbose or r.returncode != 0:
            sys.stderr.write(r.stdout + r.stderr)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed: {' '.join(cmd)}")

    with ThreadPoolExecutor(max_workers=len(jobs) or 1) as ex:
        list(ex.map(run, jobs))
    if _stale(out, objs):
        run([nvcc, *ARCH, "-shared", "-o", out, *objs, "-lcudart"])
    return out


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv))
