"""Build libea.so (the C-ABI of include/ea.h) in-tree for sm_103a with nvcc.

The translation units compile in parallel; the result lands in paper_2205_14473_gb300/_lib/.
Usage: python -m paper_2205_14473_gb300.build [--verbose]
"""
from __future__ import annotations

import concurrent.futures as futures
import os
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
LIBDIR = os.path.join(PKG, "_lib")
LIB = os.path.join(LIBDIR, "libea.so")
SOURCES = ["ea_api.cu", "ea_worker.cu", "ea_noalloc.cu", "ea_selftest.cu"] + [f"ea_server_{m}_q{q}.cu" for m in "ws" for q in range(4)]
NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")
# binary32 per operation: no FMA contraction, IEEE division and square root, denormals kept
FLAGS = ["-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-lineinfo", "-std=c++17", "--fmad=false",
         "-prec-div=true", "-prec-sqrt=true", "-ftz=false", "-Xcompiler", "-fPIC,-O2",
         "-I" + os.path.join(ROOT, "include")]


def _stale(obj: str, deps: list[str]) -> bool:
    return not os.path.exists(obj) or any(os.path.getmtime(d) > os.path.getmtime(obj) for d in deps)


def build(verbose: bool = False, force: bool = False) -> str:
    os.makedirs(LIBDIR, exist_ok=True)
    headers = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    headers.append(os.path.join(ROOT, "include", "ea.h"))
    jobs = []
    for src in SOURCES:
        path = os.path.join(CSRC, src)
        obj = os.path.join(LIBDIR, src.replace(".cu", ".o"))
        if force or _stale(obj, [path, *headers]):
            cmd = [NVCC, *FLAGS, *(["-Xptxas", "-v"] if verbose else []), "-c", path, "-o", obj]
            jobs.append(cmd)

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed:\n" + " ".join(cmd) + "\n" + r.stdout + r.stderr)
        return r.stdout + r.stderr

    with futures.ThreadPoolExecutor(max(1, len(jobs))) as ex:
        for out in ex.map(run, jobs):
            if verbose and out:
                print(out)
    objs = [os.path.join(LIBDIR, s.replace(".cu", ".o")) for s in SOURCES]
    if jobs or not os.path.exists(LIB):
        tmp = LIB + f".tmp{os.getpid()}"
        subprocess.run([NVCC, "-shared", "-o", tmp, *objs, "-gencode", "arch=compute_103a,code=sm_103a"], check=True)
        os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(verbose="--verbose" in sys.argv, force="--force" in sys.argv))
