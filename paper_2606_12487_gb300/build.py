"""Build libdptq.so (the CUDA library behind include/dptq.h) for sm_103a.

Translation units are compiled in parallel with nvcc and linked into one shared
library under ``paper_2606_12487_gb300/_build``.  Run ``python -m
paper_2606_12487_gb300.build`` or call :func:`build`.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "libdptq.so")
# DPTQ_TRACE=1 builds a separate library whose kernels record %globaltimer stamps;
# DPTQ_DEBUG=1 one whose kernels check the index arithmetic of their global accesses
# (DPTQ_CHECK in csrc/dptq_device.cuh).
TRACE = os.environ.get("DPTQ_TRACE") == "1"
DEBUG = os.environ.get("DPTQ_DEBUG") == "1"
if TRACE and DEBUG:
    raise RuntimeError("DPTQ_TRACE and DPTQ_DEBUG select different libraries: set one")
if TRACE:
    OUT_DIR = os.path.join(HERE, "_build_trace")
    LIB = os.path.join(OUT_DIR, "libdptq.so")
if DEBUG:
    OUT_DIR = os.path.join(HERE, "_build_debug")
    LIB = os.path.join(OUT_DIR, "libdptq.so")
SOURCES = ["api.cu", "rotate_quant.cu", "qgemm.cu", "static_scratch.cu", "kv_policy.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libdptq")


def _flags():
    return ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", os.path.join(ROOT, "include"),
                   *(["-DDPTQ_TRACE"] if TRACE else []),
                   *(["-DDPTQ_DEBUG"] if DEBUG else []),
                   *([f"-DDPTQ_TRACE_STAGES={int(os.environ['DPTQ_TRACE_STAGES'])}"]
                     if TRACE and os.environ.get("DPTQ_TRACE_STAGES") else []),
                   *(["-DDPTQ_TRACE_CLOCKS"] if TRACE and os.environ.get("DPTQ_TRACE_CLOCKS") == "1" else []),
                   "--ptxas-options=-v" if os.environ.get("DPTQ_PTXAS_V") else "-Xptxas=-O3"]


def _stale(lib: str, deps) -> bool:
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False) -> str:
    os.makedirs(OUT_DIR, exist_ok=True)
    headers = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    headers.append(os.path.join(ROOT, "include", "dptq.h"))
    srcs = [os.path.join(CSRC, s) for s in SOURCES]
    if not force and not _stale(LIB, srcs + headers + [__file__]):
        return LIB
    cc = nvcc()
    objs = []

    def compile_one(src):
        obj = os.path.join(OUT_DIR, os.path.basename(src) + ".o")
        cmd = [cc, *_flags(), "-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            print(r.stdout + r.stderr, file=sys.stderr)
        return obj

    with cf.ThreadPoolExecutor(max_workers=len(srcs)) as ex:
        objs = list(ex.map(compile_one, srcs))
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [cc, *ARCH, "-shared", "-o", tmp, *objs, "-lcudart_static", "-lrt", "-lpthread", "-ldl"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
