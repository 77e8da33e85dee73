"""Build libchameleon.so in-tree with nvcc for sm_103a.

Each CUDA translation unit is compiled to an object in parallel, then linked into one shared
library next to this file.  Usage: ``python -m paper_2609_33496_gb300.build [--force]``.
"""
import concurrent.futures
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libchameleon.so")
PROBE_LIB = os.path.join(HERE, "libchameleon_probe.so")   # tensor-core throughput probe (bench only)
SOURCES = ["act_quant.cu", "weights.cu", "gemm.cu", "gemm_f16.cu", "gemm_bf16.cu", "gemm_f8.cu", "gemm_f8_mx.cu",
           "gemm_small.cu", "api.cu", "noalloc.cu"]
# translation units whose quantizer arithmetic must not be contracted into FMAs
NO_FMAD = {"act_quant.cu", "weights.cu"}
HEADERS = ["common.cuh", "act_quant.cuh", "weights.cuh", "gemm.cuh", "gemm_kernel.cuh", "gemm_f8_kernel.cuh"]
PROBE_SOURCES = ["probe.cu"]

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
         "--expt-relaxed-constexpr"]


def nvcc():
    path = shutil.which("nvcc")
    if path is None:
        cand = "/usr/local/cuda/bin/nvcc"
        if os.path.exists(cand):
            return cand
        raise RuntimeError("nvcc not found")
    return path


def _inputs():
    files = [os.path.join(CSRC, s) for s in SOURCES + HEADERS]
    files.append(os.path.join(os.path.dirname(HERE), "include", "chameleon.h"))
    files.append(os.path.abspath(__file__))
    return files


def up_to_date():
    for lib in (LIB, PROBE_LIB):
        if not os.path.exists(lib):
            return False
    t = min(os.path.getmtime(LIB), os.path.getmtime(PROBE_LIB))
    return all(os.path.getmtime(f) <= t for f in _inputs() + [os.path.join(CSRC, s) for s in PROBE_SOURCES])


def _compile(src):
    obj = os.path.join(BUILD, src.replace(".cu", ".o"))
    cmd = [nvcc()] + ARCH + FLAGS + (["-fmad=false"] if src in NO_FMAD else []) + [
        "-c", os.path.join(CSRC, src), "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("nvcc failed for %s:\n%s%s" % (src, r.stdout, r.stderr))
    return obj


def build(force=False, verbose=False):
    """Compile the library if any input is newer than it; returns its path."""
    if not force and up_to_date():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    with concurrent.futures.ThreadPoolExecutor(max_workers=len(SOURCES) + len(PROBE_SOURCES)) as ex:
        objs = list(ex.map(_compile, SOURCES + PROBE_SOURCES))
    for lib, lib_objs in ((LIB, objs[:len(SOURCES)]), (PROBE_LIB, objs[len(SOURCES):])):
        tmp = lib + ".tmp"
        cmd = [nvcc()] + ARCH + ["-shared", "-cudart", "shared", "-o", tmp] + lib_objs
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("link failed:\n%s%s" % (r.stdout, r.stderr))
        os.replace(tmp, lib)
    if verbose:
        print("built", LIB)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose=True)
