"""Builds the engine's shared library in-tree for sm_103a (GB300).

    python -m paper_2608_13757_gb300.build [--force]

Each CUDA translation unit is compiled by nvcc with
``-gencode arch=compute_103a,code=sm_103a -lineinfo -O3`` in parallel, the
host loader by g++, and the objects are linked into
``paper_2608_13757_gb300/_lib/libsyncgb.so`` against the shared CUDA runtime.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
LIBDIR = os.path.join(HERE, "_lib")
LIB = os.path.join(LIBDIR, "libsyncgb.so")
CUDA_HOME = os.environ.get("CUDA_HOME", "/usr/local/cuda")
NVCC = os.path.join(CUDA_HOME, "bin", "nvcc")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
CU = ["k_tiles.cu", "k_load.cu", "k_thresholds.cu", "k_simulate.cu", "k_sweep.cu", "k_piece.cu", "k_noalloc.cu"]
CPP = ["capi.cpp"]
HEADERS = [os.path.join(CSRC, "enc.h"), os.path.join(CSRC, "progbuild.cuh"), os.path.join(CSRC, "cost.cuh"), os.path.join(CSRC, "sweep.cuh"), os.path.join(CSRC, "handle.h"), os.path.join(CSRC, "waitval.cuh"), os.path.join(ROOT, "include", "sync.h")]


def _sources():
    return [os.path.join(CSRC, f) for f in CU + CPP]


def _stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(p) > t for p in _sources() + HEADERS + [__file__])


def _compile(src: str) -> str:
    obj = os.path.join(LIBDIR, os.path.basename(src) + ".o")
    inc = ["-I", os.path.join(ROOT, "include"), "-I", CSRC]
    if src.endswith(".cu"):
        cmd = [NVCC] + ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
                               "-Xptxas", "-warn-spills", "-c", src, "-o", obj] + inc
    else:
        cmd = ["g++", "-O2", "-std=c++17", "-fPIC", "-pthread", "-Wall", "-Wextra", "-c", src, "-o", obj,
               "-I", os.path.join(CUDA_HOME, "include")] + inc
    subprocess.check_call(cmd)
    return obj


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile every CUDA/C++ source and link libsyncgb.so (skipped if fresh)."""
    if not force and not _stale():
        return LIB
    if not os.path.exists(NVCC):
        raise RuntimeError(f"nvcc not found at {NVCC}")
    os.makedirs(LIBDIR, exist_ok=True)
    with ThreadPoolExecutor(max_workers=len(CU) + len(CPP)) as ex:
        objs = list(ex.map(_compile, _sources()))
    tmp = LIB + f".tmp{os.getpid()}"
    subprocess.check_call([NVCC] + ARCH + ["-shared", "-cudart", "shared", "-o", tmp] + objs +
                          ["-Xlinker", "-rpath=" + os.path.join(CUDA_HOME, "lib64"), "-Xcompiler", "-pthread"])
    os.replace(tmp, LIB)
    if verbose:
        print("built", LIB)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose=True)
