"""Builds the CUDA library ``libdualmv.so`` in-tree with nvcc for sm_103a.

Usage: ``python -m paper_2512_22147_gb300.build`` (or ``build_library()``).
The library is a plain shared object exporting the C ABI of
``include/dualmv.h``; the Python binding loads it with ctypes.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIB_NAME = "libdualmv.so"
LIB_PATH = os.path.join(PKG, LIB_NAME)
SOURCES = [os.path.join(CSRC, "dualmv.cu")]
DEPENDS = SOURCES + [os.path.join(CSRC, n) for n in (
    "dualmv_kernels.cuh", "dualmv_f64e.cuh", "dualmv_tune.cuh", "dualmv_wide.cuh",
    "dualmv_atax.cuh", "dualmv_atax_f64.cuh", "dualmv_ops.cuh", "dualmv_probe.cuh", "dualmv_small.cuh",
    "dualmv_gemver_update.cuh")] + [
    os.path.join(INCLUDE, "dualmv.h")]

NVCC_FLAGS = [
    "-gencode", "arch=compute_103a,code=sm_103a",
    "-lineinfo", "-O3", "-std=c++17",
    "-Xcompiler", "-fPIC", "-shared",
]


def nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA 13 toolkit is required to build")


def stale() -> bool:
    if not os.path.exists(LIB_PATH):
        return True
    built = os.path.getmtime(LIB_PATH)
    return any(os.path.getmtime(p) > built for p in DEPENDS)


def build_library(force: bool = False, verbose: bool = False) -> str:
    """Compile the library if it is missing or older than its sources."""
    if not force and not stale():
        return LIB_PATH
    tmp = LIB_PATH + f".tmp{os.getpid()}"
    cmd = [nvcc(), *NVCC_FLAGS, "-I", INCLUDE, "-I", CSRC, "-o", tmp, *SOURCES]
    if verbose:
        print(" ".join(cmd), file=sys.stderr)
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB_PATH)
    return LIB_PATH


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose=True))
