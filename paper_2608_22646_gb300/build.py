"""Build the sm_103a C-ABI library ``libcai.so`` in-tree with nvcc."""
from __future__ import annotations

import os
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIB = os.path.join(PKG, "libcai.so")
LIB_DEBUG = os.path.join(PKG, "libcai_debug.so")  # CAI_DEBUG: range checks on index lists
SOURCES = ["cai.cu"]
DEPS = ["cai.cu", "ptx.cuh", "softmax.cuh", "commit.cuh", "head_kernel.cuh", "step_kernels.cuh", "pair_kernel.cuh",
        "rows_kernel.cuh", "static_head.cuh"]


def _stale(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    deps = [os.path.join(CSRC, d) for d in DEPS] + [os.path.join(INCLUDE, "cai.h")]
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False, debug: bool = False) -> str:
    """Build libcai.so (or, with debug, libcai_debug.so with CAI_DEBUG range checks)."""
    lib = LIB_DEBUG if debug else LIB
    if not force and not _stale(lib):
        return lib
    nvcc = os.environ.get("NVCC", "nvcc")
    tmp = lib + f".tmp{os.getpid()}"
    cmd = [nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-lineinfo", "-std=c++17",
           "-Xcompiler", "-fPIC", "-shared", "-I", INCLUDE, "-o", tmp]
    if debug:
        cmd += ["-DCAI_DEBUG"]
    if verbose:
        cmd += ["-Xptxas", "-v"]
    cmd += [os.path.join(CSRC, s) for s in SOURCES]
    subprocess.check_call(cmd, stdout=None if verbose else subprocess.DEVNULL)
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv, debug="--debug" in sys.argv))
