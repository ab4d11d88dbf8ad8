"""Builds libboute.so (all CUDA translation units, sm_103a only) in-tree.

nvcc compiles each .cu file to an object in parallel, then links one shared
library with the CUDA runtime linked statically. The output lives in
``_build/`` next to this file and is git-ignored.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
OUT = os.path.join(HERE, "_build")
LIB = os.path.join(OUT, "libboute.so")
# the debug build: every kernel's bounds checks compiled in (bounds.cuh)
OUT_DEBUG = os.path.join(HERE, "_build", "debug")
LIB_DEBUG = os.path.join(OUT_DEBUG, "libboute_debug.so")
NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2", "--expt-relaxed-constexpr",
         "-I", os.path.join(ROOT, "include")]


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return _sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(
        os.path.join(CSRC, "*.h")) + [os.path.join(ROOT, "include", "boute.h")]


def build(force: bool = False, verbose: bool = False, extra: list | None = None,
          debug: bool = False) -> str:
    """debug: the bounds-checked library (BOUTE_DEBUG_BOUNDS) in its own
    directory; the product library is unaffected."""
    lib, out = (LIB_DEBUG, OUT_DEBUG) if debug else (LIB, OUT)
    if not force and os.path.exists(lib) and os.path.getmtime(lib) >= max(
            os.path.getmtime(p) for p in _deps()):
        return lib
    os.makedirs(out, exist_ok=True)
    extra = (extra or []) + (["-DBOUTE_DEBUG_BOUNDS"] if debug else [])

    def compile_one(src):
        obj = os.path.join(out, os.path.basename(src) + ".o")
        cmd = [NVCC, *ARCH, *FLAGS, *extra, "-c", src, "-o", obj]
        if verbose:
            print(" ".join(cmd), flush=True)
        subprocess.run(cmd, check=True)
        return obj

    with cf.ThreadPoolExecutor(max(1, min(8, os.cpu_count() or 1))) as ex:
        objs = list(ex.map(compile_one, _sources()))
    tmp = lib + f".{os.getpid()}.tmp"
    subprocess.run([NVCC, *ARCH, "-shared", "-Xcompiler", "-fPIC", *objs, "-o", tmp], check=True)
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(force=True, verbose=True))
