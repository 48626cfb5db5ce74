"""Builds libsadmm.so in-tree from csrc/ with nvcc for sm_103a.

Each translation unit compiles in parallel; the objects link into one shared
library with the CUDA runtime linked statically, so the library loads
alongside any other CUDA user in the process.  No cmake, no torch extension
machinery: the C ABI in include/sadmm.h is the only interface.

The debug library (_build/debug/libsadmm.so, -DSADMM_DEBUG) adds index checks
to the kernels' global loads and stores: an index outside its buffer skips the
access and raises SADMM_EBOUNDS through sadmm_last_device_status.  The
binding loads it when the environment sets SADMM_DEBUG=1.
"""
from __future__ import annotations

import concurrent.futures
import os
import shutil
import subprocess
import sys
from typing import List

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(BUILD, "libsadmm.so")
DEBUG_LIB = os.path.join(BUILD, "debug", "libsadmm.so")

SOURCES = ["abi.cu", "project.cu", "pack.cu", "conv_fwd.cu", "conv_slab.cu", "admm.cu", "elements.cu", "gemm.cu",
           "bwd.cu", "bwd_slab.cu", "sparse.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    cand = os.environ.get("NVCC") or shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found: the CUDA library cannot be built")
    return cand


def common_flags(extra: List[str]) -> List[str]:
    return ARCH + ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC,-O2",
                   "-I", INCLUDE, "-I", CSRC] + extra


def _inputs() -> List[str]:
    deps = [os.path.join(CSRC, s) for s in SOURCES]
    for fn in os.listdir(CSRC):
        if fn.endswith((".cuh", ".h")):
            deps.append(os.path.join(CSRC, fn))
    deps.append(os.path.join(INCLUDE, "sadmm.h"))
    return deps


def debug_requested() -> bool:
    return os.environ.get("SADMM_DEBUG", "") not in ("", "0")


def up_to_date(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(p) <= t for p in _inputs())


def build(force: bool = False, verbose: bool = False, extra: List[str] | None = None,
          debug: bool | None = None) -> str:
    """Compile csrc/*.cu and link _build/libsadmm.so (with debug, or SADMM_DEBUG=1
    in the environment: _build/debug/libsadmm.so with -DSADMM_DEBUG).  Returns
    the library path."""
    if debug is None:
        debug = debug_requested()
    lib = DEBUG_LIB if debug else LIB
    if not force and not extra and up_to_date(lib):
        return lib
    out = os.path.dirname(lib)
    os.makedirs(out, exist_ok=True)
    flags = common_flags(list(extra or []) + (["-DSADMM_DEBUG"] if debug else []))
    exe = nvcc()

    def compile_one(src: str) -> str:
        obj = os.path.join(out, os.path.splitext(src)[0] + ".o")
        cmd = [exe] + flags + ["-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            sys.stderr.write(r.stdout + r.stderr)
        return obj

    with concurrent.futures.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(compile_one, SOURCES))
    tmp = lib + f".tmp{os.getpid()}"
    cmd = [exe] + ARCH + ["-shared", "-o", tmp] + objs + ["-cudart", "static"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True,
                extra=["-Xptxas", "-v"] if "--ptxas-v" in sys.argv else None))
