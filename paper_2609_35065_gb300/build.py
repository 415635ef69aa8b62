"""Build ``libkvs.so`` (the C-ABI library) in-tree with nvcc for sm_103a.

``python -m paper_2609_35065_gb300.build`` or ``build_library()``.  The library
lands in ``paper_2609_35065_gb300/_build/libkvs.so`` (git-ignored); it is
rebuilt when a source or the public header is newer than it.
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
OUT_DIR = os.path.join(PKG, "_build")
LIB = os.path.join(OUT_DIR, "libkvs.so")
SOURCES = [os.path.join(CSRC, f) for f in ("kvs_kernels.cu", "kvs_api.cpp", "kvs_noalloc.cu", "kvs_fp8.cu",
                                           "kvs_tier.cpp")]
DEPS = SOURCES + [os.path.join(CSRC, "kvs_internal.h"), os.path.join(CSRC, "kvs_async.cuh"), os.path.join(INCLUDE, "kvs.h")]
ARCH = "-gencode=arch=compute_103a,code=sm_103a"


def nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libkvs.so")


def command(out: str = LIB, extra: list[str] | None = None) -> list[str]:
    return [nvcc(), "-O3", "-lineinfo", "-std=c++17", ARCH, "-Xcompiler", "-fPIC,-O2,-Wall",
            "-shared", "--threads", "4", "-I", INCLUDE, *SOURCES, "-o", out, *(extra or [])]


def stale(out: str = LIB) -> bool:
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(d) > t for d in DEPS)


def build_library(force: bool = False, verbose: bool = False) -> str:
    os.makedirs(OUT_DIR, exist_ok=True)
    if force or stale():
        tmp = LIB + f".{os.getpid()}.tmp"
        cmd = command(tmp)
        if verbose:
            print(" ".join(cmd), file=sys.stderr)
        subprocess.run(cmd, check=True)
        os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose=True))
