"""Builds the GPU library ``libipmhsa.so`` in-tree with nvcc for sm_103a.

The library is the whole product path: the C ABI of include/ip_mhsa.h and
the CUDA kernels behind it.  Nothing here needs a GPU; nvcc cross-compiles.
"""
from __future__ import annotations

import os
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIB = os.path.join(PKG, "libipmhsa.so")
SOURCES = [os.path.join(CSRC, "ip_mhsa.cu")]
DEPS = SOURCES + [os.path.join(CSRC, "ip_mhsa_kernels.cuh"), os.path.join(INCLUDE, "ip_mhsa.h")]
ARCH = "-gencode=arch=compute_103a,code=sm_103a"


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the GPU library cannot be built")


def command(out: str) -> list[str]:
    return [nvcc(), ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-shared",
            "-I" + INCLUDE, "-o", out] + SOURCES


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(d) <= t for d in DEPS)


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile (if stale) and return the path of libipmhsa.so."""
    if not force and up_to_date():
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = command(tmp)
    if verbose:
        print(" ".join(cmd), flush=True)
    subprocess.run(cmd, check=True, cwd=CSRC)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force=True, verbose=True))
