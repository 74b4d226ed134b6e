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
SOURCES = [os.path.join(CSRC, f) for f in ("ip_mhsa.cu", "ip_linear.cu", "ip_norm.cu",
                                           "ip_block.cu")]
DEPS = SOURCES + [os.path.join(CSRC, f) for f in ("ip_mhsa_kernels.cuh", "ip_linear_kernels.cuh",
                                                  "ip_norm_kernels.cuh", "ip_block_kernels.cuh",
                                                  "ip_ptx.cuh",
                                                  "ip_probe.cuh", "ip_host_util.h")] + [
    os.path.join(INCLUDE, "ip_mhsa.h")]
ARCH = "-gencode=arch=compute_103a,code=sm_103a"


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the GPU library cannot be built")


FLAGS = [ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC"]


def compile_command(src: str, obj: str) -> list[str]:
    return [nvcc()] + FLAGS + ["-I" + INCLUDE, "-c", "-o", obj, src]


def link_command(objs: list[str], out: str) -> list[str]:
    return [nvcc(), ARCH, "-shared", "-o", out] + objs


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(d) <= t for d in DEPS)


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile (if stale) and return the path of libipmhsa.so."""
    if not force and up_to_date():
        return LIB
    tag = f".tmp{os.getpid()}"
    objs = [os.path.join(CSRC, os.path.basename(s) + tag + ".o") for s in SOURCES]
    try:
        # the translation units compile in parallel, then one link
        procs = []
        for src, obj in zip(SOURCES, objs):
            cmd = compile_command(src, obj)
            if verbose:
                print(" ".join(cmd), flush=True)
            procs.append((cmd, subprocess.Popen(cmd, cwd=CSRC)))
        for cmd, p in procs:
            if p.wait() != 0:
                raise subprocess.CalledProcessError(p.returncode, cmd)
        tmp = LIB + tag
        subprocess.run(link_command(objs, tmp), check=True, cwd=CSRC)
        os.replace(tmp, LIB)
    finally:
        for obj in objs:
            if os.path.exists(obj):
                os.unlink(obj)
    return LIB


if __name__ == "__main__":
    print(build(force=True, verbose=True))
