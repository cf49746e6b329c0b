"""Build libra.so (the C-ABI CUDA library) in-tree for sm_103a with nvcc.

Translation units compile in parallel into ``_build/`` and link into
``paper_2609_03430_gb300/libra.so``.  Nothing is installed anywhere else.
"""
from __future__ import annotations

import os
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libra.so")
SOURCES = ["ra_api.cu", "ra_evict.cu", "ra_attn.cu", "ra_score.cu"]
HEADERS = ["ra_internal.h", "ra_ptx.cuh"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I" + os.path.join(ROOT, "include"), "-I" + CSRC]
# Extra nvcc flags, e.g. -DRA_ATTN_S_LPS=16 ... to build another attention kernel shape.
EXTRA = os.environ.get("RA_NVCC_FLAGS", "").split()


def _inputs():
    return [os.path.join(CSRC, s) for s in SOURCES + HEADERS] + [os.path.join(ROOT, "include", "ra.h")]


def needs_build() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(p) > t for p in _inputs())


def compile_procs():
    """Start one nvcc per translation unit; returns [(popen, object path)]."""
    os.makedirs(BUILD, exist_ok=True)
    procs = []
    for s in SOURCES:
        obj = os.path.join(BUILD, s.replace(".cu", ".o"))
        cmd = ["nvcc", *ARCH, *FLAGS, *EXTRA, "-c", os.path.join(CSRC, s), "-o", obj]
        procs.append((subprocess.Popen(cmd), obj, cmd))
    return procs


def link(objs):
    tmp = LIB + f".tmp{os.getpid()}"
    subprocess.check_call(["nvcc", *ARCH, "-shared", "-o", tmp, *objs])
    os.replace(tmp, LIB)


def build(force: bool = False) -> str:
    if not force and not needs_build():
        return LIB
    procs = compile_procs()
    bad = [cmd for (p, _, cmd) in procs if p.wait() != 0]
    if bad:
        raise RuntimeError("nvcc failed: " + " ".join(bad[0]))
    link([obj for (_, obj, _) in procs])
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
