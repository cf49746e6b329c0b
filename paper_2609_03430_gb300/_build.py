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
# (source, object, extra flags): the attention file is built twice, once per kernel shape.
UNITS = [
    ("ra_api.cu", "ra_api.o", []),
    ("ra_evict.cu", "ra_evict.o", []),
    ("ra_attn.cu", "ra_attn_wide.o", ["-DRA_ATTN_NS=attn_wide", "-DRA_ATTN_TILE=48", "-DRA_ATTN_WARPS=4"]),
    ("ra_attn.cu", "ra_attn_narrow.o",
     ["-DRA_ATTN_NS=attn_narrow", "-DRA_ATTN_TILE=32", "-DRA_ATTN_WARPS=6", "-DRA_ATTN_TRANSPOSED=1"]),
    ("ra_score.cu", "ra_score.o", []),
]
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
    """Start one nvcc per translation unit; returns [(popen, object path, command)]."""
    os.makedirs(BUILD, exist_ok=True)
    procs = []
    for src, obj_name, unit_flags in UNITS:
        obj = os.path.join(BUILD, obj_name)
        cmd = ["nvcc", *ARCH, *FLAGS, *unit_flags, *EXTRA, "-c", os.path.join(CSRC, src), "-o", obj]
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
