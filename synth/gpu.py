"""ctypes binding of the GPU twin of the synthetic input generator (synth_gpu.cu).

Input generation only.  ``build()`` compiles ``synth_gpu.cu`` for sm_103a into
``synth/_build/libra_synth.so``; ``fill_rows`` writes bf16 rows into a torch
CUDA tensor from a positions tensor, bit-identical to ``synth.kv_rows``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth_gpu.cu")
_LIB = os.path.join(_HERE, "_build", "libra_synth.so")
_lib = None

NVCC_ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def build_cmd():
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    return ["nvcc", *NVCC_ARCH, "-O3", "-lineinfo", "-std=c++17", "-shared", "-Xcompiler", "-fPIC",
            "-o", _LIB, _SRC]


def needs_build() -> bool:
    return not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC)


def build(force: bool = False) -> str:
    if force or needs_build():
        subprocess.check_call(build_cmd())
    return _LIB


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB):
            raise RuntimeError("synth GPU library not built: run __graft_entry__.build()")
        lib = ctypes.CDLL(_LIB)
        lib.synth_fill_rows.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                        ctypes.c_int, ctypes.c_uint64, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                        ctypes.c_void_p, ctypes.c_void_p]
        lib.synth_fill_rows.restype = ctypes.c_int
        _lib = lib
    return _lib


def fill_rows(out, pos, seed: int, stream_id: int, layer: int, seq0: int = 0, scale=None, cuda_stream=None):
    """out: uint16/bfloat16 CUDA tensor [B][NH][n][d]; pos: int32 CUDA tensor [B][NH][n]."""
    import torch

    B, NH, n, d = out.shape
    assert pos.shape == (B, NH, n) and pos.dtype == torch.int32 and pos.is_contiguous() and out.is_contiguous()
    if scale is not None:
        assert scale.shape == (NH, d) and scale.dtype == torch.float32 and scale.is_contiguous()
    s = cuda_stream if cuda_stream is not None else torch.cuda.current_stream().cuda_stream
    rc = _load().synth_fill_rows(out.data_ptr(), pos.data_ptr(), B, NH, n, d, seed & 0xFFFFFFFFFFFFFFFF,
                                 stream_id, layer, seq0, None if scale is None else scale.data_ptr(), s)
    if rc != 0:
        raise RuntimeError(f"synth_fill_rows failed: {rc}")
    return out
