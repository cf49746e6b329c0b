"""Seeded synthetic inputs shared by the oracle side and the CUDA side.

This module holds none of the method's arithmetic: no Philox, no selection, no
softmax.  It defines integer-only generators of bf16 K/V/Q values so that the
CPU (numpy, here) and the GPU twin (``synth_gpu.cu``) produce bit-identical
tensors from positions alone.  The oracle re-derives any cache row it needs
from its position, so no expected value ever comes from the CUDA path.

Value recipe (the paper's models are not available; these stand in for the
post-RoPE keys, values and queries of Qwen3-4B/14B/32B and Phi-4-reasoning):
  * element counter  i = ((((stream*2^8 + layer)*2^12 + seq)*2^8 + head)*2^20 + pos)*2^7 + ch
    (stream 0 = K, 1 = V, 2 = Q; for Q, head = query head and pos = decode step);
  * three 64-bit words w_k = SplitMix64(seed + (3i + k + 1) * gamma)
    (Steele, Lea, Flood, OOPSLA 2014), giving twelve 16-bit uniforms x_0..x_11;
  * Irwin-Hall N(0,1) approximation:  n = sum(x) - 6*65535, value = n / 65536,
    exact in fp32 (|n| < 2^24);
  * optional per-(layer, kv head, channel) key scale (fp32), applied as one
    round-to-nearest fp32 multiply;
  * rounded to bf16 with round-to-nearest-even on the fp32 bit pattern.
"""
from __future__ import annotations

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
OFFSET_12 = 6 * 65535

STREAM_K, STREAM_V, STREAM_Q = 0, 1, 2
LIMITS = dict(layer=256, seq=4096, head=256, pos=1 << 20, ch=128)


def splitmix64_mix(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function on uint64 arrays (wrapping arithmetic)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def element_counter(stream, layer, seq, head, pos, ch) -> np.ndarray:
    u = lambda x: np.asarray(x, dtype=np.uint64)
    i = u(stream)
    i = (i << np.uint64(8)) | u(layer)
    i = (i << np.uint64(12)) | u(seq)
    i = (i << np.uint64(8)) | u(head)
    i = (i << np.uint64(20)) | u(pos)
    i = (i << np.uint64(7)) | u(ch)
    return i


def f32_to_bf16_bits(f: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16 on bit patterns (finite inputs)."""
    b = np.asarray(f, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))
    return (b >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_f32(seed: int, stream, layer, seq, head, pos, ch) -> np.ndarray:
    """The exact fp32 Irwin-Hall value (before any scale or bf16 rounding)."""
    i = element_counter(stream, layer, seq, head, pos, ch)
    s = np.uint64(seed & 0xFFFFFFFFFFFFFFFF)
    total = np.zeros(i.shape, dtype=np.int64)
    with np.errstate(over="ignore"):
        base = i * np.uint64(3)
        for k in range(3):
            w = splitmix64_mix(s + (base + np.uint64(k + 1)) * GAMMA)
            for part in range(4):
                total += ((w >> np.uint64(16 * part)) & np.uint64(0xFFFF)).astype(np.int64)
    n = total - OFFSET_12
    return n.astype(np.float32) * np.float32(1.0 / 65536.0)


def values_bf16(seed: int, stream, layer, seq, head, pos, ch, scale=None) -> np.ndarray:
    f = normal_f32(seed, stream, layer, seq, head, pos, ch)
    if scale is not None:
        f = (f * np.asarray(scale, dtype=np.float32)).astype(np.float32)
    return f32_to_bf16_bits(f)


def kv_rows(seed: int, stream: int, layer: int, seq: int, head: int, positions, d: int,
            scale_row=None) -> np.ndarray:
    """Rows [n][d] (bf16 bits) of K (stream 0) or V (stream 1) at the given positions.
    scale_row: optional fp32 [d] per-channel key scale of this (layer, kv head)."""
    pos = np.asarray(positions, dtype=np.int64).reshape(-1, 1)
    ch = np.arange(d, dtype=np.int64).reshape(1, -1)
    sc = None if scale_row is None else np.asarray(scale_row, dtype=np.float32).reshape(1, -1)
    return values_bf16(seed, stream, layer, seq, head, pos, ch, sc)


def q_rows(seed: int, layer: int, seq: int, qheads, step: int, d: int) -> np.ndarray:
    """Query rows [len(qheads)][d] (bf16 bits) of one decode step."""
    qh = np.asarray(qheads, dtype=np.int64).reshape(-1, 1)
    ch = np.arange(d, dtype=np.int64).reshape(1, -1)
    return values_bf16(seed, STREAM_Q, layer, seq, qh, step, ch)


def key_channel_scale(seed: int, layers: int, kv_heads: int, d: int, sigma: float = 0.5) -> np.ndarray:
    """Per-(layer, kv head, channel) LogNormal(0, sigma) key scales, fp32 [L][KVH][d].
    The normal deviate is the same Irwin-Hall recipe on stream 3 (pos = 0)."""
    l = np.arange(layers).reshape(-1, 1, 1)
    h = np.arange(kv_heads).reshape(1, -1, 1)
    c = np.arange(d).reshape(1, 1, -1)
    z = normal_f32(seed, 3, l, 0, h, 0, c).astype(np.float64)
    return np.exp(sigma * z).astype(np.float32)


def uniform_ints(seed: int, n: int, lo: int, hi: int) -> np.ndarray:
    """n integers uniform in [lo, hi] by SplitMix64 + rejection (portable across hosts)."""
    span = hi - lo + 1
    assert span >= 1
    limit = (1 << 64) - ((1 << 64) % span)
    out = []
    ctr = 0
    while len(out) < n:
        ctr += 1
        w = int(splitmix64_mix(np.uint64((seed + ctr * 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF)))
        if w < limit:
            out.append(lo + w % span)
    return np.array(out, dtype=np.int64)
