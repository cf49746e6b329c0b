"""Random Attention decode hot path on GB300 (sm_103a): Python binding of libra.so.

The binding only marshals arguments: every step of the path (append, random
eviction with compaction, GQA decode attention) runs in the CUDA kernels of
``libra.so``, whose C ABI is ``include/ra.h``.  Functions keep the C names.
There is no CPU fallback: importing works anywhere, but every call needs the
built library and a CUDA device, and fails loudly otherwise.

``RandomAttentionCache`` is a small convenience wrapper that allocates the
device arena with torch (PyTorch is used for device memory and streams only).
"""
from __future__ import annotations

import ctypes
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libra.so")

RA_OK = 0
RA_ERR_INVALID_ARG = -1
RA_ERR_STATE = -2
RA_ERR_CAPACITY = -3
RA_ERR_CUDA = -4
RA_ERR_DEVICE_TIMEOUT = -5
RA_ERR_UNSUPPORTED = -6
RA_MAX_BATCH = 512
(RA_KERNEL_APPEND, RA_KERNEL_SELECT, RA_KERNEL_COMPACT, RA_KERNEL_ATTN, RA_KERNEL_SCORE_STATS, RA_KERNEL_SCORE_SUM,
 RA_KERNEL_EVICT, RA_KERNEL_PLAN, RA_KERNEL_STACK) = range(9)
KERNEL_NAMES = ["append", "select", "compact", "attn", "score_stats", "score_sum", "evict", "plan", "stack"]
RA_EVICT_AUTO, RA_EVICT_TWO_KERNELS, RA_EVICT_EXACT = 0, 1, 256

# Exported C symbols and their ctypes signatures (kept in the order of include/ra.h).
_vp, _i, _u64, _sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64, ctypes.c_size_t
_i32p = ctypes.POINTER(ctypes.c_int32)
_ip = ctypes.POINTER(ctypes.c_int)
_dp = ctypes.POINTER(ctypes.c_double)
_i64p = ctypes.POINTER(ctypes.c_int64)
SIGNATURES = {
    "ra_create": (_i, [ctypes.POINTER(_vp), _i, _i, _i, _i, _i, _i, _i, _u64]),
    "ra_create_batched": (_i, [ctypes.POINTER(_vp), _i, _i, _i, _i, _i, _i32p, _i, _i, _u64]),
    "ra_device_bytes": (_sz, [_vp]),
    "ra_bind": (_i, [_vp, _vp, _sz, _vp]),
    "ra_prefill": (_i, [_vp, _i, _vp, _vp, _i, _vp]),
    "ra_restore": (_i, [_vp, _i, _i32p, _i32p, _vp, _vp, _vp, _i, _vp]),
    "ra_set_policy": (_i, [_vp, _i, _i]),
    "ra_set_compaction": (_i, [_vp, _i]),
    "ra_set_attention_shape": (_i, [_vp, _i]),
    "ra_set_eviction_kernel": (_i, [_vp, _i]),
    "ra_restore_queries": (_i, [_vp, _i, _vp, ctypes.c_float, _vp]),
    "ra_get_scores": (_i, [_vp, _i, _i, _i, ctypes.POINTER(ctypes.c_float), _i, _ip, _vp]),
    "ra_set_prompt_pool": (_i, [_vp, _i, ctypes.c_longlong]),
    "ra_admit": (_i, [_vp, _i, _i, _vp, _vp, _i, _vp]),
    "ra_set_active": (_i, [_vp, _i, _i]),
    "ra_append_kv": (_i, [_vp, _i, _vp, _vp, _vp]),
    "ra_evict": (_i, [_vp, _i, _ip, _vp]),
    "ra_decode_attn": (_i, [_vp, _i, _vp, _vp, ctypes.c_float, _vp]),
    "ra_decode_attn_noalloc": (_i, [_vp, _i, _vp, _vp, ctypes.c_float, _vp]),
    "ra_decode_layer": (_i, [_vp, _i, _vp, _vp, _vp, _vp, ctypes.c_float, _vp]),
    "ra_decode_step": (_i, [_vp, _vp, _vp, _vp, _vp, ctypes.c_float, _vp]),
    "ra_get_counters": (_i, [_vp, _i, _i, _i32p, _i32p, _i32p]),
    "ra_get_positions": (_i, [_vp, _i, _i, _i, _i32p, _i, _ip, _vp]),
    "ra_get_kv": (_i, [_vp, _i, _i, _i, _vp, _vp, _i, _ip, _vp]),
    "ra_check_device": (_i, [_vp, _vp]),
    "ra_debug_timeout_probe": (_i, [_vp, _u64, _vp]),
    "ra_profile_enable": (_i, [_vp, _i]),
    "ra_profile_read": (_i, [_vp, _i, _dp, _i64p, _dp]),
    "ra_profile_reset": (_i, [_vp]),
    "ra_last_error": (ctypes.c_char_p, [_vp]),
    "ra_destroy": (None, [_vp]),
}

_lib = None


class RAError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"{msg} (code {code})")
        self.code = code


def lib():
    """The loaded libra.so; raises if it has not been built (no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _check(rc, ctx=None):
    if rc != RA_OK:
        msg = lib().ra_last_error(ctx)
        raise RAError(rc, msg.decode() if msg else "error")
    return rc


def _stream_ptr(stream):
    import torch

    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# Thin wrappers with the C names (argument marshalling only).
def ra_create(layers, q_heads, kv_heads, head_dim, prompt_len, K, r, seed):
    ctx = ctypes.c_void_p()
    _check(lib().ra_create(ctypes.byref(ctx), layers, q_heads, kv_heads, head_dim, prompt_len, K, r, seed))
    return ctx


def ra_create_batched(layers, q_heads, kv_heads, head_dim, prompt_lens, K, r, seed):
    arr = (ctypes.c_int32 * len(prompt_lens))(*[int(x) for x in prompt_lens])
    ctx = ctypes.c_void_p()
    _check(lib().ra_create_batched(ctypes.byref(ctx), layers, q_heads, kv_heads, head_dim, len(prompt_lens), arr,
                                   K, r, seed))
    return ctx


def ra_device_bytes(ctx):
    return int(lib().ra_device_bytes(ctx))


def ra_bind(ctx, dev_ptr, nbytes, stream=None):
    return _check(lib().ra_bind(ctx, dev_ptr, nbytes, _stream_ptr(stream)), ctx)


def ra_prefill(ctx, layer, k_ptr, v_ptr, row_stride, stream=None):
    return _check(lib().ra_prefill(ctx, layer, k_ptr, v_ptr, row_stride, _stream_ptr(stream)), ctx)


def ra_restore(ctx, layer, g_list, c_list, pos_ptr, k_ptr, v_ptr, row_stride, stream=None):
    n = len(g_list)
    g = (ctypes.c_int32 * n)(*[int(x) for x in g_list])
    c = (ctypes.c_int32 * n)(*[int(x) for x in c_list])
    return _check(lib().ra_restore(ctx, layer, g, c, pos_ptr, k_ptr, v_ptr, row_stride, _stream_ptr(stream)), ctx)


RA_POLICY_RANDOM, RA_POLICY_SHARED, RA_POLICY_RECENCY, RA_POLICY_BLOCK, RA_POLICY_SNAPKV = 0, 1, 2, 3, 4


def ra_set_policy(ctx, policy, block=1):
    return _check(lib().ra_set_policy(ctx, int(policy), int(block)), ctx)


RA_COMPACT_ORDERED, RA_COMPACT_HOLEFILL, RA_COMPACT_FUSED = 0, 1, 2


RA_ATTN_SHAPE_AUTO, RA_ATTN_SHAPE_WIDE, RA_ATTN_SHAPE_NARROW = 0, 1, 2


def ra_set_attention_shape(ctx, shape):
    return _check(lib().ra_set_attention_shape(ctx, int(shape)), ctx)


def ra_set_eviction_kernel(ctx, mode):
    return _check(lib().ra_set_eviction_kernel(ctx, int(mode)), ctx)


def ra_set_compaction(ctx, mode):
    return _check(lib().ra_set_compaction(ctx, int(mode)), ctx)


def ra_restore_queries(ctx, layer, q_ptr, scale=0.0, stream=None):
    return _check(lib().ra_restore_queries(ctx, layer, q_ptr, float(scale), _stream_ptr(stream)), ctx)


def ra_get_scores(ctx, layer, seq, kv_head, capacity, stream=None):
    import numpy as np

    buf = np.zeros(max(capacity, 1), dtype=np.float32)
    n = ctypes.c_int(0)
    _check(lib().ra_get_scores(ctx, layer, seq, kv_head, buf.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), capacity,
                               ctypes.byref(n), _stream_ptr(stream)), ctx)
    return buf[: n.value].copy()


def ra_set_prompt_pool(ctx, max_prompt_len, pool_positions):
    return _check(lib().ra_set_prompt_pool(ctx, int(max_prompt_len), int(pool_positions)), ctx)


def ra_admit(ctx, seq, prompt_len, k_ptr, v_ptr, row_stride, stream=None):
    return _check(lib().ra_admit(ctx, int(seq), int(prompt_len), k_ptr, v_ptr, int(row_stride), _stream_ptr(stream)), ctx)


def ra_set_active(ctx, seq, active):
    return _check(lib().ra_set_active(ctx, seq, int(bool(active))), ctx)


def ra_append_kv(ctx, layer, k_ptr, v_ptr, stream=None):
    return _check(lib().ra_append_kv(ctx, layer, k_ptr, v_ptr, _stream_ptr(stream)), ctx)


def ra_evict(ctx, layer, stream=None):
    n = ctypes.c_int(0)
    _check(lib().ra_evict(ctx, layer, ctypes.byref(n), _stream_ptr(stream)), ctx)
    return n.value


def ra_decode_attn(ctx, layer, q_ptr, out_ptr, scale=0.0, stream=None):
    return _check(lib().ra_decode_attn(ctx, layer, q_ptr, out_ptr, float(scale), _stream_ptr(stream)), ctx)


def ra_decode_attn_noalloc(ctx, layer, q_ptr, out_ptr, scale=0.0, stream=None):
    return _check(lib().ra_decode_attn_noalloc(ctx, layer, q_ptr, out_ptr, float(scale), _stream_ptr(stream)), ctx)


def ra_decode_layer(ctx, layer, q_ptr, k_ptr, v_ptr, out_ptr, scale=0.0, stream=None):
    return _check(lib().ra_decode_layer(ctx, layer, q_ptr, k_ptr, v_ptr, out_ptr, float(scale), _stream_ptr(stream)),
                  ctx)


def ra_decode_step(ctx, q_ptr, k_ptr, v_ptr, out_ptr, scale=0.0, stream=None):
    return _check(lib().ra_decode_step(ctx, q_ptr, k_ptr, v_ptr, out_ptr, float(scale), _stream_ptr(stream)), ctx)


def ra_get_counters(ctx, seq, layer):
    g, c, n = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    _check(lib().ra_get_counters(ctx, seq, layer, ctypes.byref(g), ctypes.byref(c), ctypes.byref(n)), ctx)
    return g.value, c.value, n.value


def ra_get_positions(ctx, layer, seq, kv_head, capacity, stream=None):
    import numpy as np

    buf = np.zeros(max(capacity, 1), dtype=np.int32)
    n = ctypes.c_int(0)
    _check(lib().ra_get_positions(ctx, layer, seq, kv_head, buf.ctypes.data_as(_i32p), capacity, ctypes.byref(n),
                                  _stream_ptr(stream)), ctx)
    return buf[: n.value].copy()


def ra_get_kv(ctx, layer, seq, kv_head, capacity_rows, head_dim=128, stream=None):
    import numpy as np

    k = np.zeros((max(capacity_rows, 1), head_dim), dtype=np.uint16)
    v = np.zeros_like(k)
    n = ctypes.c_int(0)
    _check(lib().ra_get_kv(ctx, layer, seq, kv_head, k.ctypes.data, v.ctypes.data, capacity_rows, ctypes.byref(n),
                           _stream_ptr(stream)), ctx)
    return k[: n.value].copy(), v[: n.value].copy()


def ra_check_device(ctx, stream=None):
    return _check(lib().ra_check_device(ctx, _stream_ptr(stream)), ctx)


def ra_debug_timeout_probe(ctx, limit_ns, stream=None):
    return _check(lib().ra_debug_timeout_probe(ctx, int(limit_ns), _stream_ptr(stream)), ctx)


def ra_profile_enable(ctx, on=True):
    return _check(lib().ra_profile_enable(ctx, int(bool(on))), ctx)


def ra_profile_read(ctx, kind):
    ms, n, by = ctypes.c_double(), ctypes.c_int64(), ctypes.c_double()
    _check(lib().ra_profile_read(ctx, kind, ctypes.byref(ms), ctypes.byref(n), ctypes.byref(by)), ctx)
    return ms.value, n.value, by.value


def ra_profile_reset(ctx):
    return _check(lib().ra_profile_reset(ctx), ctx)


def ra_last_error(ctx=None):
    m = lib().ra_last_error(ctx)
    return m.decode() if m else ""


def ra_destroy(ctx):
    lib().ra_destroy(ctx)


class RandomAttentionCache:
    """Owns a context and its torch-allocated device arena (uint8 CUDA tensor)."""

    def __init__(self, layers, q_heads, kv_heads, head_dim, prompt_lens, K, r=64, seed=0, device=None, stream=None,
                 policy=RA_POLICY_RANDOM, block=1, compaction=RA_COMPACT_ORDERED, prompt_pool=None):
        import torch

        if isinstance(prompt_lens, int):
            prompt_lens = [prompt_lens]
        self.prompt_lens = [int(x) for x in prompt_lens]
        self.L, self.H, self.KVH, self.D = layers, q_heads, kv_heads, head_dim
        self.B, self.K, self.r, self.seed = len(self.prompt_lens), K, r, seed
        self.ctx = ra_create_batched(layers, q_heads, kv_heads, head_dim, self.prompt_lens, K, r, seed)
        if compaction != RA_COMPACT_ORDERED:
            ra_set_compaction(self.ctx, compaction)
        if policy != RA_POLICY_RANDOM:  # before sizing: the scored policy adds buffers to the arena
            ra_set_policy(self.ctx, policy, block)
        if prompt_pool is not None:  # (max_prompt_len, pool_positions), before sizing
            ra_set_prompt_pool(self.ctx, *prompt_pool)
        self.nbytes = ra_device_bytes(self.ctx)
        dev = torch.device("cuda") if device is None else torch.device(device)
        self.arena = torch.empty(self.nbytes + 256, dtype=torch.uint8, device=dev)
        base = self.arena.data_ptr()
        self.base = (base + 255) // 256 * 256
        ra_bind(self.ctx, self.base, self.nbytes, stream)

    def close(self):
        if getattr(self, "ctx", None) is not None:
            ra_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
