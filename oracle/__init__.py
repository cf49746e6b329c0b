"""CPU oracle for Random Attention's decode hot path -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
may import this package.  The product path (``paper_2609_03430_gb300``) never
does, and the two share no code: the arithmetic lives in ``ra_oracle.c``
(plain C, fp64, single-threaded), and this module is the ctypes glue plus the
per-(sequence, layer, KV head) bookkeeping of the eviction state machine.

Paper sections followed (Random Attention, arXiv 2609.03430):
  * section 2 "Periodic eviction with budget K and buffer r", Eq. 1 -- trigger
    and top-K keep;
  * section 3 -- the prompt is never a candidate; every other cached position
    draws an i.i.d. uniform score per KV head at every eviction;
  * Appendix F "Engine details" -- every r=64 steps once the cache exceeds
    K+r; keep-sets sorted chronologically; GQA query groups share their KV
    head's keep-set; keys stored post-RoPE (so attention applies no rotation);
  * section 2 "Notation" -- o_t = sum_i softmax_i(q.k_i/sqrt(d)) v_i;
  * Appendix G (a keep-set is a random permutation of slot indices) -- the
    order-free hole-filling compaction, keys drawn per position;
  * section 2 "Baselines as choices of s" -- the SnapKV window score of the
    scored comparator (window attention, max-pooled, top-K, prompt pinned).

Budget convention: ``K`` here counts retained *generated* tokens; the paper's
budget includes the prompt (K_paper = prompt_len + K), see
``paper_budget_to_generated``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ra_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_build", "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile ra_oracle.c with gcc into oracle/_build/liboracle.so."""
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        u32p = ctypes.POINTER(ctypes.c_uint32)
        i32p = ctypes.POINTER(ctypes.c_int32)
        u16p = ctypes.POINTER(ctypes.c_uint16)
        f64p = ctypes.POINTER(ctypes.c_double)
        lib.ora_philox4x32_10.argtypes = [u32p, u32p, u32p]
        lib.ora_philox4x32_10.restype = None
        lib.ora_random_key.argtypes = [ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32,
                                       ctypes.c_uint32, ctypes.c_uint32]
        lib.ora_random_key.restype = ctypes.c_uint32
        lib.ora_select_keep.argtypes = [u32p, ctypes.c_int, ctypes.c_int, i32p]
        lib.ora_select_keep.restype = ctypes.c_int
        lib.ora_should_evict.argtypes = [ctypes.c_int] * 4
        lib.ora_should_evict.restype = ctypes.c_int
        lib.ora_evict_head.argtypes = [i32p, ctypes.POINTER(ctypes.c_int), ctypes.c_int, ctypes.c_int,
                                       ctypes.c_int, ctypes.c_uint64, ctypes.c_int, ctypes.c_int, i32p]
        lib.ora_evict_head.restype = ctypes.c_int
        lib.ora_attend.argtypes = [u16p, u16p, u16p, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                   ctypes.c_double, f64p]
        lib.ora_head_stream.argtypes = [ctypes.c_uint32, ctypes.c_uint32]
        lib.ora_head_stream.restype = ctypes.c_uint32
        lib.ora_policy_key.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32,
                                       ctypes.c_uint32, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_uint32,
                                       ctypes.c_uint32, ctypes.c_int32, ctypes.c_int32, ctypes.c_uint32]
        lib.ora_policy_key.restype = ctypes.c_uint32
        lib.ora_evict_head_policy.argtypes = [i32p, ctypes.POINTER(ctypes.c_int), ctypes.c_int, ctypes.c_int,
                                              ctypes.c_int, ctypes.c_uint64, ctypes.c_int, ctypes.c_int,
                                              ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                              ctypes.c_uint32, i32p]
        lib.ora_evict_head_policy.restype = ctypes.c_int
        lib.ora_attend.restype = None
        lib.ora_position_key.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32,
                                         ctypes.c_uint32, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_int32,
                                         ctypes.c_int32, ctypes.c_uint32]
        lib.ora_position_key.restype = ctypes.c_uint32
        lib.ora_evict_head_holefill.argtypes = [i32p, ctypes.POINTER(ctypes.c_int), ctypes.c_int, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_uint64, ctypes.c_int, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                ctypes.c_uint32, i32p]
        lib.ora_evict_head_holefill.restype = ctypes.c_int
        lib.ora_window_scores.argtypes = [u16p, i32p, ctypes.c_int, ctypes.c_int, u16p, i32p, ctypes.c_int,
                                          ctypes.c_int, ctypes.c_double, f64p]
        lib.ora_window_scores.restype = None
        lib.ora_max_pool.argtypes = [f64p, ctypes.c_int, ctypes.c_int, f64p]
        lib.ora_max_pool.restype = None
        lib.ora_select_top.argtypes = [f64p, ctypes.c_int, ctypes.c_int, i32p]
        lib.ora_select_top.restype = ctypes.c_int
        lib.ora_evict_head_scored.argtypes = [i32p, ctypes.POINTER(ctypes.c_int), ctypes.c_int, ctypes.c_int,
                                              ctypes.c_int, f64p, ctypes.c_int, i32p]
        lib.ora_evict_head_scored.restype = ctypes.c_int
        _lib = lib
    return _lib


def _ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


# --------------------------------------------------------------------------- arithmetic
def philox4x32_10(ctr, key) -> np.ndarray:
    """Philox4x32-10 block (SC'11): ctr = 4 x uint32, key = 2 x uint32 -> 4 x uint32."""
    lib = _load()
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib.ora_philox4x32_10(_ptr(c, ctypes.c_uint32), _ptr(k, ctypes.c_uint32), _ptr(out, ctypes.c_uint32))
    return out


def random_key(seed: int, layer: int, head_id: int, step: int, j: int) -> int:
    """Section 3's per-candidate uniform score as a 32-bit Philox word."""
    return int(_load().ora_random_key(seed, layer, head_id, step, j))


def random_keys(seed: int, layer: int, head_id: int, step: int, n: int) -> np.ndarray:
    lib = _load()
    return np.array([lib.ora_random_key(seed, layer, head_id, step, j) for j in range(n)], dtype=np.uint32)


def select_keep(keys: np.ndarray, K: int) -> np.ndarray:
    """Eq. 1: ordinals of the K smallest (key, ordinal), ascending."""
    keys = np.ascontiguousarray(keys, dtype=np.uint32)
    out = np.zeros(max(K, 1), dtype=np.int32)
    rc = _load().ora_select_keep(_ptr(keys, ctypes.c_uint32), int(keys.size), int(K), _ptr(out, ctypes.c_int32))
    if rc != 0:
        raise ValueError("ora_select_keep: bad arguments")
    return out[:K].copy()


def should_evict(g: int, c: int, K: int, r: int) -> bool:
    return bool(_load().ora_should_evict(g, c, K, r))


def evict_head(gen: np.ndarray, g: int, K: int, r: int, seed: int, layer: int, head_id: int):
    """One eviction round on a position list; returns (new_gen, evicted_ordinals)."""
    buf = np.ascontiguousarray(gen, dtype=np.int32).copy()
    c = ctypes.c_int(int(buf.size))
    ev = np.zeros(max(int(buf.size), 1), dtype=np.int32)
    if buf.size == 0:
        return buf, ev[:0]
    m = _load().ora_evict_head(_ptr(buf, ctypes.c_int32), ctypes.byref(c), g, K, r, seed, layer, head_id,
                               _ptr(ev, ctypes.c_int32))
    if m < 0:
        raise RuntimeError("ora_evict_head failed")
    return buf[: c.value].copy(), ev[:m].copy()


POLICY_RANDOM, POLICY_SHARED, POLICY_RECENCY, POLICY_BLOCK, POLICY_SNAPKV = 0, 1, 2, 3, 4
SNAPKV_POOL_RADIUS = 3  # max-pool width 7: the paper gives no width, this is the library's stated choice


def head_stream(admissions: int, head: int) -> int:
    """Key stream of a head: the slot's earlier admissions above the head id (see ra_oracle.c)."""
    return int(_load().ora_head_stream(admissions, head))


def evict_head_policy(gen, g, K, r, seed, layer, seq, kv_heads, h, policy, block=1, admissions=0):
    """One eviction round under a policy variant (random / shared / recency / block)."""
    buf = np.ascontiguousarray(gen, dtype=np.int32).copy()
    c = ctypes.c_int(int(buf.size))
    ev = np.zeros(max(int(buf.size), 1), dtype=np.int32)
    if buf.size == 0:
        return buf, ev[:0]
    m = _load().ora_evict_head_policy(_ptr(buf, ctypes.c_int32), ctypes.byref(c), g, K, r, seed, layer, seq,
                                      kv_heads, h, policy, block, admissions, _ptr(ev, ctypes.c_int32))
    if m < 0:
        raise RuntimeError("ora_evict_head_policy failed")
    return buf[: c.value].copy(), ev[:m].copy()


def attend(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float = 0.0) -> np.ndarray:
    """fp64 decode attention of a GQA group: q [G][d], k/v [n][d] bf16 bits -> [G][d] float64."""
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    G, d = q.shape
    n = k.shape[0]
    assert k.shape == (n, d) and v.shape == (n, d)
    out = np.zeros((G, d), dtype=np.float64)
    _load().ora_attend(_ptr(q, ctypes.c_uint16), _ptr(k, ctypes.c_uint16), _ptr(v, ctypes.c_uint16),
                       n, G, d, float(scale), _ptr(out, ctypes.c_double))
    return out


COMPACT_ORDERED, COMPACT_HOLEFILL = 0, 1


def position_key(policy, seed, layer, seq, kv_heads, h, step, position, block=1, admissions=0) -> int:
    """Policy score of the candidate at `position` when slots carry no order."""
    return int(_load().ora_position_key(policy, seed, layer, seq, kv_heads, h, step, position, block, admissions))


def evict_head_holefill(gen, g, K, r, seed, layer, seq, kv_heads, h, policy=POLICY_RANDOM, block=1, admissions=0):
    """One eviction round with hole-filling compaction; returns (new_gen, evicted_ordinals)."""
    buf = np.ascontiguousarray(gen, dtype=np.int32).copy()
    c = ctypes.c_int(int(buf.size))
    ev = np.zeros(max(int(buf.size), 1), dtype=np.int32)
    if buf.size == 0:
        return buf, ev[:0]
    m = _load().ora_evict_head_holefill(_ptr(buf, ctypes.c_int32), ctypes.byref(c), g, K, r, seed, layer, seq,
                                        kv_heads, h, policy, block, admissions, _ptr(ev, ctypes.c_int32))
    if m < 0:
        raise RuntimeError("ora_evict_head_holefill failed")
    return buf[: c.value].copy(), ev[:m].copy()


def window_scores(q: np.ndarray, q_pos, k: np.ndarray, k_pos, scale: float = 0.0) -> np.ndarray:
    """SnapKV window score of every key (section 2): attention from the window queries
    q [n_q][G][d] (bf16 bits) at positions q_pos, summed over queries and heads, each
    query seeing the keys k [n_k][d] whose positions k_pos are not after its own."""
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    qp = np.ascontiguousarray(q_pos, dtype=np.int32)
    kp = np.ascontiguousarray(k_pos, dtype=np.int32)
    n_q, G, d = q.shape
    n_k = k.shape[0]
    assert k.shape == (n_k, d) and qp.shape == (n_q,) and kp.shape == (n_k,)
    out = np.zeros(max(n_k, 1), dtype=np.float64)
    _load().ora_window_scores(_ptr(q, ctypes.c_uint16), _ptr(qp, ctypes.c_int32), n_q, G, _ptr(k, ctypes.c_uint16),
                              _ptr(kp, ctypes.c_int32), n_k, d, float(scale), _ptr(out, ctypes.c_double))
    return out[:n_k].copy()


def max_pool(s, radius: int = SNAPKV_POOL_RADIUS) -> np.ndarray:
    """Max over the window |j - i| <= radius, clipped to the ends."""
    s = np.ascontiguousarray(s, dtype=np.float64)
    out = np.zeros(max(s.size, 1), dtype=np.float64)
    _load().ora_max_pool(_ptr(s, ctypes.c_double), int(s.size), int(radius), _ptr(out, ctypes.c_double))
    return out[: s.size].copy()


def select_top(s, K: int) -> np.ndarray:
    """Indices of the K largest scores (ties: lower index first), ascending."""
    s = np.ascontiguousarray(s, dtype=np.float64)
    out = np.zeros(max(K, 1), dtype=np.int32)
    if _load().ora_select_top(_ptr(s, ctypes.c_double), int(s.size), int(K), _ptr(out, ctypes.c_int32)) != 0:
        raise ValueError("ora_select_top: bad arguments")
    return out[:K].copy()


def evict_head_scored(gen, g, K, r, raw_scores, radius=SNAPKV_POOL_RADIUS):
    """One scored eviction round: raw_scores[j] ranks candidate j (j < c - r) after max-pooling."""
    buf = np.ascontiguousarray(gen, dtype=np.int32).copy()
    raw = np.ascontiguousarray(raw_scores, dtype=np.float64)
    c = ctypes.c_int(int(buf.size))
    ev = np.zeros(max(int(buf.size), 1), dtype=np.int32)
    if not should_evict(g, int(buf.size), K, r):
        return buf, ev[:0]
    if raw.size != buf.size - r:
        raise ValueError(f"need {buf.size - r} candidate scores, got {raw.size}")
    m = _load().ora_evict_head_scored(_ptr(buf, ctypes.c_int32), ctypes.byref(c), g, K, r,
                                      _ptr(raw, ctypes.c_double), int(radius), _ptr(ev, ctypes.c_int32))
    if m < 0:
        raise RuntimeError("ora_evict_head_scored failed")
    return buf[: c.value].copy(), ev[:m].copy()


def paper_budget_to_generated(K_paper: int, prompt_len: int) -> int:
    """Section 3 keeps the prompt with score +inf inside the top-K, so the
    paper's budget K_paper holds the prompt; this library's K counts the
    generated tokens kept: K = K_paper - prompt_len."""
    if K_paper < prompt_len:
        raise ValueError("the method is defined for budgets that hold the prompt")
    return K_paper - prompt_len


# --------------------------------------------------------------------------- state machine
class OracleCache:
    """Bookkeeping of the cached positions of selected (seq, layer, kv_head) units.

    Per (seq, layer): g = generated tokens appended, and per KV head the list of
    cached generated positions in slot order.  The prompt (positions
    0..prompt_len-1) is implicit and never moves.  Call order per step and layer:
    append -> evict -> attend (the library's stated reading; the paper does not
    fix the order within a step).
    """

    def __init__(self, layers, kv_heads, prompt_lens, K, r, seed, heads=None, policy=0, block=1, compaction=0):
        self.L = layers
        self.KVH = kv_heads
        self.prompt_lens = [int(x) for x in prompt_lens]
        self.B = len(self.prompt_lens)
        self.K = K
        self.r = r
        self.seed = seed
        self.policy, self.block, self.compaction = policy, block, compaction
        self.g = np.zeros((self.B, layers), dtype=np.int64)
        # heads: iterable of (seq, layer, kv_head) to track; None = all
        if heads is None:
            heads = [(b, l, h) for b in range(self.B) for l in range(layers) for h in range(kv_heads)]
        self.gen = {tuple(u): np.zeros(0, dtype=np.int32) for u in heads}
        self.n_evictions = np.zeros((self.B, layers), dtype=np.int64)
        self.admissions = [0] * self.B  # requests each slot took after the first batch

    def restore(self, seq, layer, g, positions_by_head):
        self.g[seq, layer] = g
        for h in range(self.KVH):
            if (seq, layer, h) in self.gen:
                self.gen[(seq, layer, h)] = np.asarray(positions_by_head[h], dtype=np.int32).copy()

    def admit(self, seq, prompt_len):
        """A new request in slot `seq` (the previous one finished): its own prompt of prompt_len
        positions, nothing generated or cached in any layer, the slot's next key stream."""
        self.prompt_lens[seq] = int(prompt_len)
        self.admissions[seq] += 1
        for l in range(self.L):
            self.g[seq, l] = 0
            self.n_evictions[seq, l] = 0
            for h in range(self.KVH):
                if (seq, l, h) in self.gen:
                    self.gen[(seq, l, h)] = np.zeros(0, dtype=np.int32)

    def c(self, seq, layer):
        """Cached generated count (identical for every head of a (seq, layer))."""
        for h in range(self.KVH):
            key = (seq, layer, h)
            if key in self.gen:
                return int(self.gen[key].size)
        raise KeyError((seq, layer))

    def append(self, seq, layer):
        pos = self.prompt_lens[seq] + int(self.g[seq, layer])
        for h in range(self.KVH):
            key = (seq, layer, h)
            if key in self.gen:
                self.gen[key] = np.append(self.gen[key], np.int32(pos))
        self.g[seq, layer] += 1
        return pos

    def evict(self, seq, layer, scorer=None):
        """Returns {kv_head: evicted ordinals} for the tracked heads if the trigger fired.

        Under the scored policy, scorer(seq, layer, kv_head, cached_positions) returns the raw
        window score of each candidate (all cached generated slots but the newest r)."""
        g = int(self.g[seq, layer])
        fired = {}
        for h in range(self.KVH):
            key = (seq, layer, h)
            if key not in self.gen:
                continue
            cur = self.gen[key]
            if not should_evict(g, int(cur.size), self.K, self.r):
                continue
            a = self.admissions[seq]
            if self.compaction == COMPACT_HOLEFILL:
                new, ev = evict_head_holefill(cur, g, self.K, self.r, self.seed, layer, seq, self.KVH, h,
                                              self.policy, self.block, a)
            elif self.policy == POLICY_RANDOM:
                new, ev = evict_head(cur, g, self.K, self.r, self.seed, layer, head_stream(a, seq * self.KVH + h))
            elif self.policy == POLICY_SNAPKV:
                new, ev = evict_head_scored(cur, g, self.K, self.r, scorer(seq, layer, h, cur))
            else:
                new, ev = evict_head_policy(cur, g, self.K, self.r, self.seed, layer, seq, self.KVH, h,
                                            self.policy, self.block, a)
            self.gen[key] = new
            fired[h] = ev
        if fired:
            self.n_evictions[seq, layer] += 1
        return fired

    def positions(self, seq, layer, h):
        """All attended positions of a head: prompt then cached generated, in slot order."""
        return np.concatenate([np.arange(self.prompt_lens[seq], dtype=np.int32), self.gen[(seq, layer, h)]])
