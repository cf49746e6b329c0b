"""Helpers for the GPU parity tests: drive the C ABI and the oracle side by side.

Inputs come from the shared seeded generator (synth); the oracle side keeps its
own position bookkeeping (oracle.OracleCache) and re-derives every K/V row it
attends over from its position -- nothing expected is ever read back from the
CUDA path except the values under test.
"""
import numpy as np

import oracle
import synth

MAX_ABS = 2e-2     # attention tolerance (bf16 inputs, fp32 accumulation, bf16 output)
MEAN_REL = 5e-3    # sum |o - o*| / sum |o*|
# Window scores of the scored comparator (sums of softmax weights, fp32 logits and exp2 on the GPU):
# each weight carries a relative error of order 1e-5 (fp32 dot products of bf16 rows, the merged
# softmax statistics, exp2); 1e-3 relative leaves two orders of margin.
SCORE_RTOL = 1e-3
SCORE_ATOL = 1e-7


def bf16_to_f64(x):
    return synth.bf16_bits_to_f32(np.asarray(x).view(np.uint16)).astype(np.float64)


def check_scores(got, ref, what=""):
    got = np.asarray(got, dtype=np.float64)
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    err = np.abs(got - ref)
    bad = err > SCORE_RTOL * np.abs(ref) + SCORE_ATOL
    assert not bad.any(), f"{what}: {int(bad.sum())} scores off, worst {float((err / (np.abs(ref) + 1e-30)).max()):.3g}"


def check_scored_decision(got, ref, K, what=""):
    """The kernel decides with its fp32 scores; where the fp64 scores decide differently, the
    candidates concerned must sit at the threshold (their pooled fp64 score within tolerance of
    the K-th largest)."""
    if K == 0 or got.size == 0:
        return 0
    pg = oracle.max_pool(np.asarray(got, dtype=np.float64))
    pr = oracle.max_pool(ref)
    kg, kr = set(oracle.select_top(pg, K).tolist()), set(oracle.select_top(pr, K).tolist())
    thr = np.sort(pr)[::-1][K - 1]
    for j in kg ^ kr:
        assert abs(pr[j] - thr) <= SCORE_RTOL * thr + SCORE_ATOL, f"{what}: candidate {j} far from the threshold"
    return len(kg ^ kr)


def check_attention(got_bits, ref, what=""):
    got = bf16_to_f64(got_bits)
    err = np.abs(got - ref)
    mx = float(err.max()) if err.size else 0.0
    rel = float(err.sum() / max(np.abs(ref).sum(), 1e-30)) if err.size else 0.0
    assert mx < MAX_ABS and rel < MEAN_REL, f"{what}: max-abs {mx:.3g} mean-rel {rel:.3g}"
    return mx, rel


class Runner:
    """A small workload run through the C ABI with an oracle mirror of every head."""

    def __init__(self, L, H, KVH, prompt_lens, K, r, eseed, dseed, key_scale=None, D=128, fused=False, policy=0,
                 block=1, compaction=0, attn_shape=0, prompt_pool=None):
        import torch

        import paper_2609_03430_gb300 as ra

        self.ra, self.torch = ra, torch
        self.L, self.H, self.KVH, self.D = L, H, KVH, D
        self.G = H // KVH
        self.lp = list(prompt_lens)
        self.B = len(self.lp)
        self.K, self.r, self.eseed, self.dseed = K, r, eseed, dseed
        self.key_scale = key_scale  # fp32 [L][KVH][D] or None
        self.req = [0] * self.B  # requests each slot took after the first (their rows differ: see sid)
        self.cache = ra.RandomAttentionCache(L, H, KVH, D, self.lp, K, r, eseed, policy=policy, block=block,
                                             compaction=compaction, prompt_pool=prompt_pool)
        self.ctx = self.cache.ctx
        if attn_shape:
            ra.ra_set_attention_shape(self.ctx, attn_shape)
        self.orc = oracle.OracleCache(L, KVH, self.lp, K, r, eseed, policy=policy, block=block, compaction=compaction)
        self.policy = policy
        self.qsteps = [[] for _ in range(self.B)]  # step index of each of a sequence's decode steps
        self.step_scale = []  # attention scale of every step (the window's weights use it)
        self.scored_rounds = 0
        self.near_ties = 0
        self.dev = torch.device("cuda")
        self.step_idx = 0
        self.fused = fused  # True: one ra_decode_layer call per layer instead of append/evict/attend
        self.active = [True] * self.B
        maxlp = max(max(self.lp), 1)
        for l in range(L):
            k = np.zeros((self.B, KVH, maxlp, D), np.uint16)
            v = np.zeros_like(k)
            for b in range(self.B):
                for h in range(KVH):
                    if self.lp[b]:
                        k[b, h, : self.lp[b]] = self.krows(l, b, h, np.arange(self.lp[b]))
                        v[b, h, : self.lp[b]] = self.vrows(l, b, h, np.arange(self.lp[b]))
            tk, tv = self.up(k), self.up(v)
            ra.ra_prefill(self.ctx, l, tk.data_ptr(), tv.data_ptr(), maxlp)
        torch.cuda.synchronize()

    def up(self, a):
        return self.torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(self.dev)

    def sid(self, b):
        """The generator's sequence index of slot b's current request."""
        return b + 64 * self.req[b]

    def krows(self, l, b, h, pos):
        sc = None if self.key_scale is None else self.key_scale[l, h]
        return synth.kv_rows(self.dseed, 0, l, self.sid(b), h, pos, self.D, sc)

    def vrows(self, l, b, h, pos):
        return synth.kv_rows(self.dseed, 1, l, self.sid(b), h, pos, self.D)

    def qrows(self, l, b, step):
        return synth.q_rows(self.dseed, l, self.sid(b), np.arange(self.H), step, self.D)

    def admit(self, b, prompt_len):
        """Finish slot b's request and admit a new one with its own prompt (ra_admit)."""
        self.set_active(b, False)
        self.req[b] += 1
        self.qsteps[b] = []  # the new request's decode steps
        self.lp[b] = prompt_len
        k = np.zeros((self.L, self.KVH, max(prompt_len, 1), self.D), np.uint16)
        v = np.zeros_like(k)
        for l in range(self.L):
            for h in range(self.KVH):
                if prompt_len:
                    k[l, h, :prompt_len] = self.krows(l, b, h, np.arange(prompt_len))
                    v[l, h, :prompt_len] = self.vrows(l, b, h, np.arange(prompt_len))
        tk, tv = self.up(k), self.up(v)
        self.ra.ra_admit(self.ctx, b, prompt_len, tk.data_ptr(), tv.data_ptr(), max(prompt_len, 1))
        self.torch.cuda.synchronize()
        self.orc.admit(b, prompt_len)
        self.active[b] = True

    def set_active(self, b, on):
        self.active[b] = on
        self.ra.ra_set_active(self.ctx, b, on)

    def step(self, check_attn_layers=(), scale=0.0):
        """One decode step over all layers; returns {layer: n_fired} and checks attention where asked."""
        fired = {}
        outs = {}
        for b in range(self.B):
            if self.active[b]:
                self.qsteps[b].append(self.step_idx)
        self.step_scale.append(scale)
        scored = self.policy == oracle.POLICY_SNAPKV
        # (fused calls: layer 0's call may run every layer's round of the step, so each layer's
        # evictions are counted from the step's start)
        start = ([[self.ra.ra_get_counters(self.ctx, b, l)[2] for b in range(self.B)] for l in range(self.L)]
                 if self.fused else None)
        for l in range(self.L):
            k = np.zeros((self.B, self.KVH, self.D), np.uint16)
            v = np.zeros_like(k)
            for b in range(self.B):
                if not self.active[b]:
                    continue
                pos = self.orc.append(b, l)
                for h in range(self.KVH):
                    k[b, h] = self.krows(l, b, h, [pos])[0]
                    v[b, h] = self.vrows(l, b, h, [pos])[0]
            tk, tv = self.up(k), self.up(v)  # keep both alive: a freed temporary would be reused for the next
            q = np.stack([self.qrows(l, b, self.step_idx) for b in range(self.B)])
            out = self.torch.zeros((self.B, self.H, self.D), dtype=self.torch.int16, device=self.dev)
            tq = self.up(q)
            if not scored:
                nf = sum(1 for b in range(self.B) if self.active[b] and self.orc.evict(b, l))
            if self.fused:
                self.ra.ra_decode_layer(self.ctx, l, tq.data_ptr(), tk.data_ptr(), tv.data_ptr(), out.data_ptr(), scale)
                n = sum(self.ra.ra_get_counters(self.ctx, b, l)[2] - start[l][b] for b in range(self.B))
            else:
                self.ra.ra_append_kv(self.ctx, l, tk.data_ptr(), tv.data_ptr())
                n = self.ra.ra_evict(self.ctx, l)
                self.ra.ra_decode_attn(self.ctx, l, tq.data_ptr(), out.data_ptr(), scale)
            if scored:  # the oracle's round needs the kernel's scores of this step
                nf = sum(1 for b in range(self.B) if self.active[b] and self.orc.evict(b, l, scorer=self.scorer))
            assert n == nf, (l, n, nf)
            fired[l] = n
            if l in check_attn_layers:
                outs[l] = (q, out)
        for l, (q, out) in outs.items():
            self.check_layer_attention(l, q, out.cpu().numpy(), scale)
        self.step_idx += 1
        return fired

    def window(self, l, b, h, g):
        """Query rows [r][G][D] and positions of the window at an eviction after token g."""
        steps = range(g - self.r, g)  # 1-based decode steps of the window
        heads = np.arange(h * self.G, (h + 1) * self.G)
        q = np.stack([synth.q_rows(self.dseed, l, self.sid(b), heads, self.qsteps[b][s - 1], self.D) for s in steps])
        return q, np.array([self.lp[b] + s - 1 for s in steps], dtype=np.int32)

    def scorer(self, b, l, h, cur):
        """Oracle scorer of the scored policy: the fp64 window scores must match the kernel's within
        tolerance; the round then follows the kernel's fp32 scores (see check_scored_decision)."""
        g, n = int(self.orc.g[b, l]), cur.size - self.r
        q, qpos = self.window(l, b, h, g)
        kpos = self.orc.positions(b, l, h)
        scales = {self.step_scale[self.qsteps[b][s - 1]] for s in range(g - self.r, g)}
        assert len(scales) == 1, "one attention scale per window"
        ref = oracle.window_scores(q, qpos, self.krows(l, b, h, kpos), kpos, scales.pop())[self.lp[b]:self.lp[b] + n]
        got = self.ra.ra_get_scores(self.ctx, l, b, h, self.K + 2 * self.r)
        what = f"scores l{l} b{b} h{h} g{g}"
        check_scores(got, ref, what)
        self.near_ties += check_scored_decision(got, ref, self.K, what)
        self.scored_rounds += 1
        return got.astype(np.float64)

    def check_layer_attention(self, l, q, got, scale=0.0):
        for b in range(self.B):
            if not self.active[b]:
                continue
            for h in range(self.KVH):
                pos = self.orc.positions(b, l, h)
                ref = oracle.attend(q[b, h * self.G:(h + 1) * self.G], self.krows(l, b, h, pos),
                                    self.vrows(l, b, h, pos), scale)
                check_attention(got[b, h * self.G:(h + 1) * self.G], ref, f"layer {l} seq {b} head {h}")

    def check_state(self, layers=None):
        """Bit-exact: positions and cached K/V rows of every head equal the oracle's."""
        for l in range(self.L) if layers is None else layers:
            for b in range(self.B):
                g, c, nev = self.ra.ra_get_counters(self.ctx, b, l)
                assert g == self.orc.g[b, l] and nev == self.orc.n_evictions[b, l]
                for h in range(self.KVH):
                    want = self.orc.gen[(b, l, h)]
                    assert c == want.size
                    got = self.ra.ra_get_positions(self.ctx, l, b, h, self.K + 2 * self.r)
                    np.testing.assert_array_equal(got, want, err_msg=f"positions l{l} b{b} h{h}")
                    kk, vv = self.ra.ra_get_kv(self.ctx, l, b, h, self.lp[b] + self.K + 2 * self.r)
                    allpos = self.orc.positions(b, l, h)
                    np.testing.assert_array_equal(kk, self.krows(l, b, h, allpos), err_msg=f"K rows l{l} b{b} h{h}")
                    np.testing.assert_array_equal(vv, self.vrows(l, b, h, allpos), err_msg=f"V rows l{l} b{b} h{h}")

    def restore_full(self, g, layers=(0,)):
        """Every sequence of the given layers: g tokens generated, the newest K + 2r - 1 of them cached
        (one append short of capacity), prompt as prefilled; the oracle mirror gets the same state.
        With g + 1 a multiple of r, the next step fires a round over K + r candidates."""
        c = self.K + 2 * self.r - 1
        for l in layers:
            pos = np.zeros((self.B, self.KVH, c), np.int32)
            kk = np.zeros((self.B, self.KVH, c, self.D), np.uint16)
            vv = np.zeros_like(kk)
            for b in range(self.B):
                p = self.lp[b] + np.arange(g - c, g)
                for h in range(self.KVH):
                    pos[b, h] = p
                    kk[b, h] = self.krows(l, b, h, p)
                    vv[b, h] = self.vrows(l, b, h, p)
                    self.orc.gen[(b, l, h)] = p.astype(np.int32)
                self.orc.g[b, l] = g
            tp = self.torch.from_numpy(pos).cuda()
            tk, tv = self.up(kk), self.up(vv)
            self.ra.ra_restore(self.ctx, l, [g] * self.B, [c] * self.B, tp.data_ptr(), tk.data_ptr(), tv.data_ptr(), c)
            self.torch.cuda.synchronize()
        self.step_idx = g

    def close(self):
        self.ra.ra_check_device(self.ctx)
        self.cache.close()
