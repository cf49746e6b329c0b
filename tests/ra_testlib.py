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


def bf16_to_f64(x):
    return synth.bf16_bits_to_f32(np.asarray(x).view(np.uint16)).astype(np.float64)


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
                 block=1):
        import torch

        import paper_2609_03430_gb300 as ra

        self.ra, self.torch = ra, torch
        self.L, self.H, self.KVH, self.D = L, H, KVH, D
        self.G = H // KVH
        self.lp = list(prompt_lens)
        self.B = len(self.lp)
        self.K, self.r, self.eseed, self.dseed = K, r, eseed, dseed
        self.key_scale = key_scale  # fp32 [L][KVH][D] or None
        self.cache = ra.RandomAttentionCache(L, H, KVH, D, self.lp, K, r, eseed)
        self.ctx = self.cache.ctx
        self.orc = oracle.OracleCache(L, KVH, self.lp, K, r, eseed, policy=policy, block=block)
        if policy:
            ra.ra_set_policy(self.ctx, policy, block)
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

    def krows(self, l, b, h, pos):
        sc = None if self.key_scale is None else self.key_scale[l, h]
        return synth.kv_rows(self.dseed, 0, l, b, h, pos, self.D, sc)

    def vrows(self, l, b, h, pos):
        return synth.kv_rows(self.dseed, 1, l, b, h, pos, self.D)

    def set_active(self, b, on):
        self.active[b] = on
        self.ra.ra_set_active(self.ctx, b, on)

    def step(self, check_attn_layers=(), scale=0.0):
        """One decode step over all layers; returns {layer: n_fired} and checks attention where asked."""
        fired = {}
        outs = {}
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
            q = np.stack([synth.q_rows(self.dseed, l, b, np.arange(self.H), self.step_idx, self.D)
                          for b in range(self.B)])
            out = self.torch.zeros((self.B, self.H, self.D), dtype=self.torch.int16, device=self.dev)
            tq = self.up(q)
            nf = sum(1 for b in range(self.B) if self.active[b] and self.orc.evict(b, l))
            if self.fused:
                before = [self.ra.ra_get_counters(self.ctx, b, l)[2] for b in range(self.B)]
                self.ra.ra_decode_layer(self.ctx, l, tq.data_ptr(), tk.data_ptr(), tv.data_ptr(), out.data_ptr(), scale)
                n = sum(self.ra.ra_get_counters(self.ctx, b, l)[2] - before[b] for b in range(self.B))
            else:
                self.ra.ra_append_kv(self.ctx, l, tk.data_ptr(), tv.data_ptr())
                n = self.ra.ra_evict(self.ctx, l)
                self.ra.ra_decode_attn(self.ctx, l, tq.data_ptr(), out.data_ptr(), scale)
            assert n == nf, (l, n, nf)
            fired[l] = n
            if l in check_attn_layers:
                outs[l] = (q, out)
        for l, (q, out) in outs.items():
            self.check_layer_attention(l, q, out.cpu().numpy(), scale)
        self.step_idx += 1
        return fired

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

    def close(self):
        self.ra.ra_check_device(self.ctx)
        self.cache.close()
