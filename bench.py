#!/usr/bin/env python3
"""Decode-throughput benchmark of the Random Attention hot path on GB300.

A step is one decode step of the whole layer stack through the C ABI
(``ra_decode_step``): for every layer, append the new token's K/V, run the
periodic random eviction (fires every r steps per sequence), and GQA decode
attention over the compacted caches.  Caches start at steady state
(K + r cached generated tokens per head right after an eviction, plus the
prompt), filled on the device by the seeded generator.

Prints ONE JSON line (rank 0).  ``--impl reference`` times the CPU oracle
(the slow, plain reference of what the path computes) on a bounded sample of
the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "decode tokens/sec (all layers, 1 GB300) and % of HBM peak GB/s per kernel"
UNIT = "tokens/s"
D = 128


def _workloads():
    """The five synthetic workloads (shapes of the paper's models; values from synth)."""
    w = {
        1: dict(name="qwen3-4b-shape 1 layer batch 1", L=1, H=32, KVH=8, B=1, lp=[128], K=256, r=64, gen=[1024],
                key_scale=False, dseed=1, eseed=0),
        2: dict(name="qwen3-4b-shape", L=36, H=32, KVH=8, B=16, lp=[512] * 16, K=2048, r=64, gen=[32768] * 16,
                key_scale=True, dseed=2, eseed=2),
        3: dict(name="qwen3-14b-shape", L=40, H=40, KVH=8, B=64, lp=[2048] * 64, K=4096, r=64, gen=[32768] * 64,
                key_scale=False, dseed=3, eseed=3),
        4: dict(name="qwen3-32b-shape", L=64, H=64, KVH=8, B=32, lp=[1024] * 32, K=8192, r=64, gen=[32768] * 32,
                key_scale=False, dseed=4, eseed=4),
    }
    lp5 = synth.uniform_ints(5, 48, 256, 4096).tolist()
    gen5 = synth.uniform_ints(55, 48, 8192, 32768).tolist()
    w[5] = dict(name="phi-4-reasoning-shape ragged", L=40, H=40, KVH=10, B=48, lp=lp5, K=4096, r=64, gen=gen5,
                key_scale=False, dseed=5, eseed=5)
    return w


WORKLOADS = _workloads()
DEFAULT_CONFIG = 4         # the largest workload that fits one GPU (Qwen3-32B shape, ~78 GB of cache)
COMPARATOR_CONFIGS = (5,)  # workloads that also time the scored comparator on the same caches
POLICY_SNAPKV = 4
# order-preserving (the method's engine) / order-free in place / order-preserving inside the attention pass
COMPACTIONS = {"ordered": 0, "holefill": 1, "fused": 2}
WINDOW_STEP0 = 1 << 20     # synthetic step index of the first restored window query (row u: WINDOW_STEP0 + u)


def steady_state(w, rank=0):
    """Per-sequence (g0, c0) at steady state: phase = the steps since the sequence's last eviction,
    c0 = K + r + phase, positions the newest c0 generated ones.  The ragged workload draws every
    sequence's phase and progress; the equal-length ones spread the phases evenly over [0, r)
    (sequence b at b r / B), as requests that joined a continuous batch at different times, so
    that any window of steps holds eviction rounds in proportion to its length (about B / r
    sequences evict per step) instead of all sequences on one step every r."""
    K, r, B = w["K"], w["r"], w["B"]
    if w["B"] == 1 and w["L"] == 1:  # the small config starts empty (full run from step 0)
        return [0] * B, [0] * B
    ragged = len(set(w["lp"])) > 1
    g0, c0 = [], []
    for b in range(B):
        if ragged:
            phase = int(synth.uniform_ints(1000 + b, 1, 0, r - 1)[0])
            lo_epochs = -(-(K + 2 * r) // r)
            hi_epochs = max((w["gen"][b] - 2048) // r, lo_epochs)
            ep = int(synth.uniform_ints(2000 + b, 1, lo_epochs, hi_epochs)[0])
        else:  # last eviction at a step of at least K + 2r (the first one possible), mid-generation
            phase, ep = (b * r) // B, max(8192, -(-(K + 2 * r) // r) * r) // r
        ge = ep * r
        g0.append(ge + phase)
        c0.append(K + r + phase)
    return g0, c0


def describe(w):
    lp = w["lp"]
    lp_s = str(lp[0]) if len(set(lp)) == 1 else f"U[256,4096] (mean {np.mean(lp):.0f})"
    return (f"{w['name']}: {w['L']} layers, {w['H']}q/{w['KVH']}kv heads, d=128, batch {w['B']}, prompt {lp_s}, "
            f"K={w['K']}, r={w['r']}")


def decode_call(ra, ctx, calls, q, k, v, out, stream):
    """One decode step through the public API: ra_decode_step over the stacked layers, or
    ra_decode_layer for layers 0 .. L-1 in order (q, k, v, out: [L][...] device tensors)."""
    if calls == "step":
        ra.ra_decode_step(ctx, q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), 0.0, stream)
    else:
        for l in range(q.shape[0]):
            ra.ra_decode_layer(ctx, l, q[l].data_ptr(), k[l].data_ptr(), v[l].data_ptr(), out[l].data_ptr(), 0.0, stream)


class Workload:
    """Device-side setup of one workload through the public API."""

    def __init__(self, cfg, rank=0, ring=4, policy=0, compaction=0, calls="step"):
        import torch

        import paper_2609_03430_gb300 as ra
        import synth.gpu as sg

        self.torch, self.ra, self.sg = torch, ra, sg
        self.calls = calls
        self.w = w = WORKLOADS[cfg]
        self.cfg = cfg
        self.L, self.H, self.KVH, self.B, self.K, self.r = w["L"], w["H"], w["KVH"], w["B"], w["K"], w["r"]
        self.G = self.H // self.KVH
        self.lp = w["lp"]
        self.dseed = w["dseed"] + 1000003 * rank
        self.eseed = w["eseed"] + (rank << 32)
        self.dev = torch.device("cuda", torch.cuda.current_device())
        self.stream = torch.cuda.current_stream()
        self.policy = policy
        self.cache = ra.RandomAttentionCache(self.L, self.H, self.KVH, D, self.lp, self.K, self.r, self.eseed,
                                             policy=policy, compaction=compaction)
        self.ctx = self.cache.ctx
        self.key_scale = None
        if w["key_scale"]:
            self.key_scale = torch.from_numpy(synth.key_channel_scale(self.dseed, self.L, self.KVH, D)).to(self.dev)
        self.g0, self.c0 = steady_state(w, rank)
        self._fill()
        if policy == POLICY_SNAPKV:
            self._fill_window()
        self.ring = ring
        self._make_inputs(ring)

    def _scale(self, l):
        return None if self.key_scale is None else self.key_scale[l].contiguous()

    def _fill(self):
        torch = self.torch
        B, KVH = self.B, self.KVH
        maxlp = max(max(self.lp), 1)
        ppos = torch.full((B, KVH, maxlp), -1, dtype=torch.int32)
        for b in range(B):
            ppos[b, :, : self.lp[b]] = torch.arange(self.lp[b], dtype=torch.int32)
        ppos = ppos.to(self.dev)
        maxc = max(max(self.c0), 1)
        gpos = torch.full((B, KVH, maxc), -1, dtype=torch.int32)
        for b in range(B):
            c, g = self.c0[b], self.g0[b]
            gpos[b, :, :c] = torch.arange(self.lp[b] + g - c, self.lp[b] + g, dtype=torch.int32)
        gpos = gpos.to(self.dev)
        kp = torch.empty((B, KVH, maxlp, D), dtype=torch.int16, device=self.dev)
        vp = torch.empty_like(kp)
        kg = torch.empty((B, KVH, maxc, D), dtype=torch.int16, device=self.dev)
        vg = torch.empty_like(kg)
        for l in range(self.L):
            self.sg.fill_rows(kp, ppos, self.dseed, 0, l, 0, self._scale(l))
            self.sg.fill_rows(vp, ppos, self.dseed, 1, l, 0)
            self.ra.ra_prefill(self.ctx, l, kp.data_ptr(), vp.data_ptr(), maxlp)
            if max(self.c0) > 0:
                self.sg.fill_rows(kg, gpos, self.dseed, 0, l, 0, self._scale(l))
                self.sg.fill_rows(vg, gpos, self.dseed, 1, l, 0)
                self.ra.ra_restore(self.ctx, l, self.g0, self.c0, gpos.data_ptr(), kg.data_ptr(), vg.data_ptr(), maxc)
        torch.cuda.synchronize()
        del kp, vp, kg, vg

    def _fill_window(self):
        """Scored policy: the window of the r steps before the start, synthetic queries (row u of every
        (seq, query head) is the generator's query for step index WINDOW_STEP0 + u)."""
        torch = self.torch
        B, H, r = self.B, self.H, self.r
        pos = (WINDOW_STEP0 + torch.arange(r, dtype=torch.int32)).repeat(B, H, 1).contiguous().to(self.dev)
        qw = torch.empty((B, H, r, D), dtype=torch.int16, device=self.dev)
        for l in range(self.L):
            self.sg.fill_rows(qw, pos, self.dseed, 2, l, 0)
            self.ra.ra_restore_queries(self.ctx, l, qw.data_ptr())
        torch.cuda.synchronize()
        del qw

    def evictions(self):
        """Eviction rounds so far, summed over (sequence, layer)."""
        return sum(self.ra.ra_get_counters(self.ctx, b, l)[2] for b in range(self.B) for l in range(self.L))

    def _make_inputs(self, ring):
        """Device-resident inputs of `ring` distinct steps (cycled): q [L][B][H][d], k/v [L][B][KVH][d]."""
        torch = self.torch
        L, B, H, KVH = self.L, self.B, self.H, self.KVH
        self.q = torch.empty((ring, L, B, H, D), dtype=torch.int16, device=self.dev)
        self.kn = torch.empty((ring, L, B, KVH, D), dtype=torch.int16, device=self.dev)
        self.vn = torch.empty_like(self.kn)
        self.out = torch.empty((L, B, H, D), dtype=torch.int16, device=self.dev)
        for t in range(ring):
            qpos = torch.full((B, H, 1), t, dtype=torch.int32, device=self.dev)
            npos = torch.tensor([[self.lp[b] + self.g0[b] + t] * KVH for b in range(B)], dtype=torch.int32,
                                device=self.dev).reshape(B, KVH, 1)
            for l in range(L):
                self.sg.fill_rows(self.q[t, l].view(B, H, 1, D), qpos, self.dseed, 2, l, 0)
                self.sg.fill_rows(self.kn[t, l].view(B, KVH, 1, D), npos, self.dseed, 0, l, 0, self._scale(l))
                self.sg.fill_rows(self.vn[t, l].view(B, KVH, 1, D), npos, self.dseed, 1, l, 0)
        torch.cuda.synchronize()

    def step(self, t):
        i = t % self.ring
        decode_call(self.ra, self.ctx, self.calls, self.q[i], self.kn[i], self.vn[i], self.out, self.stream)

    def bytes_per_step(self):
        """Algorithmic cache bytes read by attention in one step (all layers), at the current state."""
        tot = 0
        for b in range(self.B):
            _, c, _ = self.ra.ra_get_counters(self.ctx, b, 0)
            tot += self.KVH * (self.lp[b] + c) * 2 * D * 2
        return tot * self.L


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons (started before, stopped after)."""

    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0, t1):
        rows = []
        for ts, line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            rows.append((ts, parts))
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["clock samples unavailable"]}
        inside = [p for ts, p in rows if t0 <= ts <= t1 + 0.15] or [p for ts, p in rows]
        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(p[2]) for p in inside if num(p[2]) is not None]
        mx = [num(p[3]) for p in inside if num(p[3]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for p in inside for i in range(4) if p[6 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(inside)}


def profiled_traffic(cfg):
    """DRAM bytes per attention launch from the committed ncu record, if it was taken on the
    current kernel source for this workload's layer shape; else None."""
    import hashlib

    try:
        with open(os.path.join(ROOT, "profiles", "attn_kernel_traffic.json")) as f:
            rec = json.load(f)
        src = os.path.join(ROOT, "paper_2609_03430_gb300", "csrc", "ra_attn.cu")
        digest = hashlib.sha256(open(src, "rb").read()).hexdigest()
        if rec.get("kernel_source_sha256") != digest:
            return None
        per_cfg = rec.get("traffic_bytes_per_launch", {})
        return per_cfg.get(str(cfg))
    except Exception:
        return None


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


def dist_env():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("LOCAL_RANK", "0"))


def reduce_over_ranks(ms, units, world):
    """max of per-rank times, sum of per-rank units (barrier implied by the collectives)."""
    if world == 1:
        return ms, units
    import torch
    import torch.distributed as dist

    dev = torch.device("cuda", torch.cuda.current_device()) if dist.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([ms], dtype=torch.float64, device=dev)
    u = torch.tensor([units], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u.item())


# --------------------------------------------------------------------------- CPU oracle timing
def oracle_sample(w, budget_s=12.0, rank=0):
    """Time the oracle (single-threaded C, fp64) on a bounded slice of the workload: attention for
    every KV head of one (sequence, layer) at its steady-state length plus one eviction round per
    head; extrapolated to tokens/s of the full layer stack.  Inputs are generated before timing."""
    import oracle

    oracle.build()
    g0, c0 = steady_state(w, rank)
    b = 0
    lp, K, r, KVH, G = w["lp"][b], w["K"], w["r"], w["KVH"], w["H"] // w["KVH"]
    c = max(c0[b], 1) + r // 2  # mean steady-state length between evictions
    g = max(g0[b], c)
    pos = np.concatenate([np.arange(lp), lp + g - c + np.arange(c)])
    heads = []
    for h in range(KVH):
        heads.append((synth.q_rows(w["dseed"], 0, b, np.arange(h * G, (h + 1) * G), 0, D),
                      synth.kv_rows(w["dseed"], 0, 0, b, h, pos, D), synth.kv_rows(w["dseed"], 1, 0, b, h, pos, D)))
    gen = (lp + np.arange(K + 2 * r)).astype(np.int32)
    t_attn, n_attn, t_ev, n_ev = 0.0, 0, 0.0, 0
    t_start = time.perf_counter()
    while time.perf_counter() - t_start < budget_s or n_attn == 0:
        for (q, kk, vv) in heads:
            t0 = time.perf_counter()
            oracle.attend(q, kk, vv)
            t_attn += time.perf_counter() - t0
            n_attn += 1
        for h in range(KVH):
            t0 = time.perf_counter()
            oracle.evict_head(gen, 8192, K, r, w["eseed"], 0, h)
            t_ev += time.perf_counter() - t0
            n_ev += 1
    per_head_step = t_attn / n_attn + (t_ev / n_ev) / r  # eviction every r steps
    per_token = per_head_step * KVH * w["L"]
    return {"value": 1.0 / per_token, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": (f"seq 0 of {describe(w)}: {n_attn} KV-head attention passes at length {lp + c} "
                       f"(fp64, G={G}) and {n_ev} eviction rounds of {K + r} candidates, "
                       f"{time.perf_counter() - t_start:.1f} s single-threaded; extrapolated x{KVH} heads x "
                       f"{w['L']} layers per token, eviction amortised over r={r} steps"),
            "nproc": os.cpu_count()}


def run_reference(args, w):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    per_step = []
    total = args.cpu_seconds if args.cpu_seconds_set else 60.0
    budget = max(0.05, min(10.0, total / max(1, args.steps + args.warmup)))
    res = None
    for i in range(args.warmup + args.steps):
        res = oracle_sample(w, budget_s=budget)
        if i >= args.warmup:
            per_step.append(1.0 / res["value"])
    ms = 1000.0 * statistics.mean(per_step)
    value = 1.0 / statistics.mean(per_step)
    cpu = dict(res)
    cpu["value"] = value
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_dict(w, args), "cpu_baseline": cpu,
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def config_dict(w, args):
    return {"workload": describe(w), "config_index": args.config, "batch": w["B"], "layers": w["L"],
            "q_heads": w["H"], "kv_heads": w["KVH"], "head_dim": D, "K": w["K"], "r": w["r"],
            "prompt_mean": float(np.mean(w["lp"])), "start": "steady state: K + r + phase cached generated rows per head, phase = steps since the "
                      "sequence's last eviction (spread evenly over [0, r) for equal-length batches, drawn "
                      "for the ragged one)",
            "l2": "inputs larger than L2 (every step streams the whole cache)", "parallelism": f"replicas x{args.gpus}",
            "policy": getattr(args, "policy", "random"), "compaction": getattr(args, "compaction", "ordered"),
            "calls": "ra_decode_layer per layer" if getattr(args, "calls", "step") == "layer" else "ra_decode_step"}


# --------------------------------------------------------------------------- GPU run
def timed_steps(wl, steps, t_next, barrier):
    """Device time per step of `steps` whole-stack decode steps: CUDA events on the stream only at
    its ends (no per-kernel events, which would break the overlap of consecutive launches)."""
    import torch

    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    wall0 = time.time()
    e0.record(wl.stream)
    for t in range(t_next, t_next + steps):
        wl.step(t)
    e1.record(wl.stream)
    barrier()
    wall1 = time.time()
    return e0.elapsed_time(e1) / steps, t_next + steps, wall0, wall1


def evented_steps(wl, steps, t_next):
    """The same number of steps again with CUDA events around every launch (on the launching
    stream): per-kernel durations and algorithmic bytes, and the eviction rounds they covered."""
    import torch

    ra = wl.ra
    rounds0 = wl.evictions()
    ra.ra_profile_reset(wl.ctx)
    ra.ra_profile_enable(wl.ctx, True)
    for t in range(t_next, t_next + steps):
        wl.step(t)
    torch.cuda.synchronize()
    ra.ra_profile_enable(wl.ctx, False)
    kern = {}
    for kind, name in enumerate(ra.KERNEL_NAMES):
        kms, n, by = ra.ra_profile_read(wl.ctx, kind)
        if n:
            kern[name] = {"launches": n, "ms_total": kms, "us_per_launch": 1000.0 * kms / n,
                          "bytes_per_launch": by / n,
                          "algorithmic_GBps": (by / (kms * 1e-3) / 1e9) if kms > 0 else None}
    ra.ra_check_device(wl.ctx)
    return kern, wl.evictions() - rounds0, t_next + steps


def attention_window(wl, steps, t_next):
    """Attention launch duration as the timed region runs it: `steps` more whole-stack steps with
    CUDA events only at the step boundaries (on the launching stream), so the launches inside a
    step keep the overlap they have in the timed region.  A step in which no sequence evicts
    launches nothing but the attention kernel of every layer; those steps give the duration
    (their device time / their attention launches) and bytes (the library's algorithmic count)."""
    import torch

    ra = wl.ra
    kind = ra.KERNEL_NAMES.index("attn")

    def evictions_layer0():  # the host mirror's counts; every layer of a sequence evicts on the same step
        return sum(ra.ra_get_counters(wl.ctx, b, 0)[2] for b in range(wl.B))

    ev_kinds = [ra.KERNEL_NAMES.index(n) for n in EVICT_KINDS if n in ra.KERNEL_NAMES]

    def evict_bytes():  # algorithmic bytes of the eviction launches so far (library count)
        return sum(ra.ra_profile_read(wl.ctx, k)[2] for k in ev_kinds)

    # (host bookkeeping between steps stays light -- a few calls -- so that the host keeps ahead of
    # the device; every layer of a sequence evicts on the same step, so rounds = sequences x layers)
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    marks = []
    evs[0].record(wl.stream)
    n0, e0 = evictions_layer0(), evict_bytes()
    _, l0, b0 = ra.ra_profile_read(wl.ctx, kind)
    for i, t in enumerate(range(t_next, t_next + steps)):
        wl.step(t)
        evs[i + 1].record(wl.stream)
        n1, e1 = evictions_layer0(), evict_bytes()
        _, l1, b1 = ra.ra_profile_read(wl.ctx, kind)
        marks.append((n1 != n0, l1 - l0, b1 - b0, (n1 - n0) * wl.L, e1 - e0))
        n0, e0, l0, b0 = n1, e1, l1, b1
    torch.cuda.synchronize()
    steps_ms = [(evs[i].elapsed_time(evs[i + 1]),) + m for i, m in enumerate(marks)]
    clean = [(ms, n, by) for (ms, fired, n, by, _, _) in steps_ms if not fired and n > 0]
    evicting = [(ms, by, rounds, eby) for (ms, fired, n, by, rounds, eby) in steps_ms if fired and n > 0]
    return clean, evicting, t_next + steps


def eviction_window(clean, evicting):
    """The eviction's cost on the critical path, measured in the step-boundary pass: a step in
    which sequences evict takes its attention time (its attention bytes at the eviction-free
    steps' attention bandwidth) plus what the eviction adds; that difference, over the steps'
    (sequence, layer) rounds and eviction bytes.  It includes what overlaps: the eviction's row
    loads start under programmatic dependent launch during the previous attention's tail."""
    if not clean or not evicting:
        return None
    attn_ms_per_byte = sum(c[0] for c in clean) / sum(c[2] for c in clean)
    extra_ms = sum(ms - by * attn_ms_per_byte for (ms, by, _, _) in evicting)
    rounds = sum(e[2] for e in evicting)
    ebytes = sum(e[3] for e in evicting)
    if rounds <= 0:
        return None
    # the prediction's own noise: the clean steps' spread of time per byte, over the evicting
    # steps' attention bytes; a difference within twice that is not resolved
    rates = [c[0] / c[2] for c in clean if c[2] > 0]
    mean = sum(rates) / len(rates)
    sd = (sum((x - mean) ** 2 for x in rates) / len(rates)) ** 0.5
    noise_ms = sd * sum(by * by for (_, by, _, _) in evicting) ** 0.5
    out = {"steps": len(evicting), "rounds": rounds, "bytes_per_round": ebytes / rounds,
           "noise_us_per_round": 1000.0 * noise_ms / rounds}
    if extra_ms <= 2.0 * noise_ms:
        return dict(out, resolved=False, us_per_round_at_most=1000.0 * (max(extra_ms, 0.0) + 2.0 * noise_ms) / rounds)
    return dict(out, resolved=True, us_per_round=1000.0 * extra_ms / rounds, GBps=ebytes / (extra_ms * 1e-3) / 1e9)


def attention_roofline(a, clean, steps, layers, peaks, peak_src, traffic):
    """The bench line's roofline of the attention kernel.  a: its per-launch-event totals (the
    serialized measurement); clean: (device ms, launches, algorithmic bytes) of the eviction-free
    steps of the step-boundary pass.  The duration is the windowed one when such steps exist, else
    the serialized one; achieved = algorithmic bytes per launch / duration."""
    if not a:
        return None
    serialized = {"us_per_launch": a["us_per_launch"], "achieved": a["algorithmic_GBps"],
                  "frac": a["algorithmic_GBps"] / peaks["hbm_gbs"],
                  "timing": "CUDA events around every attention launch on its stream, in a second pass "
                            "of the same number of steps (the events between launches defeat their "
                            "overlap, so this duration is an upper bound)"}
    if clean:
        win_ms = sum(c[0] for c in clean)
        win_n = sum(c[1] for c in clean)
        by_launch = sum(c[2] for c in clean) / win_n
        us_launch = 1000.0 * win_ms / win_n
        timing = (f"CUDA events at the step boundaries on the launching stream, over the {len(clean)} of "
                  f"{steps} steps of a third pass in which no sequence evicts: such a step launches "
                  f"only the {layers} layers' attention kernels, overlapped as in the timed region; "
                  f"duration = their device time / {win_n} launches")
    else:  # every step evicts somewhere (ragged phases): the per-launch events are all there is
        by_launch, us_launch, timing = a["bytes_per_launch"], a["us_per_launch"], serialized["timing"]
    achieved = by_launch / (us_launch * 1e-6) / 1e9
    return {"kernel": "attn_kernel (split-K decode attention)", "bound": "hbm", "target": TARGET, "achieved": achieved,
            "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
            "peak_source": f"{peak_src} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured"
            else "fallback 6.8 TB/s", "frac_of_nominal_8TBps": achieved / 8000.0,
            "algorithmic_bytes_per_launch": by_launch, "us_per_launch": us_launch,
            "traffic": traffic, "timing": timing, "serialized": serialized}


EVICT_KINDS = ("score_stats", "score_sum", "select", "compact", "evict", "stack")
EVICT_KERNELS = {  # the copy kernel priced by the eviction roofline, in order of preference
    "stack": "compact_stack_kernel (every layer's order-preserving compaction of the sequences firing at a "
             "step, in place, one launch per step, from evicted sets computed a step ahead)",
    "evict": "evict_kernel (selection and order-preserving compaction of one layer's round, one cluster per head)",
    "compact": "compact_kernel (order-preserving compaction of one layer's round)",
}
TARGET = ("the >= 0.70-of-HBM-bandwidth target is judged on frac, against the measured copy bandwidth; "
          "frac_of_nominal_8TBps is the same achieved figure over the nominal 8 TB/s")


STACK_FILL = ("fill_stack_kernel (every layer's order-free refill of the m evicted slots per head of the sequences "
              "firing at a step, in place, one launch per step, from evicted sets computed a step ahead)")


def eviction_roofline(kern, rounds, peaks, peak_src, traffic=None, holefill=None, windowed=None,
                      compaction="ordered"):
    """The bench line's roofline of the eviction: its copy kernel (the fused select + compaction
    kernel when the library ran it, else the compaction kernel) at its algorithmic bytes -- the
    survivors' K, V and position read and written, 2 (2 d 2 + 4) bytes per row -- over its
    per-launch CUDA-event duration, and the whole round (every eviction kernel's time per
    (sequence, layer) round).  holefill: (kernels, rounds) of the order-free run, whose select
    kernel moves the m refilled rows itself."""
    name = next((n for n in EVICT_KERNELS if n in kern and kern[n]["ms_total"]), None)
    if name is None or not rounds:
        return None
    k = kern[name]
    achieved = k["bytes_per_launch"] / (k["us_per_launch"] * 1e-6) / 1e9
    round_ms = sum(kern[n]["ms_total"] for n in EVICT_KINDS if n in kern)
    round_bytes = sum(kern[n]["bytes_per_launch"] * kern[n]["launches"] for n in EVICT_KINDS if n in kern)
    label = STACK_FILL if (name == "stack" and compaction == "holefill") else EVICT_KERNELS[name]
    out = {"kernel": label, "bound": "hbm", "target": TARGET, "achieved": achieved,
           "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
           "peak_source": f"{peak_src} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured"
           else "fallback 6.8 TB/s", "frac_of_nominal_8TBps": achieved / 8000.0,
           "algorithmic_bytes_per_launch": k["bytes_per_launch"], "us_per_launch": k["us_per_launch"],
           "launches": k["launches"], "traffic": traffic,
           "timing": "CUDA events around every eviction launch on its stream, in a second pass of the same "
                     "number of steps (events between launches defeat programmatic dependent launch, so "
                     "the duration includes the launch's own start-up)",
           "round": {"rounds": rounds, "us_per_round": 1000.0 * round_ms / rounds,
                     "bytes_per_round": round_bytes / rounds,
                     "frac": (round_bytes / (round_ms * 1e-3) / 1e9 / peaks["hbm_gbs"]) if round_ms else None,
                     "what": "every eviction kernel's evented time and algorithmic bytes per (sequence, layer) "
                             "round"}}
    for other in EVICT_KERNELS:  # the other copy kernels that ran (first eviction step, per-layer forms)
        o = kern.get(other)
        if other != name and o and o["ms_total"]:
            out.setdefault("also", {})[other] = {
                "launches": o["launches"], "us_per_launch": o["us_per_launch"],
                "achieved": o["bytes_per_launch"] / (o["us_per_launch"] * 1e-6) / 1e9,
                "frac": o["bytes_per_launch"] / (o["us_per_launch"] * 1e-6) / 1e9 / peaks["hbm_gbs"]}
    if "plan" in kern and kern["plan"]["ms_total"]:
        out["plan"] = {"launches": kern["plan"]["launches"], "us_per_launch": kern["plan"]["us_per_launch"],
                       "what": "plan_kernel: the next step's evicted sets, on a side stream beside the attention "
                               "(not on the critical path; not in the round figures)"}
    if windowed is not None:
        out["windowed"] = dict(windowed, frac=windowed["GBps"] / peaks["hbm_gbs"] if windowed.get("GBps") else None,
                               what="step-boundary pass: (device time of the steps in which sequences evict - their "
                                    "attention bytes at the eviction-free steps' attention bandwidth) per (sequence, "
                                    "layer) round; the eviction's cost on the critical path, overlap included")
    if holefill is not None:
        hk, hr = holefill
        what = {"stack": "order-free compaction, whole-stack step: fill_stack_kernel refills every layer's m "
                         "evicted slots per head in place, 2 m (2 d 2 + 4) bytes per head, one launch per step",
                "select": "order-free compaction, per layer: the select kernel refills the m evicted slots in "
                          "place, 2 m (2 d 2 + 4) bytes per head"}
        for name, key in (("stack", "holefill_fill"), ("select", "holefill_select")):
            k = hk.get(name)
            if k and hr and k["ms_total"]:
                out[key] = {
                    "launches": k["launches"], "us_per_launch": k["us_per_launch"],
                    "bytes_per_launch": k["bytes_per_launch"],
                    "achieved": k["bytes_per_launch"] / (k["us_per_launch"] * 1e-6) / 1e9,
                    "frac": k["bytes_per_launch"] / (k["us_per_launch"] * 1e-6) / 1e9 / peaks["hbm_gbs"],
                    "us_per_round": 1000.0 * k["ms_total"] / hr, "what": what[name]}
    return out


def _eviction_us_per_round(kern, names, rounds):
    if not rounds:
        return None
    return 1000.0 * sum(kern[n]["ms_total"] for n in names if n in kern) / rounds


def run_comparator(args, rank, world, barrier, peaks, random_ms, random_kern, random_rounds):
    """The scored comparator (SnapKV-style window top-K, prompt pinned) on the same caches: the
    workload rebuilt from the same seeds with the scored policy and a restored query window,
    timed like the main run; per-round cost of its eviction kernels next to the random policy's."""
    wl = Workload(args.config, rank=rank, policy=POLICY_SNAPKV)
    for t in range(args.warmup):
        wl.step(t)
    wl.ra.ra_check_device(wl.ctx)
    ms, t_next, _, _ = timed_steps(wl, args.steps, args.warmup, barrier)
    kern, rounds, _ = evented_steps(wl, args.steps, t_next)
    ms_step, units = reduce_over_ranks(ms, float(wl.B), world)
    M = wl.r * wl.G
    score = {}
    for name in ("score_stats", "score_sum"):
        k = kern.get(name)
        if k and k["ms_total"] > 0:
            # algorithmic bytes of these kinds are the key rows read; each costs 2 * M * 128 flops
            tflops = k["bytes_per_launch"] * M / (k["us_per_launch"] * 1e-6) / 1e12
            score[name] = dict(k, tensor_TFLOPs=tflops, bound="tensor",
                               frac_of_bf16_peak=tflops / peaks["bf16_tflops"])
    wl.cache.close()
    return {"policy": "snapkv-style window top-K: window = the last r queries, scores summed over the "
                      "query heads of the group, max-pool width 7, prompt pinned, r-token buffer unscored",
            "value": units / (ms_step * 1e-3), "unit": UNIT, "ms_per_step": ms_step,
            "step_time_vs_random": ms_step / random_ms,
            "rounds_in_evented_pass": {"random": random_rounds, "snapkv": rounds},
            "eviction_us_per_round": {
                "random": _eviction_us_per_round(random_kern, EVICT_KINDS, random_rounds),
                "snapkv": _eviction_us_per_round(kern, EVICT_KINDS, rounds),
                "what": "evented kernel time of a step's eviction launches / (sequence, layer) rounds they ran"},
            "score_kernels": score, "kernels": kern}


def run_holefill_variant(args, rank, world, barrier, peaks, ordered_ms, ordered_kern, ordered_rounds):
    """Order-free (hole-filling) compaction on the same caches: the workload rebuilt from the same
    seeds with the evicted slots refilled in place, timed like the main run."""
    wl = Workload(args.config, rank=rank, compaction=COMPACTIONS["holefill"])
    for t in range(args.warmup):
        wl.step(t)
    wl.ra.ra_check_device(wl.ctx)
    cache_bytes = wl.bytes_per_step()
    ms, t_next, _, _ = timed_steps(wl, args.steps, args.warmup, barrier)
    kern, rounds, _ = evented_steps(wl, args.steps, t_next)
    ms_step, units = reduce_over_ranks(ms, float(wl.B), world)
    wl.cache.close()
    return {"compaction": "order-free: keys per position, evicted slots refilled in place from the newest "
                          "ones (one fill launch per eviction step from evicted sets computed a step ahead; "
                          "the select kernel where none was computed)",
            "value": units / (ms_step * 1e-3), "unit": UNIT, "ms_per_step": ms_step,
            "step_time_vs_ordered": ms_step / ordered_ms,
            "step_effective_frac": cache_bytes / (ms_step * 1e-3) / 1e9 / peaks["hbm_gbs"],
            "eviction_us_per_round": {
                "ordered": _eviction_us_per_round(ordered_kern, EVICT_KINDS, ordered_rounds),
                "holefill": _eviction_us_per_round(kern, EVICT_KINDS, rounds),
                "what": "evented kernel time of a step's eviction launches / (sequence, layer) rounds they ran"},
            "rounds_in_evented_pass": rounds, "kernels": kern}


def run_per_layer_variant(args, rank, world, barrier, stacked_ms):
    """The same step through the per-layer call a real model makes (ra_decode_layer for layers
    0 .. L-1 in order: layer 0's call opens the step), on the same caches rebuilt from the same
    seeds, timed like the main run."""
    wl = Workload(args.config, rank=rank, compaction=COMPACTIONS[args.compaction], calls="layer")
    for t in range(args.warmup):
        wl.step(t)
    wl.ra.ra_check_device(wl.ctx)
    ms, _, _, _ = timed_steps(wl, args.steps, args.warmup, barrier)
    ms_step, units = reduce_over_ranks(ms, float(wl.B), world)
    wl.cache.close()
    return {"calls": "ra_decode_layer per layer, in layer order", "value": units / (ms_step * 1e-3), "unit": UNIT,
            "ms_per_step": ms_step, "step_time_vs_stacked": ms_step / stacked_ms}


def run_ours(args, w):
    import torch

    import paper_2609_03430_gb300 as ra

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    main_policy = POLICY_SNAPKV if args.policy == "snapkv" else 0
    wl = Workload(args.config, rank=rank, policy=main_policy, compaction=COMPACTIONS[args.compaction],
                  calls=args.calls)
    stream = wl.stream
    ctx = wl.ctx

    def barrier():
        if world > 1:
            import torch.distributed as dist

            dist.barrier()
        torch.cuda.synchronize()

    for t in range(args.warmup):
        wl.step(t)
    ra.ra_check_device(ctx)
    attn_bytes_before = wl.bytes_per_step()

    # Timed region: K whole-stack decode steps.
    ra.ra_profile_reset(ctx)
    clocks = ClockSampler(torch.cuda.current_device())
    clocks.start()
    time.sleep(0.3)
    ms, t_next, wall0, wall1 = timed_steps(wl, args.steps, args.warmup, barrier)
    clocks.stop()
    launches = sum(ra.ra_profile_read(ctx, kind)[1] for kind in range(len(ra.KERNEL_NAMES)))

    # Kernel durations: the same number of steps again with CUDA events around every launch ...
    kern, rounds, t_next = evented_steps(wl, args.steps, t_next)
    # ... and once more with events only at the step boundaries (attention launches overlapped).
    clean, evicting, t_next = attention_window(wl, args.steps, t_next)
    win_evict = eviction_window(clean, evicting)

    ms_step, units = reduce_over_ranks(ms, float(wl.B), world)
    value = units / (ms_step * 1e-3)

    # e2e: the same steps with host buffers -- H2D of each step's inputs from pinned memory,
    # ra_decode_step, D2H of its outputs, all inside the timed region.  The copies run on a second
    # stream into double-buffered device buffers, as a serving loop would issue them: step t + 1's
    # inputs upload while step t computes, and step t's outputs download while step t + 1 does.
    e2e = None
    if not args.no_e2e:
        hq = torch.empty(wl.q[0].shape, dtype=torch.int16).pin_memory()
        hk = torch.empty(wl.kn[0].shape, dtype=torch.int16).pin_memory()
        hv = torch.empty(wl.vn[0].shape, dtype=torch.int16).pin_memory()
        ho = [torch.empty(wl.out.shape, dtype=torch.int16).pin_memory() for _ in range(2)]
        hq.copy_(wl.q[0].cpu()); hk.copy_(wl.kn[0].cpu()); hv.copy_(wl.vn[0].cpu())
        dq = [torch.empty_like(wl.q[0]) for _ in range(2)]
        dk = [torch.empty_like(wl.kn[0]) for _ in range(2)]
        dv = [torch.empty_like(wl.vn[0]) for _ in range(2)]
        do = [torch.empty_like(wl.out) for _ in range(2)]
        cs = torch.cuda.Stream()
        ev = lambda: torch.cuda.Event()  # noqa: E731
        up, done, down = [ev(), ev()], [ev(), ev()], [ev(), ev()]

        def upload(i):
            dq[i].copy_(hq, non_blocking=True)
            dk[i].copy_(hk, non_blocking=True)
            dv[i].copy_(hv, non_blocking=True)
            up[i].record(cs)

        barrier()
        f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        f0.record(stream)
        cs.wait_event(f0)
        with torch.cuda.stream(cs):
            upload(0)
        for t in range(args.steps):
            i, j = t % 2, (t + 1) % 2
            if t + 1 < args.steps:
                with torch.cuda.stream(cs):
                    if t >= 1:
                        cs.wait_event(done[j])  # buffer j's last user, step t - 1, has finished
                    upload(j)
            stream.wait_event(up[i])
            if t >= 2:
                stream.wait_event(down[i])  # step t - 2's outputs are read back from buffer i
            decode_call(ra, ctx, wl.calls, dq[i], dk[i], dv[i], do[i], stream)
            done[i].record(stream)
            with torch.cuda.stream(cs):
                cs.wait_event(done[i])
                ho[i].copy_(do[i], non_blocking=True)
                down[i].record(cs)
        stream.wait_event(down[(args.steps - 1) % 2])
        f1.record(stream)
        barrier()
        e2e_ms, e2e_units = reduce_over_ranks(f0.elapsed_time(f1) / args.steps, float(wl.B), world)
        e2e = {"value": e2e_units / (e2e_ms * 1e-3), "unit": UNIT,
               "h2d_bytes_per_step": int(hq.numel() * 2 + hk.numel() * 2 + hv.numel() * 2),
               "d2h_bytes_per_step": int(ho[0].numel() * 2), "ms_per_step": e2e_ms,
               "copies": "pinned host buffers; H2D and D2H on a second stream, double-buffered, "
                         "overlapped with the neighbouring steps' compute"}
        del hq, hk, hv, ho, dq, dk, dv, do
    wl.cache.close()
    del wl

    peaks, peak_src = measured_peaks()
    roof = attention_roofline(kern.get("attn"), clean, args.steps, w["L"], peaks, peak_src,
                              args.traffic if args.traffic is not None else profiled_traffic(args.config))
    comparator = None
    if main_policy == 0 and (args.comparator == "on" or
                             (args.comparator == "auto" and args.config in COMPARATOR_CONFIGS)):
        comparator = run_comparator(args, rank, world, barrier, peaks, ms_step, kern, rounds)
    holefill = None
    if main_policy == 0 and args.compaction == "ordered" and args.variants == "on":
        holefill = run_holefill_variant(args, rank, world, barrier, peaks, ms_step, kern, rounds)
    per_layer = None
    if main_policy == 0 and args.calls == "step" and args.variants == "on":
        per_layer = run_per_layer_variant(args, rank, world, barrier, ms_step)
    roof_evict = eviction_roofline(kern, rounds, peaks, peak_src, args.traffic_evict,
                                   (holefill["kernels"], holefill["rounds_in_evented_pass"]) if holefill else None,
                                   win_evict, args.compaction)
    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = oracle_sample(w, budget_s=args.cpu_seconds, rank=0)
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": config_dict(w, args),
                "roofline": roof, "roofline_evict": roof_evict, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches,
                "clocks": clocks.summary(wall0, wall1), "kernels": kern,
                "attn_cache_bytes_per_step": attn_bytes_before,
                "step_effective": {"GBps": attn_bytes_before / (ms_step * 1e-3) / 1e9,
                                   "frac": attn_bytes_before / (ms_step * 1e-3) / 1e9 / peaks["hbm_gbs"],
                                   "what": "cache bytes streamed per step / device time per step "
                                           "(all kernels of the step, launches overlapped)"}}
        if comparator is not None:
            line["comparator"] = comparator
        if holefill is not None:
            line["holefill_variant"] = holefill
        if per_layer is not None:
            line["per_layer_variant"] = per_layer
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=256)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--config", type=int, default=DEFAULT_CONFIG, choices=sorted(WORKLOADS))
    ap.add_argument("--calls", choices=["step", "layer"], default="step",
                    help="the public call a step goes through: ra_decode_step, or ra_decode_layer per layer")
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--layers", type=int, default=None,
                    help="override the layer count (only to shrink profiler captures; not a benchmark workload)")
    ap.add_argument("--policy", choices=["random", "snapkv"], default="random",
                    help="eviction policy of the timed run (random: the method; snapkv: the scored comparator)")
    ap.add_argument("--compaction", choices=sorted(COMPACTIONS), default="ordered",
                    help="eviction compaction of the timed run (holefill: order-free, in place)")
    ap.add_argument("--variants", choices=["on", "off"], default="on",
                    help="also time order-free (hole-filling) compaction on the same caches")
    ap.add_argument("--comparator", choices=["auto", "on", "off"], default="auto",
                    help="also time the scored comparator on the same caches (auto: the ragged workload)")
    ap.add_argument("--traffic", type=float, default=None,
                    help="ncu dram bytes per attention launch (from a committed profile), if current")
    ap.add_argument("--traffic-evict", type=float, default=None,
                    help="ncu dram bytes per eviction copy launch (from a committed profile), if current")
    args = ap.parse_args(argv)
    args.cpu_seconds_set = any(a.startswith("--cpu-seconds") for a in (argv if argv is not None else sys.argv[1:]))
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    w = WORKLOADS[args.config]
    if args.layers is not None:
        w = dict(w, L=args.layers, name=w["name"] + f" (truncated to {args.layers} layers for profiling)")
        WORKLOADS[args.config] = w
    if args.impl == "reference":
        return run_reference(args, w)
    return run_ours(args, w)


if __name__ == "__main__":
    sys.exit(main())
