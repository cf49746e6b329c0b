"""Parity at the full workload sizes, in the launch configuration bench.py times.

Each workload is set up exactly as the benchmark does (steady-state caches
filled on the device by the seeded generator, ``ra_decode_step`` over the whole
layer stack), then run for r + 2 steps, so that every sequence evicts once,
with step inputs generated for their true positions.  The oracle replays the
sampled heads from the same start state: their survivor positions and their
cached K/V bytes must match bit-exactly, and the last step's attention output
of sampled (sequence, layer, KV head) slices must be within tolerance of the
fp64 oracle.
"""
import numpy as np
import pytest

from conftest import cuda_available
from ra_testlib import check_attention

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]


def _samples(w, n_heads, n_attn, seed):
    rng = np.random.default_rng(seed)
    heads = {(int(rng.integers(w["B"])), int(rng.integers(w["L"])), int(rng.integers(w["KVH"])))
             for _ in range(n_heads)}
    heads |= {(0, 0, 0), (w["B"] - 1, w["L"] - 1, w["KVH"] - 1)}
    attn = sorted(heads)[:n_attn]
    return sorted(heads), attn


@pytest.mark.parametrize("cfg,compaction", [(2, 0), (3, 0), (4, 0), (5, 0), (4, 1), (5, 1)],
                         ids=["cfg2", "cfg3", "cfg4", "cfg5", "cfg4-holefill", "cfg5-holefill"])
def test_workload_parity_sampled(cfg, compaction):
    import torch

    import bench
    import oracle
    import paper_2609_03430_gb300 as ra
    import synth
    import synth.gpu as sg

    torch.cuda.set_device(0)
    wl = bench.Workload(cfg, ring=1, compaction=compaction)
    w = wl.w
    L, B, H, KVH, K, r, D = wl.L, wl.B, wl.H, wl.KVH, wl.K, wl.r, 128
    G = H // KVH
    heads, attn_heads = _samples(w, 64, 8, cfg)
    orc = oracle.OracleCache(L, KVH, wl.lp, K, r, wl.eseed, heads=heads, compaction=compaction)
    for (b, l, h) in heads:
        c, g = wl.c0[b], wl.g0[b]
        orc.gen[(b, l, h)] = np.arange(wl.lp[b] + g - c, wl.lp[b] + g, dtype=np.int32)
        orc.g[b, l] = g
    dev = wl.dev
    q = torch.empty((L, B, H, D), dtype=torch.int16, device=dev)
    kn = torch.empty((L, B, KVH, D), dtype=torch.int16, device=dev)
    vn = torch.empty_like(kn)
    out = torch.empty((L, B, H, D), dtype=torch.int16, device=dev)
    steps = r + 2
    for t in range(steps):
        qpos = torch.full((B, H, 1), t, dtype=torch.int32, device=dev)
        npos = torch.tensor([[wl.lp[b] + wl.g0[b] + t] * KVH for b in range(B)], dtype=torch.int32,
                            device=dev).reshape(B, KVH, 1)
        for l in range(L):
            sg.fill_rows(q[l].view(B, H, 1, D), qpos, wl.dseed, 2, l, 0)
            sg.fill_rows(kn[l].view(B, KVH, 1, D), npos, wl.dseed, 0, l, 0, wl._scale(l))
            sg.fill_rows(vn[l].view(B, KVH, 1, D), npos, wl.dseed, 1, l, 0)
        ra.ra_decode_step(wl.ctx, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), out.data_ptr(), 0.0)
        for (b, l) in sorted({(b, l) for (b, l, _) in heads}):
            orc.append(b, l)
            orc.evict(b, l)
    torch.cuda.synchronize()
    ra.ra_check_device(wl.ctx)
    fired = 0
    for (b, l, h) in heads:
        g, c, nev = ra.ra_get_counters(wl.ctx, b, l)
        assert g == orc.g[b, l] and c == orc.gen[(b, l, h)].size
        fired += nev > 0
        got = ra.ra_get_positions(wl.ctx, l, b, h, K + 2 * r)
        np.testing.assert_array_equal(got, orc.gen[(b, l, h)], err_msg=f"positions {(b, l, h)}")
    assert fired == len(heads)  # every sampled head evicted at least once
    sc_np = None if wl.key_scale is None else wl.key_scale.cpu().numpy()
    got_out = out.cpu().numpy()
    for (b, l, h) in attn_heads:
        pos = orc.positions(b, l, h)
        krow = synth.kv_rows(wl.dseed, 0, l, b, h, pos, D, None if sc_np is None else sc_np[l, h])
        vrow = synth.kv_rows(wl.dseed, 1, l, b, h, pos, D)
        kk, vv = ra.ra_get_kv(wl.ctx, l, b, h, wl.lp[b] + K + 2 * r)
        np.testing.assert_array_equal(kk, krow, err_msg=f"K rows {(b, l, h)}")
        np.testing.assert_array_equal(vv, vrow, err_msg=f"V rows {(b, l, h)}")
        qv = synth.q_rows(wl.dseed, l, b, np.arange(h * G, (h + 1) * G), steps - 1, D)
        ref = oracle.attend(qv, krow, vrow)
        check_attention(got_out[l, b, h * G:(h + 1) * G], ref, f"cfg {cfg} slice {(b, l, h)}")
    wl.cache.close()


def test_config2_every_head_index_replay():
    """Config 2 (the Qwen3-4B shape) at full size, every one of its 4 608 (sequence, layer, KV head)
    units: the oracle replays each head's rounds over r + 2 steps of the benchmark's launch
    configuration, and every head's surviving positions must match bit-exactly."""
    import torch

    import bench
    import oracle
    import paper_2609_03430_gb300 as ra
    import synth.gpu as sg

    torch.cuda.set_device(0)
    wl = bench.Workload(2, ring=1)
    L, B, H, KVH, K, r, D = wl.L, wl.B, wl.H, wl.KVH, wl.K, wl.r, 128
    orc = oracle.OracleCache(L, KVH, wl.lp, K, r, wl.eseed)
    for b in range(B):
        c, g = wl.c0[b], wl.g0[b]
        for l in range(L):
            for h in range(KVH):
                orc.gen[(b, l, h)] = np.arange(wl.lp[b] + g - c, wl.lp[b] + g, dtype=np.int32)
            orc.g[b, l] = g
    dev = wl.dev
    q = torch.empty((L, B, H, D), dtype=torch.int16, device=dev)
    kn = torch.empty((L, B, KVH, D), dtype=torch.int16, device=dev)
    vn = torch.empty_like(kn)
    out = torch.empty((L, B, H, D), dtype=torch.int16, device=dev)
    for t in range(r + 2):
        qpos = torch.full((B, H, 1), t, dtype=torch.int32, device=dev)
        npos = torch.tensor([[wl.lp[b] + wl.g0[b] + t] * KVH for b in range(B)], dtype=torch.int32,
                            device=dev).reshape(B, KVH, 1)
        for l in range(L):
            sg.fill_rows(q[l].view(B, H, 1, D), qpos, wl.dseed, 2, l, 0)
            sg.fill_rows(kn[l].view(B, KVH, 1, D), npos, wl.dseed, 0, l, 0, wl._scale(l))
            sg.fill_rows(vn[l].view(B, KVH, 1, D), npos, wl.dseed, 1, l, 0)
        ra.ra_decode_step(wl.ctx, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), out.data_ptr(), 0.0)
        for b in range(B):
            for l in range(L):
                orc.append(b, l)
                orc.evict(b, l)
    torch.cuda.synchronize()
    ra.ra_check_device(wl.ctx)
    for b in range(B):
        for l in range(L):
            g, c, nev = ra.ra_get_counters(wl.ctx, b, l)
            assert g == orc.g[b, l] and nev == 1  # every head evicted once in the window
            for h in range(KVH):
                got = ra.ra_get_positions(wl.ctx, l, b, h, K + 2 * r)
                np.testing.assert_array_equal(got, orc.gen[(b, l, h)], err_msg=f"positions {(b, l, h)}")
    wl.cache.close()


def test_scored_comparator_parity_full_size():
    """The scored comparator at the ragged workload's full size (the configuration bench.py times it
    in): query window restored, r + 2 steps so that every sequence scores once; sampled heads' raw
    scores within tolerance of the fp64 oracle, keep-sets equal to the oracle's round on the kernel's
    scores (fp64 disagreements only at the threshold), survivors and attention as for the method."""
    import torch

    import bench
    import oracle
    import paper_2609_03430_gb300 as ra
    import synth
    import synth.gpu as sg
    from ra_testlib import check_scored_decision, check_scores

    torch.cuda.set_device(0)
    cfg = 5
    wl = bench.Workload(cfg, ring=1, policy=bench.POLICY_SNAPKV)
    w = wl.w
    L, B, H, KVH, K, r, D = wl.L, wl.B, wl.H, wl.KVH, wl.K, wl.r, 128
    G = H // KVH
    heads, attn_heads = _samples(w, 10, 4, 77)
    orc = oracle.OracleCache(L, KVH, wl.lp, K, r, wl.eseed, heads=heads, policy=oracle.POLICY_SNAPKV)
    for (b, l, h) in heads:
        c, g = wl.c0[b], wl.g0[b]
        orc.gen[(b, l, h)] = np.arange(wl.lp[b] + g - c, wl.lp[b] + g, dtype=np.int32)
        orc.g[b, l] = g

    def step_index(b, s):  # generator step index of sequence b's 1-based decode step s
        g0 = wl.g0[b]
        return bench.WINDOW_STEP0 + s - (g0 - r + 1) if s <= g0 else s - g0 - 1

    rounds = [0]

    def scorer(b, l, h, cur):
        g, n = int(orc.g[b, l]), cur.size - r
        steps = range(g - r, g)
        qh = np.arange(h * G, (h + 1) * G)
        q = np.stack([synth.q_rows(wl.dseed, l, b, qh, step_index(b, s), D) for s in steps])
        qpos = np.array([wl.lp[b] + s - 1 for s in steps], dtype=np.int32)
        kpos = orc.positions(b, l, h)
        krow = synth.kv_rows(wl.dseed, 0, l, b, h, kpos, D)
        ref = oracle.window_scores(q, qpos, krow, kpos)[wl.lp[b]:wl.lp[b] + n]
        got = ra.ra_get_scores(wl.ctx, l, b, h, K + 2 * r)
        check_scores(got, ref, f"scores {(b, l, h)} g{g}")
        check_scored_decision(got, ref, K, f"decision {(b, l, h)} g{g}")
        rounds[0] += 1
        return got.astype(np.float64)

    dev = wl.dev
    q = torch.empty((L, B, H, D), dtype=torch.int16, device=dev)
    kn = torch.empty((L, B, KVH, D), dtype=torch.int16, device=dev)
    vn = torch.empty_like(kn)
    out = torch.empty((L, B, H, D), dtype=torch.int16, device=dev)
    steps = r + 2
    for t in range(steps):
        qpos = torch.full((B, H, 1), t, dtype=torch.int32, device=dev)
        npos = torch.tensor([[wl.lp[b] + wl.g0[b] + t] * KVH for b in range(B)], dtype=torch.int32,
                            device=dev).reshape(B, KVH, 1)
        for l in range(L):
            sg.fill_rows(q[l].view(B, H, 1, D), qpos, wl.dseed, 2, l, 0)
            sg.fill_rows(kn[l].view(B, KVH, 1, D), npos, wl.dseed, 0, l, 0)
            sg.fill_rows(vn[l].view(B, KVH, 1, D), npos, wl.dseed, 1, l, 0)
        ra.ra_decode_step(wl.ctx, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), out.data_ptr(), 0.0)
        torch.cuda.synchronize()
        for (b, l) in sorted({(b, l) for (b, l, _) in heads}):
            orc.append(b, l)
            orc.evict(b, l, scorer=scorer)
    ra.ra_check_device(wl.ctx)
    assert rounds[0] >= len(heads)  # every sampled head scored at least once
    for (b, l, h) in heads:
        got = ra.ra_get_positions(wl.ctx, l, b, h, K + 2 * r)
        np.testing.assert_array_equal(got, orc.gen[(b, l, h)], err_msg=f"positions {(b, l, h)}")
    got_out = out.cpu().numpy()
    for (b, l, h) in attn_heads:
        pos = orc.positions(b, l, h)
        kk, vv = ra.ra_get_kv(wl.ctx, l, b, h, wl.lp[b] + K + 2 * r)
        np.testing.assert_array_equal(kk, synth.kv_rows(wl.dseed, 0, l, b, h, pos, D), err_msg=f"K rows {(b, l, h)}")
        np.testing.assert_array_equal(vv, synth.kv_rows(wl.dseed, 1, l, b, h, pos, D), err_msg=f"V rows {(b, l, h)}")
        qv = synth.q_rows(wl.dseed, l, b, np.arange(h * G, (h + 1) * G), steps - 1, D)
        ref = oracle.attend(qv, synth.kv_rows(wl.dseed, 0, l, b, h, pos, D), synth.kv_rows(wl.dseed, 1, l, b, h, pos, D))
        check_attention(got_out[l, b, h * G:(h + 1) * G], ref, f"slice {(b, l, h)}")
    wl.cache.close()


def test_config2_full_length_sampled():
    """The Qwen3-4B-shape workload over its whole generation: the 32768 decode steps from an empty
    generated cache (prompts only), through the growth phase (no eviction until K + 2r tokens) and
    then an eviction round every r steps, about 480 rounds per (sequence, layer).  Step inputs come
    from the seeded generator for their true positions.  The oracle replays sampled heads through
    every round: survivor positions and cached K/V bytes bit-exact, and the last step's attention of
    sampled slices within tolerance of the fp64 oracle."""
    import torch

    import bench
    import oracle
    import paper_2609_03430_gb300 as ra
    import synth
    import synth.gpu as sg

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    w = bench.WORKLOADS[2]
    L, H, KVH, B, K, r, D = w["L"], w["H"], w["KVH"], w["B"], w["K"], w["r"], 128
    G = H // KVH
    lp, steps = w["lp"], w["gen"][0]
    dseed, eseed = w["dseed"], w["eseed"]
    cache = ra.RandomAttentionCache(L, H, KVH, D, lp, K, r, eseed)
    ctx = cache.ctx
    key_scale = torch.from_numpy(synth.key_channel_scale(dseed, L, KVH, D)).to(dev)
    maxlp = max(lp)
    ppos = torch.tensor([[list(range(lp[b])) + [-1] * (maxlp - lp[b])] * KVH for b in range(B)],
                        dtype=torch.int32, device=dev)
    kp = torch.empty((B, KVH, maxlp, D), dtype=torch.int16, device=dev)
    vp = torch.empty_like(kp)
    for l in range(L):
        sg.fill_rows(kp, ppos, dseed, 0, l, 0, key_scale[l].contiguous())
        sg.fill_rows(vp, ppos, dseed, 1, l, 0)
        ra.ra_prefill(ctx, l, kp.data_ptr(), vp.data_ptr(), maxlp)
    del kp, vp

    heads, attn_heads = _samples(w, 8, 4, 202)
    orc = oracle.OracleCache(L, KVH, lp, K, r, eseed, heads=heads)
    pairs = sorted({(b, l) for (b, l, _) in heads})
    CH = 64  # steps whose inputs are generated at once
    qch = torch.empty((L, B, H, CH, D), dtype=torch.int16, device=dev)
    kch = torch.empty((L, B, KVH, CH, D), dtype=torch.int16, device=dev)
    vch = torch.empty_like(kch)
    q = torch.empty((L, B, H, D), dtype=torch.int16, device=dev)
    kn = torch.empty((L, B, KVH, D), dtype=torch.int16, device=dev)
    vn = torch.empty_like(kn)
    out = torch.empty((L, B, H, D), dtype=torch.int16, device=dev)
    lp_t = torch.tensor(lp, dtype=torch.int32, device=dev).view(B, 1, 1)
    for t0 in range(0, steps, CH):
        ar = torch.arange(t0, t0 + CH, dtype=torch.int32, device=dev).view(1, 1, CH)
        npos = (lp_t + ar).expand(B, KVH, CH).contiguous()
        qpos = ar.expand(B, H, CH).contiguous()
        for l in range(L):
            sg.fill_rows(qch[l], qpos, dseed, 2, l, 0)
            sg.fill_rows(kch[l], npos, dseed, 0, l, 0, key_scale[l].contiguous())
            sg.fill_rows(vch[l], npos, dseed, 1, l, 0)
        for i in range(min(CH, steps - t0)):
            q.copy_(qch[:, :, :, i, :])
            kn.copy_(kch[:, :, :, i, :])
            vn.copy_(vch[:, :, :, i, :])
            ra.ra_decode_step(ctx, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), out.data_ptr(), 0.0)
            for (b, l) in pairs:
                orc.append(b, l)
                orc.evict(b, l)
    torch.cuda.synchronize()
    ra.ra_check_device(ctx)
    rounds = (steps - (K + 2 * r)) // r + 1
    for (b, l, h) in heads:
        g, c, nev = ra.ra_get_counters(ctx, b, l)
        assert g == steps == orc.g[b, l] and c == orc.gen[(b, l, h)].size
        assert nev == orc.n_evictions[b, l] == rounds
        got = ra.ra_get_positions(ctx, l, b, h, K + 2 * r)
        np.testing.assert_array_equal(got, orc.gen[(b, l, h)], err_msg=f"positions {(b, l, h)}")
    sc_np = key_scale.cpu().numpy()
    got_out = out.cpu().numpy()
    for (b, l, h) in attn_heads:
        pos = orc.positions(b, l, h)
        krow = synth.kv_rows(dseed, 0, l, b, h, pos, D, sc_np[l, h])
        vrow = synth.kv_rows(dseed, 1, l, b, h, pos, D)
        kk, vv = ra.ra_get_kv(ctx, l, b, h, lp[b] + K + 2 * r)
        np.testing.assert_array_equal(kk, krow, err_msg=f"K rows {(b, l, h)}")
        np.testing.assert_array_equal(vv, vrow, err_msg=f"V rows {(b, l, h)}")
        qv = synth.q_rows(dseed, l, b, np.arange(h * G, (h + 1) * G), steps - 1, D)
        check_attention(got_out[l, b, h * G:(h + 1) * G], oracle.attend(qv, krow, vrow), f"full length slice {(b, l, h)}")
    cache.close()
