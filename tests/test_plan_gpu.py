"""Evicted sets computed one step ahead (ra_decode_step): the random draw needs no cache data but
positions, so while a step's attention runs, a kernel on a side stream computes the next step's
evicted sets, and at the firing step one launch moves every layer's rows.  Checked against the
oracle, bit-exact, over several rounds with sequences firing on different steps, in both layouts:
- ordered (order-preserving compaction, in place): random, shared draw, protected recency (the
  exact radix passes), the exact passes forced for the random draw, block draws of 16 positions
  (keys read positions; ties resolved by the radix sweep);
- order-free (the evicted slots refilled from the newest rows, the step's token included): keys
  per position for random, shared, recency and block draws.
Attention of the last step within tolerance.
"""
import numpy as np
import pytest

from conftest import cuda_available
from ra_testlib import Runner, check_attention

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]


def _restore_phased(run, phases, epoch):
    """Sequence b: last eviction at step epoch * r, then phases[b] appends (K + r + phase cached)."""
    import paper_2609_03430_gb300 as ra

    cmax = run.K + run.r + max(phases)
    for l in range(run.L):
        pos = np.full((run.B, run.KVH, cmax), -1, np.int32)
        kk = np.zeros((run.B, run.KVH, cmax, run.D), np.uint16)
        vv = np.zeros_like(kk)
        gs, cs = [], []
        for b in range(run.B):
            g = epoch * run.r + phases[b]
            c = run.K + run.r + phases[b]
            p = run.lp[b] + np.arange(g - c, g)
            for h in range(run.KVH):
                pos[b, h, :c] = p
                kk[b, h, :c] = run.krows(l, b, h, p)
                vv[b, h, :c] = run.vrows(l, b, h, p)
                run.orc.gen[(b, l, h)] = p.astype(np.int32)
            run.orc.g[b, l] = g
            gs.append(g)
            cs.append(c)
        tp = run.torch.from_numpy(pos).cuda()
        tk, tv = run.up(kk), run.up(vv)
        ra.ra_restore(run.ctx, l, gs, cs, tp.data_ptr(), tk.data_ptr(), tv.data_ptr(), cmax)
        run.torch.cuda.synchronize()


def _step_all(run, t):
    """One ra_decode_step over every layer; the oracle appends and evicts in the same order."""
    import paper_2609_03430_gb300 as ra

    L, B, H, KVH, D = run.L, run.B, run.H, run.KVH, run.D
    q = np.zeros((L, B, H, D), np.uint16)
    k = np.zeros((L, B, KVH, D), np.uint16)
    v = np.zeros_like(k)
    fired = 0
    for l in range(L):
        for b in range(B):
            pos = run.orc.append(b, l)
            for h in range(KVH):
                k[l, b, h] = run.krows(l, b, h, [pos])[0]
                v[l, b, h] = run.vrows(l, b, h, [pos])[0]
            q[l, b] = __import__("synth").q_rows(run.dseed, l, b, np.arange(H), t, D)
            fired += bool(run.orc.evict(b, l))
    tq, tk, tv = run.up(q), run.up(k), run.up(v)
    out = run.torch.zeros((L, B, H, D), dtype=run.torch.int16, device="cuda")
    ra.ra_decode_step(run.ctx, tq.data_ptr(), tk.data_ptr(), tv.data_ptr(), out.data_ptr())
    run.torch.cuda.synchronize()
    return q, out.cpu().numpy(), fired


CASES = [(0, 1, 0, 0), (1, 1, 0, 0), (2, 1, 0, 0), (0, 1, 256, 0), (3, 16, 0, 0),
         (0, 1, 0, 1), (1, 1, 0, 1), (2, 1, 0, 1), (0, 1, 256, 1), (3, 16, 0, 1)]
IDS = ["random", "shared", "recency", "random-exact", "block16",
       "orderfree-random", "orderfree-shared", "orderfree-recency", "orderfree-random-exact", "orderfree-block16"]


@pytest.mark.parametrize("policy,block,mode,compaction", CASES, ids=IDS)
def test_evicted_sets_computed_ahead_match_the_oracle(policy, block, mode, compaction):
    import oracle
    import paper_2609_03430_gb300 as ra

    K, r = 480, 32
    run = Runner(L=3, H=24, KVH=4, prompt_lens=[40, 0, 17, 300, 5], K=K, r=r, eseed=61 + policy, dseed=62,
                 policy=policy, block=block, compaction=compaction)
    ra.ra_set_eviction_kernel(run.ctx, mode)
    phases = [0, 7, 31, 16, 30]
    _restore_phased(run, phases, epoch=40)
    ra.ra_profile_reset(run.ctx)
    total = 0
    for t in range(2 * r + 3):  # every sequence fires twice
        q, got, fired = _step_all(run, t)
        total += fired
        if t % 11 == 0:
            run.check_state()
    assert total >= 2 * run.B * run.L
    run.check_state()
    for l in range(run.L):
        for b in range(run.B):
            for h in range(run.KVH):
                pos = run.orc.positions(b, l, h)
                G = run.G
                ref = oracle.attend(q[l, b, h * G:(h + 1) * G], run.krows(l, b, h, pos), run.vrows(l, b, h, pos))
                check_attention(got[l, b, h * G:(h + 1) * G], ref, f"layer {l} seq {b} head {h}")
    _, n_plan, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_PLAN)
    _, n_stack, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_STACK)
    assert n_plan > 0 and n_stack > 0
    run.close()


@pytest.mark.parametrize("policy,block", [(0, 1), (3, 16)], ids=["random", "block16"])
def test_per_layer_calls_in_order_form_steps(policy, block):
    """ra_decode_layer for layers 0 .. L-1 in order: layer 0's call runs the step's whole-stack
    eviction from the sets computed during the previous step, exactly as ra_decode_step does.
    Bit-exact against the oracle, with attention checked on some steps."""
    import paper_2609_03430_gb300 as ra

    K, r = 480, 32
    run = Runner(L=3, H=24, KVH=4, prompt_lens=[40, 0, 17, 300, 5], K=K, r=r, eseed=81 + policy, dseed=82,
                 fused=True, policy=policy, block=block)
    _restore_phased(run, [0, 7, 31, 16, 30], epoch=40)
    ra.ra_profile_reset(run.ctx)
    for t in range(2 * r + 3):
        run.step(check_attn_layers=(0, 2) if t % 9 == 0 else ())
        if t % 11 == 0:
            run.check_state()
    run.check_state()
    assert int(run.orc.n_evictions.min()) >= 2
    _, n_plan, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_PLAN)
    _, n_stack, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_STACK)
    assert n_plan > 0 and n_stack > 0
    run.close()


@pytest.mark.parametrize("compaction", [0, 1], ids=["ordered", "orderfree"])
def test_evicted_sets_computed_ahead_with_fewer_candidates_than_a_warp(compaction):
    """K + r < 32 candidates per head (K = 4, r = 8: 12), so a warp's lanes outnumber them."""
    import oracle
    import paper_2609_03430_gb300 as ra

    K, r = 4, 8
    run = Runner(L=2, H=8, KVH=2, prompt_lens=[3, 0, 20], K=K, r=r, eseed=91, dseed=92, compaction=compaction)
    _restore_phased(run, [0, 3, 7], epoch=6)
    ra.ra_profile_reset(run.ctx)
    for t in range(3 * r + 1):
        q, got, _ = _step_all(run, t)
        run.check_state()
    for l in range(run.L):
        for b in range(run.B):
            for h in range(run.KVH):
                pos = run.orc.positions(b, l, h)
                G = run.G
                ref = oracle.attend(q[l, b, h * G:(h + 1) * G], run.krows(l, b, h, pos), run.vrows(l, b, h, pos))
                check_attention(got[l, b, h * G:(h + 1) * G], ref, f"layer {l} seq {b} head {h}")
    _, n_stack, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_STACK)
    assert n_stack > 0
    run.close()


@pytest.mark.parametrize("compaction", [0, 1], ids=["ordered", "orderfree"])
def test_stacked_and_per_layer_steps_interleaved(compaction):
    """ra_decode_step and in-order ra_decode_layer steps, alternating in runs of different lengths:
    the sets computed during one form's step serve the other's, bit-exact against the oracle."""
    import paper_2609_03430_gb300 as ra

    K, r = 96, 16
    run = Runner(L=3, H=16, KVH=4, prompt_lens=[12, 0, 40, 7], K=K, r=r, eseed=95, dseed=96, fused=True,
                 compaction=compaction)
    _restore_phased(run, [0, 5, 15, 9], epoch=20)
    ra.ra_profile_reset(run.ctx)
    forms = ([0] * 3 + [1] * 2 + [0] + [1] * 5) * 6  # 0: the stacked call, 1: per-layer calls
    for t, form in enumerate(forms[:3 * r + 2]):
        if form == 0:
            _step_all(run, t)
        else:
            run.step_idx = t
            run.step()
        if t % 5 == 0:
            run.check_state()
    run.check_state()
    assert int(run.orc.n_evictions.min()) >= 2
    _, n_stack, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_STACK)
    assert n_stack > 0
    run.close()


@pytest.mark.parametrize("compaction", [0, 1], ids=["ordered", "orderfree"])
def test_evicted_sets_computed_ahead_with_the_largest_buffer(compaction):
    """r = 512, the largest buffer the sets computed ahead serve: each round evicts 512 per head, more
    than the sampled cut's list holds, so the plan kernel takes its exact radix passes."""
    import paper_2609_03430_gb300 as ra

    K, r = 1024, 512
    run = Runner(L=2, H=8, KVH=2, prompt_lens=[5, 0, 30], K=K, r=r, eseed=97, dseed=98, compaction=compaction)
    _restore_phased(run, [r - 4, r - 11, r - 21], epoch=6)  # each fires within 21 steps, planned a step ahead
    ra.ra_profile_reset(run.ctx)
    for t in range(24):
        _step_all(run, t)
    run.check_state()
    assert int(run.orc.n_evictions.min()) >= 1
    _, n_stack, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_STACK)
    assert n_stack == 3
    run.close()
