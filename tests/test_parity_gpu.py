"""GPU parity: the CUDA path through the C ABI against the oracle, element by element.

Eviction (survivor positions and compacted K/V bytes) must match bit-exactly;
attention must be within max-abs 2e-2 and mean-rel 5e-3 of the fp64 oracle.
"""
import numpy as np
import pytest

from conftest import cuda_available
from ra_testlib import Runner, check_attention

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]


@pytest.mark.parametrize("fused", [False, True], ids=["separate-calls", "fused-layer"])
def test_config1_full_run(fused):
    """Qwen3-4B attention shape, one layer, batch 1, prompt 128, K=256, r=64, 1024 steps, seed 0:
    eleven evictions; state checked bit-exactly after each, attention every 8th step and at firings."""
    run = Runner(L=1, H=32, KVH=8, prompt_lens=[128], K=256, r=64, eseed=0, dseed=1, fused=fused)
    n_fire = 0
    for step in range(1024):
        g_next = step + 1
        firing = g_next % 64 == 0 and g_next >= 384
        fired = run.step(check_attn_layers=(0,) if (step % 8 == 7 or firing or step < 3) else ())
        n_fire += fired[0]
        if fired[0]:
            run.check_state()
    assert n_fire == 11
    run.check_state()
    run.close()


@pytest.mark.parametrize("fused", [False, True], ids=["separate-calls", "fused-layer"])
def test_ragged_batch_layers_and_finishing(fused):
    """Ragged prompts (including an empty one), G=5, K not a multiple of r, two layers,
    a sequence that finishes mid-run."""
    run = Runner(L=2, H=40, KVH=8, prompt_lens=[0, 17, 100, 33, 250], K=100, r=32, eseed=5, dseed=3, fused=fused)
    for step in range(420):
        if step == 200:
            run.set_active(3, False)
        fired = run.step(check_attn_layers=(0, 1) if step % 37 == 0 or step in (191, 192, 193, 419) else ())
        if any(fired.values()):
            run.check_state()
    run.check_state()
    run.close()


@pytest.mark.parametrize("shape", [1, 2], ids=["wide", "narrow"])
@pytest.mark.parametrize("G", [1, 2, 3, 4, 6, 7, 8])
def test_group_sizes(G, shape):
    """Every group size through both attention kernel shapes (48-row tiles x 4 warps, 32 x 6)."""
    run = Runner(L=1, H=2 * G, KVH=2, prompt_lens=[70, 1], K=48, r=16, eseed=G, dseed=10 + G, fused=G % 2 == 0,
                 attn_shape=shape)
    for step in range(150):
        fired = run.step(check_attn_layers=(0,) if step % 25 == 0 or step in (95, 96, 97) else ())
        if any(fired.values()):
            run.check_state()
    run.close()


@pytest.mark.parametrize("policy,block,fused", [(1, 1, True), (2, 1, False), (3, 4, True), (3, 16, False)],
                         ids=["shared-draw", "recency", "block4", "block16"])
def test_policy_variants(policy, block, fused):
    """The controls the paper contrasts with the method, run by the same kernels: survivors bit-exact."""
    run = Runner(L=2, H=16, KVH=4, prompt_lens=[30, 0, 77], K=96, r=32, eseed=11, dseed=6, fused=fused,
                 policy=policy, block=block)
    for step in range(330):
        fired = run.step(check_attn_layers=(1,) if step % 60 == 0 else ())
        if any(fired.values()):
            run.check_state()
    run.close()


def test_degenerate_budgets():
    # K = 0: only the recent buffer survives; r = 1 evicts at every step once the cache exceeds K + 1
    for (K, r), fused in [((0, 8), False), ((5, 1), False), ((3, 2), False), ((0, 8), True), ((5, 1), True),
                          ((3, 2), True)]:
        run = Runner(L=1, H=4, KVH=2, prompt_lens=[9], K=K, r=r, eseed=K + r, dseed=2, fused=fused)
        for step in range(60):
            fired = run.step(check_attn_layers=(0,) if step % 7 == 0 else ())
            if any(fired.values()):
                run.check_state()
        run.close()


def test_attention_long_restored_state():
    """Attention over restored caches long enough that heads span several warps' ranges,
    with ragged lengths (prompt only, generated only, both)."""
    import torch

    import oracle
    import paper_2609_03430_gb300 as ra
    import synth

    L, H, KVH, D, K, r = 1, 16, 4, 128, 3000, 64
    lps = [0, 4096, 1000, 7]
    run = Runner(L=L, H=H, KVH=KVH, prompt_lens=lps, K=K, r=r, eseed=1, dseed=4)
    gs = [3100, 0, 3127, 40]
    cs = [3100, 0, 3127, 40]
    stride = max(cs)
    pos = np.zeros((len(lps), KVH, stride), np.int32)
    kk = np.zeros((len(lps), KVH, stride, D), np.uint16)
    vv = np.zeros_like(kk)
    for b in range(len(lps)):
        for h in range(KVH):
            p = lps[b] + np.arange(gs[b] - cs[b], gs[b])
            pos[b, h, : cs[b]] = p
            kk[b, h, : cs[b]] = run.krows(0, b, h, p)
            vv[b, h, : cs[b]] = run.vrows(0, b, h, p)
            run.orc.gen[(b, 0, h)] = p.astype(np.int32)
        run.orc.g[b, 0] = gs[b]
    tp = torch.from_numpy(pos).cuda()
    tkk, tvv = run.up(kk), run.up(vv)
    ra.ra_restore(run.ctx, 0, gs, cs, tp.data_ptr(), tkk.data_ptr(), tvv.data_ptr(), stride)
    for scale in (0.0, 0.02):
        q = np.stack([synth.q_rows(4, 0, b, np.arange(H), 7, D) for b in range(len(lps))])
        out = torch.zeros((len(lps), H, D), dtype=torch.int16, device="cuda")
        tq = run.up(q)
        ra.ra_decode_attn(run.ctx, 0, tq.data_ptr(), out.data_ptr(), scale)
        got = out.cpu().numpy()
        G = H // KVH
        for b in range(len(lps)):
            for h in range(KVH):
                p = run.orc.positions(b, 0, h)
                ref = oracle.attend(q[b, h * G:(h + 1) * G], run.krows(0, b, h, p), run.vrows(0, b, h, p), scale)
                if p.size == 0:
                    assert np.all(got[b, h * G:(h + 1) * G] == 0)
                else:
                    check_attention(got[b, h * G:(h + 1) * G], ref, f"seq {b} head {h}")
    run.close()


def test_capacity_error_leaves_state_unchanged():
    import paper_2609_03430_gb300 as ra

    run = Runner(L=1, H=4, KVH=2, prompt_lens=[3], K=8, r=4, eseed=0, dseed=0)
    k = run.up(np.zeros((1, 2, 128), np.uint16))
    for _ in range(8 + 2 * 4):
        ra.ra_append_kv(run.ctx, 0, k.data_ptr(), k.data_ptr())  # never evict
    before = ra.ra_get_counters(run.ctx, 0, 0)
    with pytest.raises(ra.RAError) as e:
        ra.ra_append_kv(run.ctx, 0, k.data_ptr(), k.data_ptr())
    assert e.value.code == ra.RA_ERR_CAPACITY
    assert ra.ra_get_counters(run.ctx, 0, 0) == before
    run.cache.close()


def test_synth_gpu_twin_is_bit_identical():
    import torch

    import synth
    import synth.gpu as sg

    B, NH, n, D = 3, 5, 37, 128
    rng = np.random.default_rng(0)
    pos = rng.integers(0, 40000, size=(B, NH, n)).astype(np.int32)
    pos[1, 2, 5] = -1
    scale = synth.key_channel_scale(9, 2, NH, D)[1]
    for stream, sc in [(0, None), (1, None), (0, scale), (2, None)]:
        out = torch.empty((B, NH, n, D), dtype=torch.int16, device="cuda")
        sg.fill_rows(out, torch.from_numpy(pos).cuda(), 77, stream, 1, 5,
                     None if sc is None else torch.from_numpy(sc).cuda())
        got = out.cpu().numpy().view(np.uint16)
        for b in range(B):
            for h in range(NH):
                want = synth.kv_rows(77, stream, 1, 5 + b, h, np.maximum(pos[b, h], 0), D,
                                     None if sc is None else sc[h])
                want[pos[b, h] < 0] = 0
                np.testing.assert_array_equal(got[b, h], want)
