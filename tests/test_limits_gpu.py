"""Parity at the library's size limits: the random eviction with K + r at the selection's maximum
candidate count (32768 keys staged in shared memory), in both call forms and both compaction
layouts, and the scored comparator with both of its limits at once (a 512-row query window and
K + r = 16384 candidates).  Caches are restored one step before a firing, so the first step evicts
from a full cache."""
import numpy as np
import pytest

from conftest import cuda_available
from ra_testlib import Runner, check_attention

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]


@pytest.mark.parametrize("fused,compaction", [(False, 0), (True, 0), (True, 1)],
                         ids=["separate-ordered", "fused-ordered", "fused-holefill"])
def test_random_eviction_at_max_candidates(fused, compaction):
    K, r = 32768 - 64, 64  # K + r = 32768 candidates per head
    run = Runner(L=1, H=4, KVH=2, prompt_lens=[64, 5], K=K, r=r, eseed=11, dseed=12, fused=fused,
                 compaction=compaction)
    g = 640 * r - 1  # the next step's token makes g a multiple of r with K + r candidates: it fires
    run.restore_full(g)
    fired = run.step(check_attn_layers=(0,))
    assert fired[0] == run.B
    run.check_state()
    for _ in range(2):  # and the steps after it, on the compacted cache
        assert run.step(check_attn_layers=(0,))[0] == 0
    run.check_state()
    run.close()


def test_scored_comparator_at_max_window_and_candidates():
    """The scored comparator with a 512-row window (r = 64, G = 8: two tcgen05 products per K-step,
    one accumulator buffer) and K + r = 16384 candidates (the scored select's maximum).  The window is
    loaded with ra_restore_queries, one step before a firing; the firing step's raw scores must match
    the oracle's fp64 window scores element by element, its keep-set the oracle's round on the
    kernel's scores, and survivors, bytes and attention the oracle's."""
    import torch

    import oracle
    import paper_2609_03430_gb300 as ra
    import synth
    from ra_testlib import check_scored_decision, check_scores

    L, H, KVH, D, lp, r = 1, 16, 2, 128, 64, 64
    K = 16384 - r
    G = H // KVH
    dseed, eseed = 21, 22
    W0 = 1 << 20  # generator step index of the restored window's row 0
    for fused in (False, True):
        cache = ra.RandomAttentionCache(L, H, KVH, D, [lp], K, r, eseed, policy=ra.RA_POLICY_SNAPKV)
        ctx = cache.ctx
        dev = torch.device("cuda")

        def up(a):
            return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev)

        pk = np.stack([synth.kv_rows(dseed, 0, 0, 0, h, np.arange(lp), D) for h in range(KVH)])[None]
        pv = np.stack([synth.kv_rows(dseed, 1, 0, 0, h, np.arange(lp), D) for h in range(KVH)])[None]
        tpk, tpv = up(pk), up(pv)
        ra.ra_prefill(ctx, 0, tpk.data_ptr(), tpv.data_ptr(), lp)
        g0 = 300 * r - 1  # the next step's token fires a round over K + r candidates
        c0 = K + 2 * r - 1
        gpos = lp + np.arange(g0 - c0, g0)
        kg = np.stack([synth.kv_rows(dseed, 0, 0, 0, h, gpos, D) for h in range(KVH)])[None]
        vg = np.stack([synth.kv_rows(dseed, 1, 0, 0, h, gpos, D) for h in range(KVH)])[None]
        tpos = torch.from_numpy(np.broadcast_to(gpos.astype(np.int32), (1, KVH, c0)).copy()).to(dev)
        tkg, tvg = up(kg), up(vg)
        ra.ra_restore(ctx, 0, [g0], [c0], tpos.data_ptr(), tkg.data_ptr(), tvg.data_ptr(), c0)
        qw = np.stack([synth.q_rows(dseed, 0, 0, np.arange(H), W0 + u, D) for u in range(r)], axis=1)[None]
        tqw = up(qw)  # [1][H][r][D]: row u = the query of decode step g0 - r + 1 + u
        ra.ra_restore_queries(ctx, 0, tqw.data_ptr())
        orc = oracle.OracleCache(L, KVH, [lp], K, r, eseed, policy=oracle.POLICY_SNAPKV)
        for h in range(KVH):
            orc.gen[(0, 0, h)] = gpos.astype(np.int32)
        orc.g[0, 0] = g0

        def scorer(b, l, h, cur):
            g, n = int(orc.g[b, l]), cur.size - r
            steps = range(g - r, g)  # 1-based decode steps of the window: the restored ones
            qh = np.arange(h * G, (h + 1) * G)
            q = np.stack([synth.q_rows(dseed, 0, 0, qh, W0 + s - (g0 - r + 1), D) for s in steps])
            qpos = np.array([lp + s - 1 for s in steps], dtype=np.int32)
            kpos = orc.positions(b, l, h)
            ref = oracle.window_scores(q, qpos, synth.kv_rows(dseed, 0, 0, 0, h, kpos, D), kpos)[lp:lp + n]
            got = ra.ra_get_scores(ctx, 0, 0, h, K + 2 * r)
            check_scores(got, ref, f"scores h{h} fused={fused}")
            check_scored_decision(got, ref, K, f"decision h{h} fused={fused}")
            return got.astype(np.float64)

        pos = orc.append(0, 0)
        kn = np.stack([synth.kv_rows(dseed, 0, 0, 0, h, [pos], D)[0] for h in range(KVH)])[None]
        vn = np.stack([synth.kv_rows(dseed, 1, 0, 0, h, [pos], D)[0] for h in range(KVH)])[None]
        q = synth.q_rows(dseed, 0, 0, np.arange(H), 0, D)[None]
        tkn, tvn, tq = up(kn), up(vn), up(q)
        out = torch.zeros((1, H, D), dtype=torch.int16, device=dev)
        if fused:
            ra.ra_decode_layer(ctx, 0, tq.data_ptr(), tkn.data_ptr(), tvn.data_ptr(), out.data_ptr())
        else:
            ra.ra_append_kv(ctx, 0, tkn.data_ptr(), tvn.data_ptr())
            assert ra.ra_evict(ctx, 0) == 1
            ra.ra_decode_attn(ctx, 0, tq.data_ptr(), out.data_ptr())
        torch.cuda.synchronize()
        assert orc.evict(0, 0, scorer=scorer)
        ra.ra_check_device(ctx)
        got_out = out.cpu().numpy()
        for h in range(KVH):
            np.testing.assert_array_equal(ra.ra_get_positions(ctx, 0, 0, h, K + 2 * r), orc.gen[(0, 0, h)])
            p = orc.positions(0, 0, h)
            krow, vrow = synth.kv_rows(dseed, 0, 0, 0, h, p, D), synth.kv_rows(dseed, 1, 0, 0, h, p, D)
            kk, vv = ra.ra_get_kv(ctx, 0, 0, h, lp + K + 2 * r)
            np.testing.assert_array_equal(kk, krow)
            np.testing.assert_array_equal(vv, vrow)
            check_attention(got_out[0, h * G:(h + 1) * G], oracle.attend(q[0, h * G:(h + 1) * G], krow, vrow),
                            f"attention h{h} fused={fused}")
        cache.close()
