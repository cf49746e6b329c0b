"""Admission of new requests into finished slots (prompt pages + ra_admit), through the C ABI,
against the oracle: sequences finish mid-run and their slots take requests with prompts of other
lengths (longer, shorter, empty); every head's survivors and cached rows stay bit-exact, and
attention over the paged prompts stays within tolerance -- in both call forms, through the fused
layer step, and through the whole-stack step whose evicted sets are computed ahead.  Host-side
refusals (active slot, prompt too long, pool exhausted) leave the state unchanged.
"""
import numpy as np
import pytest

from conftest import cuda_available
from ra_testlib import Runner

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]

# (step, slot, new prompt length): longer than any creation prompt, empty, short, several pages
ADMISSIONS = [(20, 1, 1100), (45, 3, 0), (60, 0, 7), (90, 1, 385)]


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
def test_finished_slots_take_new_requests(fused):
    import paper_2609_03430_gb300 as ra

    run = Runner(L=2, H=24, KVH=4, prompt_lens=[40, 300, 0, 900], K=48, r=16, eseed=71, dseed=72, fused=fused,
                 prompt_pool=(1200, 3000))
    plan = {s: (b, lp) for s, b, lp in ADMISSIONS}
    for step in range(175):  # the last admitted request reaches its first eviction (K + 2r steps)
        if step in plan:
            b, lp = plan[step]
            run.admit(b, lp)
            run.check_state()
        run.step(check_attn_layers=(0, 1) if step % 10 == 0 else ())
    assert all(n >= 1 for n in run.orc.n_evictions[:, 0])  # every current request evicted
    run.check_state()
    run.close()


@pytest.mark.parametrize("compaction", [0, 1], ids=["ordered", "orderfree"])
def test_admission_through_the_whole_stack_step(compaction):
    """ra_decode_step (evicted sets computed one step ahead) with admissions between steps, in both
    layouts (order-free: keys per position, read by the plans)."""
    import paper_2609_03430_gb300 as ra
    import synth

    run = Runner(L=3, H=16, KVH=4, prompt_lens=[250, 17, 0], K=32, r=16, eseed=73, dseed=74,
                 prompt_pool=(800, 1800), compaction=compaction)
    dev = run.dev
    for step in range(120):
        if step == 30:
            run.admit(2, 640)
        if step == 55:
            run.admit(0, 3)
        L, B, H, KVH, D = run.L, run.B, run.H, run.KVH, run.D
        q = np.zeros((L, B, H, D), np.uint16)
        k = np.zeros((L, B, KVH, D), np.uint16)
        v = np.zeros_like(k)
        for l in range(L):
            for b in range(B):
                pos = run.orc.append(b, l)
                for h in range(KVH):
                    k[l, b, h] = run.krows(l, b, h, [pos])[0]
                    v[l, b, h] = run.vrows(l, b, h, [pos])[0]
                q[l, b] = run.qrows(l, b, step)
                run.orc.evict(b, l)
        tq, tk, tv = run.up(q), run.up(k), run.up(v)
        out = run.torch.zeros((L, B, H, D), dtype=run.torch.int16, device=dev)
        ra.ra_decode_step(run.ctx, tq.data_ptr(), tk.data_ptr(), tv.data_ptr(), out.data_ptr())
        run.torch.cuda.synchronize()
        if step % 17 == 0:
            run.check_state()
            got = out.cpu().numpy()
            for l in range(L):
                run.check_layer_attention(l, q[l], got[l])
    run.check_state()
    _, n_plan, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_PLAN)
    assert n_plan > 0
    run.close()


def test_admission_refusals_leave_the_state_unchanged():
    import torch

    import paper_2609_03430_gb300 as ra

    run = Runner(L=1, H=8, KVH=2, prompt_lens=[100, 200], K=16, r=8, eseed=75, dseed=76, prompt_pool=(400, 700))
    for _ in range(5):
        run.step()
    lib = ra.lib()
    s = torch.cuda.current_stream().cuda_stream
    buf = torch.zeros((1, 2, 512, 128), dtype=torch.int16, device="cuda")
    assert lib.ra_admit(run.ctx, 0, 50, buf.data_ptr(), buf.data_ptr(), 512, s) == ra.RA_ERR_STATE  # still active
    run.set_active(0, False)
    assert lib.ra_admit(run.ctx, 0, 401, buf.data_ptr(), buf.data_ptr(), 512, s) == ra.RA_ERR_CAPACITY  # too long
    assert lib.ra_admit(run.ctx, 2, 10, buf.data_ptr(), buf.data_ptr(), 512, s) == ra.RA_ERR_INVALID_ARG
    # pool: 700 positions -> 4 pages; slot 1 holds 2 (200 positions), slot 0 may take 2 of its own + 0 free
    assert lib.ra_admit(run.ctx, 0, 385, buf.data_ptr(), buf.data_ptr(), 512, s) == ra.RA_ERR_CAPACITY
    run.set_active(0, True)
    for _ in range(3):  # nothing changed: the run goes on bit-exact
        run.step(check_attn_layers=(0,))
    run.check_state()
    run.close()
