"""GPU parity of order-free (hole-filling) compaction.

Keys follow positions and the evicted slots are refilled in place from the newest
slots, so the slot layout is deterministic: positions and K/V bytes of every slot
must equal the oracle's bit-exactly after every round, and attention (a sum over
the cached set) must match the fp64 oracle within tolerance.
"""
import pytest

from conftest import cuda_available
from ra_testlib import Runner

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]

HOLEFILL = 1


@pytest.mark.parametrize("policy,block,fused", [(0, 1, True), (0, 1, False), (1, 1, True), (2, 1, False), (3, 8, True)],
                         ids=["random-fused", "random-separate", "shared", "recency", "block8"])
def test_holefill_policies(policy, block, fused):
    run = Runner(L=2, H=16, KVH=4, prompt_lens=[30, 0, 77], K=96, r=32, eseed=13, dseed=7, fused=fused, policy=policy,
                 block=block, compaction=HOLEFILL)
    n_fired = 0
    for step in range(330):
        fired = run.step(check_attn_layers=(0, 1) if step % 41 == 0 or step in (159, 160, 161, 191, 192) else ())
        n_fired += fired[0]
        if any(fired.values()):
            run.check_state()
    assert n_fired == 3 * 6  # sequences x rounds (g = 160, 192, ..., 320)
    run.check_state()
    run.close()


@pytest.mark.parametrize("fused", [False, True], ids=["separate-calls", "fused-layer"])
def test_holefill_ragged_finishing(fused):
    """G = 5, K not a multiple of r, a sequence that finishes mid-run, ten rounds of refilling."""
    run = Runner(L=1, H=40, KVH=8, prompt_lens=[0, 17, 100, 250], K=100, r=32, eseed=3, dseed=9, fused=fused,
                 compaction=HOLEFILL)
    for step in range(480):
        if step == 300:
            run.set_active(2, False)
        fired = run.step(check_attn_layers=(0,) if step % 53 == 0 or step in (159, 160, 479) else ())
        if any(fired.values()):
            run.check_state()
    run.check_state()
    run.close()
