"""GPU parity of compaction fused into the attention pass (RA_COMPACT_FUSED).

The fused step's attention kernel reads each evicting head's old region, gives
the evicted rows no weight and writes the survivors (and the step's token) to
their slots in the new region.  The result must be the ordered layout exactly:
positions and K/V bytes equal the oracle's (ordered compaction) bit-exactly, and
attention matches the fp64 oracle within tolerance -- including rounds whose
evicted rows form long runs (protected recency, the scored comparator).
"""
import pytest

from conftest import cuda_available
from ra_testlib import Runner

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]

FUSED = 2


@pytest.mark.parametrize("policy,block", [(0, 1), (2, 1), (3, 16), (4, 1)], ids=["random", "recency", "block16", "scored"])
def test_fused_compaction_policies(policy, block):
    run = Runner(L=2, H=16, KVH=4, prompt_lens=[30, 0, 77], K=96, r=32, eseed=17, dseed=5, fused=True,
                 policy=policy, block=block, compaction=FUSED)
    n_fired = 0
    for step in range(330):
        fired = run.step(check_attn_layers=(0, 1) if step % 31 == 0 or step in (159, 160, 191, 192) else ())
        n_fired += fired[0]
        if any(fired.values()):
            run.check_state()
    assert n_fired == 3 * 6
    run.close()


def test_fused_compaction_config1_shape():
    """Qwen3-4B attention shape, r = 64 (a full 64-bit evicted mask per tile), 600 steps."""
    run = Runner(L=1, H=32, KVH=8, prompt_lens=[128], K=256, r=64, eseed=0, dseed=1, fused=True, compaction=FUSED)
    for step in range(600):
        fired = run.step(check_attn_layers=(0,) if step % 16 == 15 or step in (383, 384) else ())
        if fired[0]:
            run.check_state()
    run.check_state()
    run.close()
