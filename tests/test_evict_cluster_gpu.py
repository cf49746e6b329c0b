"""The one-launch eviction (selection and order-preserving compaction in one cluster per head)
against the oracle, bit-exact: survivor positions and the cached K/V rows of every head, at the
firing step and the steps after it.

Cluster sizes 2, 3, 5 and 16 are forced, next to the automatic shape (which also splits each
head's copy over several clusters) and the two-kernel path, under every key-per-ordinal policy:
the random draw and the shared draw (32-bit keys: the sampled cut, or with RA_EVICT_EXACT the
radix passes, whose first digit leaves ~N/256 boundary candidates to rank), protected recency
(keys below 2^11: two digits carry no information, the boundary is found on the third), and
block-contiguous draws with blocks of 16 (ties ranked by ordinal among the gathered candidates)
and of 1024 (more ties than the gather holds: the all-ties path, largest ordinals evicted first,
CTA by CTA).  Both call forms: ra_evict after the append, and the fused step with the token pending.
"""
import numpy as np
import pytest

from conftest import cuda_available
from ra_testlib import Runner

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]

POLICIES = [(0, 1), (1, 1), (2, 1), (3, 16), (3, 1024)]


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("policy,block", POLICIES, ids=["random", "shared", "recency", "block16", "block1024"])
@pytest.mark.parametrize("mode", [0, 256, 1, 2, 3, 5, 16, 3 | 256],
                         ids=["auto", "auto-exact", "two-kernels", "cl2", "cl3", "cl5", "cl16", "cl3-exact"])
def test_one_launch_eviction_matches_the_oracle(mode, policy, block, fused):
    import paper_2609_03430_gb300 as ra

    K, r = 2048 - 64, 64  # K + r = 2048 candidates per head
    run = Runner(L=1, H=16, KVH=4, prompt_lens=[33, 0, 200], K=K, r=r, eseed=31 + policy, dseed=32, fused=fused,
                 policy=policy, block=block)
    ra.ra_set_eviction_kernel(run.ctx, mode)
    run.restore_full(50 * r - 1)
    ra.ra_profile_reset(run.ctx)
    assert run.step(check_attn_layers=(0,))[0] == run.B
    run.check_state()
    _, n_evict, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_EVICT)
    _, n_compact, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_COMPACT)
    assert (n_evict, n_compact) == ((0, 1) if mode == 1 else (1, 0))
    for _ in range(2):
        assert run.step(check_attn_layers=(0,))[0] == 0
    run.check_state()
    run.close()


def test_one_launch_eviction_with_many_heads_in_waves():
    """40 sequences x 8 KV heads firing together: 320 heads, more clusters than run at once, so the
    launch runs in waves; two rounds in a row (the separate calls: no sets are computed ahead, so
    both rounds take the cluster kernel)."""
    import paper_2609_03430_gb300 as ra

    K, r = 512, 32
    run = Runner(L=1, H=32, KVH=8, prompt_lens=[7 * (b % 5) for b in range(40)], K=K, r=r, eseed=41, dseed=42,
                 fused=False)
    run.restore_full(40 * r - 1)
    for _ in range(r + 1):
        run.step()
    assert int(run.orc.n_evictions[:, 0].min()) == 2
    run.check_state()
    _, n_evict, _ = ra.ra_profile_read(run.ctx, ra.RA_KERNEL_EVICT)
    assert n_evict == 2
    run.close()
