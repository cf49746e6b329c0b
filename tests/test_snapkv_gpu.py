"""GPU parity of the scored comparator (SnapKV-style window top-K, prompt pinned).

At every scored round the kernel's raw window scores are compared element by
element with the fp64 oracle's (section 2's SnapKV score: attention from the
last r queries, summed over the query heads of the group); the round's keep-set
must then be exactly the oracle's max-pool + top-K applied to the kernel's
scores, and where the fp64 scores would decide differently the candidates
involved must sit at the threshold.  K/V state and attention are checked as for
the random policy.
"""
import numpy as np
import pytest

from conftest import cuda_available
from ra_testlib import Runner

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]

SNAPKV = 4


@pytest.mark.parametrize("fused", [False, True], ids=["separate-calls", "fused-layer"])
def test_snapkv_ragged_batch(fused):
    """G=4, r=32 (128 window rows), ragged prompts including an empty one, two layers."""
    run = Runner(L=2, H=16, KVH=4, prompt_lens=[30, 0, 77], K=96, r=32, eseed=11, dseed=21, fused=fused,
                 policy=SNAPKV)
    for step in range(330):
        fired = run.step(check_attn_layers=(0, 1) if step % 41 == 0 or step in (159, 160, 161, 329) else ())
        if any(fired.values()):
            run.check_state()
    assert run.scored_rounds == 2 * 3 * 4 * 6  # layers x sequences x heads x rounds (g = 160, 192, ..., 320)
    run.check_state()
    run.close()


@pytest.mark.parametrize("G,r,K,lp", [(1, 16, 40, [50]), (5, 32, 64, [200, 3]), (6, 64, 64, [130]), (8, 64, 80, [64, 0])],
                         ids=["rows16", "rows160", "rows384", "rows512"])
def test_snapkv_window_shapes(G, r, K, lp):
    """Window row counts that use 1, 2, 3 and 4 M tiles per warp, prompts shorter and longer than a tile."""
    run = Runner(L=1, H=2 * G, KVH=2, prompt_lens=lp, K=K, r=r, eseed=G, dseed=30 + G, fused=G % 2 == 0,
                 policy=SNAPKV)
    first = (K + r) // r * r + r  # the first multiple of r above K + r
    n_fired = 0
    for step in range(first + r + 3):
        fired = run.step(check_attn_layers=(0,) if step in (first - 2, first - 1, first + r - 1) else ())
        n_fired += fired[0]
        if fired[0]:
            run.check_state()
    assert n_fired == 2 * len(lp) and run.scored_rounds == n_fired * 2
    run.close()


def test_snapkv_key_scale_and_scale_argument():
    """Keys with a per-channel LogNormal(0, 0.5) scale (peaked attention), non-default attention scale."""
    rng = np.random.default_rng(3)
    ks = np.exp(rng.normal(0.0, 0.5, size=(1, 2, 128))).astype(np.float32)
    run = Runner(L=1, H=8, KVH=2, prompt_lens=[40, 90], K=48, r=16, eseed=2, dseed=8, key_scale=ks, fused=True,
                 policy=SNAPKV)
    n_fired = 0
    for step in range(120):
        fired = run.step(check_attn_layers=(0,) if step % 30 == 0 else (), scale=0.05)
        n_fired += fired[0]
        if fired[0]:
            run.check_state()
    assert n_fired > 0 and run.scored_rounds == n_fired * 2
    run.close()
