"""Pins of the oracle's policy variants (the controls the paper contrasts with Random
Attention, section 5 and Appendix D) against what their definitions fix."""
import numpy as np

import oracle


def rounds(policy, block=1, K=40, r=16, heads=4, n_rounds=30, seed=9):
    """Drive every head from the same start state through n_rounds evictions; returns per-round keep-sets."""
    out = []
    gens = [np.arange(1000, 1000 + K + 2 * r, dtype=np.int32) for _ in range(heads)]
    g = 5 * r  # a firing step
    for rd in range(n_rounds):
        ks = []
        for h in range(heads):
            new, ev = oracle.evict_head_policy(gens[h], g, K, r, seed, 2, 1, heads, h, policy, block)
            ks.append((gens[h].copy(), new.copy(), ev))
            gens[h] = np.append(new, np.arange(1000 + K + 2 * r + rd * r, 1000 + K + 3 * r + rd * r, dtype=np.int32))
        g += r
        out.append(ks)
    return out


def test_random_policy_equals_the_method():
    gen = np.arange(500, 500 + 40 + 32, dtype=np.int32)
    a = oracle.evict_head(gen, 64, 40, 16, 3, 1, 1 * 4 + 2)
    b = oracle.evict_head_policy(gen, 64, 40, 16, 3, 1, 1, 4, 2, oracle.POLICY_RANDOM)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])


def test_shared_draw_is_identical_across_heads_and_uniform():
    res = rounds(oracle.POLICY_SHARED, heads=4, n_rounds=200)
    incl = np.zeros(40 + 16)
    for ks in res:
        for h in range(1, 4):
            np.testing.assert_array_equal(ks[h][2], ks[0][2])  # same evicted ordinals in every head
        mask = np.ones(56, dtype=bool)
        mask[ks[0][2]] = False
        incl += mask
    p = 40 / 56
    z = (incl - 200 * p) / np.sqrt(200 * p * (1 - p))
    assert np.abs(z).max() < 5


def test_random_heads_differ():
    res = rounds(oracle.POLICY_RANDOM, heads=4, n_rounds=20)
    assert any(not np.array_equal(ks[0][2], ks[1][2]) for ks in res)


def test_protected_recency_keeps_the_newest_window():
    for K, r in [(40, 16), (7, 3), (0, 5)]:
        res = rounds(oracle.POLICY_RECENCY, K=K, r=r, heads=1, n_rounds=6)
        for ks in res:
            before, after, ev = ks[0]
            n = before.size - r
            np.testing.assert_array_equal(ev, np.arange(n - K))  # the oldest candidates go
            np.testing.assert_array_equal(after, before[n - K:])  # a contiguous recent window remains


def test_block_policy_keeps_whole_blocks():
    S = 8
    res = rounds(oracle.POLICY_BLOCK, block=S, K=48, r=16, heads=3, n_rounds=40)
    cut_blocks = 0
    for ks in res:
        for before, after, ev in ks:
            n = before.size - 16
            cand = before[:n]
            kept = np.setdiff1d(cand, before[ev])
            for blk in np.unique(cand // S):
                members = cand[cand // S == blk]
                k = np.isin(members, kept)
                if 0 < k.sum() < members.size:
                    cut_blocks += 1
                    # a cut block keeps its lowest-ordinal members (ties go to the lower ordinal)
                    assert np.all(k[: k.sum()]) and not np.any(k[k.sum():])
    # at most one block per round is split by the budget boundary
    assert cut_blocks <= sum(len(ks) for ks in res)


def test_block_size_one_is_a_uniform_draw():
    res = rounds(oracle.POLICY_BLOCK, block=1, heads=1, n_rounds=300)
    incl = np.zeros(56)
    for ks in res:
        mask = np.ones(56, dtype=bool)
        mask[ks[0][2]] = False
        incl += mask
    p = 40 / 56
    z = (incl - 300 * p) / np.sqrt(300 * p * (1 - p))
    assert np.abs(z).max() < 5
