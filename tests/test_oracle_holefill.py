"""Pins of the oracle's order-free (hole-filling) compaction.

Attention is a sum over the cached set (section 2, "Notation"), so slot order
carries nothing: a round may refill the evicted slots from the newest ones
instead of moving every survivor.  Keys are drawn per position, which makes the
kept set independent of the slot layout.  Pinned by: the round's invariants
(what moves, what stays, sizes), layout invariance, uniform per-position
inclusion (chi-square), agreement with the pinned select on position keys, and
the policy variants' defining properties.
"""
import numpy as np
import pytest
from scipy.stats import chi2

import oracle

R = oracle.POLICY_RANDOM


def _round(gen, g, K, r, seed=7, layer=1, seq=2, kvh=4, h=1, policy=R, block=1):
    return oracle.evict_head_holefill(np.asarray(gen, np.int32), g, K, r, seed, layer, seq, kvh, h, policy, block)


def test_no_round_without_trigger():
    gen = np.arange(50, 50 + 100, dtype=np.int32)
    new, ev = _round(gen, 63, 40, 16)  # 63 % 16 != 0
    np.testing.assert_array_equal(new, gen)
    assert ev.size == 0
    new, ev = _round(gen[:56], 64, 40, 16)  # c - r = 40, not above K
    assert ev.size == 0 and new.size == 56


@pytest.mark.parametrize("K,r,c", [(96, 32, 160), (40, 16, 71), (0, 8, 16), (5, 64, 70), (3, 2, 7), (5, 1, 7)])
def test_round_invariants(K, r, c):
    """The evicted slots take the rows of slots c - m .. c - 2 in order, and the newest row ends
    in the new last slot (whose own row, when kept, fills the last evicted slot); every other
    slot keeps its row; the cache shrinks by m; the kept set is exactly K candidates plus the
    whole buffer."""
    rng = np.random.default_rng(K + r)
    gen = np.sort(rng.choice(10_000, size=c, replace=False)).astype(np.int32)
    g = (c // r + 1) * r  # a firing step (g multiple of r)
    new, ev = _round(gen, g, K, r)
    n = c - r
    m = n - K
    last = c - m - 1
    assert ev.size == m and new.size == c - m
    assert np.all(np.diff(ev) > 0) and (ev.size == 0 or ev[-1] < n)
    for i, e in enumerate(ev[:-1]):
        assert new[e] == gen[c - m + i]
    assert new[last] == gen[c - 1]  # the newest row is the last
    if ev[-1] != last:
        assert new[ev[-1]] == gen[last]
    untouched = np.setdiff1d(np.arange(c - m), np.append(ev, last))
    np.testing.assert_array_equal(new[untouched], gen[untouched])
    kept_cand = set(gen[:n].tolist()) - set(gen[ev].tolist())
    assert len(kept_cand) == K
    assert set(new.tolist()) == kept_cand | set(gen[n:].tolist())


def test_beyond_capacity_is_rejected():
    """More than K + 2r cached slots would make the newest slots overlap the evicted ones."""
    gen = np.arange(20, dtype=np.int32)
    with pytest.raises(RuntimeError):
        _round(gen, 24, 0, 8)


def test_kept_set_is_position_keyed_topk():
    """The kept set equals the K smallest (key, ordinal) of the pinned select, keys drawn per
    position from the pinned Philox key."""
    K, r, seed, layer, seq, kvh, h = 48, 16, 11, 3, 1, 2, 0
    gen = (200 + 3 * np.arange(K + 2 * r)).astype(np.int32)
    g = 160
    n = gen.size - r
    keys = np.array([oracle.random_key(seed, layer, seq * kvh + h, g, int(p)) for p in gen[:n]], dtype=np.uint32)
    keep = oracle.select_keep(keys, K)
    new, _ = oracle.evict_head_holefill(gen, g, K, r, seed, layer, seq, kvh, h)
    assert set(new.tolist()) == set(gen[keep].tolist()) | set(gen[n:].tolist())


def test_layout_invariance():
    """Permuting the candidates' slots leaves the kept set unchanged (keys follow positions)."""
    K, r = 64, 32
    rng = np.random.default_rng(5)
    gen = (1000 + np.arange(K + 2 * r)).astype(np.int32)
    g = 192
    base, _ = _round(gen, g, K, r)
    for _ in range(5):
        perm = gen.copy()
        perm[: K + r] = rng.permutation(perm[: K + r])
        new, _ = _round(perm, g, K, r)
        assert set(new.tolist()) == set(base.tolist())


def test_uniform_inclusion_per_position():
    """Each candidate position survives with probability K/N (chi-square over 4000 rounds)."""
    K, r = 24, 8
    N = K + r
    gen = (500 + np.arange(K + 2 * r)).astype(np.int32)
    counts = np.zeros(N)
    rounds = 4000
    for s in range(rounds):
        new, _ = _round(gen, 64, K, r, seed=s)
        kept = np.isin(gen[:N], new)
        counts += kept
    expected = rounds * K / N
    stat = (((counts - expected) ** 2) / expected).sum() * (N / (N - K))  # inclusion is Bernoulli(K/N)
    assert stat < chi2.ppf(0.999, N - 1)


def test_policy_variants_by_position():
    K, r = 40, 16
    rng = np.random.default_rng(9)
    gen = np.sort(rng.choice(5000, size=K + 2 * r, replace=False)).astype(np.int32)
    gen[: K + r] = rng.permutation(gen[: K + r])  # candidates in arbitrary slot order
    n = K + r
    g = 80
    # recency: keep the K newest candidate positions, wherever their slots are
    new, _ = _round(gen, g, K, r, policy=oracle.POLICY_RECENCY)
    newest = np.sort(gen[:n])[-K:]
    assert set(new.tolist()) == set(newest.tolist()) | set(gen[n:].tolist())
    # shared: every head keeps the same set
    sets = [set(_round(gen, g, K, r, h=h, policy=oracle.POLICY_SHARED)[0].tolist()) for h in range(4)]
    assert all(x == sets[0] for x in sets)
    # independent draws differ across heads
    rsets = [set(_round(gen, g, K, r, h=h)[0].tolist()) for h in range(4)]
    assert len({frozenset(x) for x in rsets}) > 1
    # block: positions of one block share a key, so at most one block is cut
    blk = 8
    new, _ = _round(gen, g, K, r, policy=oracle.POLICY_BLOCK, block=blk)
    kept = set(new.tolist())
    cand_blocks = {}
    for p in gen[:n]:
        cand_blocks.setdefault(int(p) // blk, []).append(int(p) in kept)
    partial = [b for b, v in cand_blocks.items() if any(v) and not all(v)]
    assert len(partial) <= 1


def test_repeated_rounds_keep_distinct_positions():
    """Over many rounds (appending between them) the cache is always a set of distinct positions
    with exactly K + r entries after each round."""
    K, r, lp = 32, 16, 10
    gen = np.zeros(0, np.int32)
    g = 0
    for step in range(400):
        gen = np.append(gen, np.int32(lp + g))
        g += 1
        before = gen.size
        gen, ev = _round(gen, g, K, r, seed=3)
        if ev.size:
            assert gen.size == K + r and before == K + 2 * r
        assert len(set(gen.tolist())) == gen.size
        assert gen[-1] == lp + g - 1  # the newest token is always cached, in the last slot
