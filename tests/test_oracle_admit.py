"""Oracle pins for admission: a finished slot takes a new request (NEXT-4's serving follow-on).

The new request restarts the slot's state (its own prompt, nothing generated or cached) and
draws its own random stream -- the admission count sits above the head id in Philox's fourth
counter word, the paper's per-request seed read per request rather than per slot.  Pinned by:
the creation batch keeps exactly the keys it had before admissions existed; streams of
(admission, head) pairs never collide; an admitted request follows the same cadence and round
invariants; its keep-sets differ from the previous occupant's at the same step; and over many
admissions each candidate is kept with probability K/N (chi-square), so the new streams stay
uniform.
"""
import numpy as np
from scipy import stats

import oracle


def test_creation_batch_keys_are_unchanged():
    seed, layer, g, K, r = 11, 3, 640, 96, 32
    gen = 50 + np.arange(K + 2 * r - 0, dtype=np.int32)[: K + r + 32]
    for seq, kvh, h in [(0, 4, 0), (3, 8, 5), (511, 32, 31)]:
        a, _ = oracle.evict_head(gen, g, K, r, seed, layer, seq * kvh + h)
        b, _ = oracle.evict_head(gen, g, K, r, seed, layer, oracle.head_stream(0, seq * kvh + h))
        c, _ = oracle.evict_head_policy(gen, g, K, r, seed, layer, seq, kvh, h, oracle.POLICY_RANDOM)
        np.testing.assert_array_equal(a, b)
        np.testing.assert_array_equal(a, c)


def test_streams_of_admissions_and_heads_never_collide():
    ids = {oracle.head_stream(a, x) for a in range(4) for x in range(0, 512 * 32, 7)}
    assert len(ids) == 4 * len(range(0, 512 * 32, 7))


def test_admitted_request_restarts_the_slot():
    K, r = 64, 16
    orc = oracle.OracleCache(2, 2, [30, 5], K, r, seed=9)
    for _ in range(K + 3 * r):
        for l in range(2):
            for b in range(2):
                orc.append(b, l)
                orc.evict(b, l)
    assert orc.n_evictions[0, 0] == 2
    orc.admit(0, 77)
    assert orc.prompt_lens[0] == 77 and orc.admissions == [1, 0]
    assert orc.g[0, 0] == 0 and orc.n_evictions[0, 1] == 0 and orc.c(0, 1) == 0
    fired_at = []
    for step in range(K + 3 * r):
        for l in range(2):
            pos = orc.append(0, l)
            if l == 0 and step == 0:
                assert pos == 77  # positions restart after the new prompt
            if orc.evict(0, l) and l == 0:
                fired_at.append(int(orc.g[0, 0]))
    assert fired_at == [K + 2 * r, K + 3 * r]  # the same cadence as a first request
    for l in range(2):
        for h in range(2):
            p = orc.positions(0, l, h)
            assert p[:77].tolist() == list(range(77)) and np.all(np.diff(p) > 0) and p.size == 77 + K + r


def test_admissions_draw_new_uniform_keep_sets():
    seed, layer, K, r, kvh, seq, h = 5, 1, 48, 16, 8, 7, 3
    N = K + r
    g = 10 * r
    gen = np.arange(N + r, dtype=np.int32)
    first, _ = oracle.evict_head_policy(gen, g, K, r, seed, layer, seq, kvh, h, oracle.POLICY_RANDOM, 1, 0)
    counts = np.zeros(N)
    differ = 0
    rounds = 3000
    for a in range(1, rounds + 1):
        kept, _ = oracle.evict_head_policy(gen, g, K, r, seed, layer, seq, kvh, h, oracle.POLICY_RANDOM, 1, a)
        assert kept.size == K + r and np.all(np.diff(kept) > 0) and np.array_equal(kept[K:], gen[N:])
        counts[kept[:K]] += 1
        differ += not np.array_equal(kept, first)
    assert differ >= rounds - 1  # a new request does not replay its predecessor's draw
    expected = rounds * K / N
    chi2 = float(((counts - expected) ** 2 / expected).sum())
    assert stats.chi2.sf(chi2, N - 1) > 1e-4, chi2
