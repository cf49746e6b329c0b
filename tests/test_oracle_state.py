"""Pins of the oracle's eviction state machine (section 2 trigger, section 3 policy,
Appendix F engine details) against invariants and the paper's closed forms."""
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "survival_closed_form.txt")


def run_head(steps, K, r, lp=0, seed=0, layer=0, head_id=0, g0=0, gen0=None):
    gen = np.zeros(0, dtype=np.int32) if gen0 is None else np.asarray(gen0, dtype=np.int32)
    fired = []
    g = g0
    for _ in range(steps):
        gen = np.append(gen, np.int32(lp + g))
        g += 1
        if oracle.should_evict(g, gen.size, K, r):
            new, ev = oracle.evict_head(gen, g, K, r, seed, layer, head_id)
            fired.append((g, gen.copy(), new, ev))
            gen = new
    return gen, fired


def test_trigger_cadence_config1():
    """K=256, r=64, 1024 decode steps: fires first when the cache holds K+2r (g=384)
    and then every r steps: g = 384, 448, ..., 1024 -> 11 evictions."""
    gen, fired = run_head(1024, 256, 64, lp=128)
    assert [f[0] for f in fired] == list(range(384, 1025, 64))
    assert len(fired) == 11
    for g, before, after, ev in fired:
        assert before.size == 256 + 128 and after.size == 256 + 64 and ev.size == 64


def test_round_invariants():
    K, r, lp = 96, 32, 50
    gen, fired = run_head(2000, K, r, lp=lp, seed=99, layer=3, head_id=7)
    seen_evicted = set()
    for g, before, after, ev in fired:
        n = before.size - r
        # exactly K candidates kept, the r newest untouched, order preserved
        assert after.size == K + r
        np.testing.assert_array_equal(after[K:], before[n:])
        assert np.all(np.diff(after) > 0)
        assert set(after.tolist()) <= set(before.tolist())
        # evicted ordinals are candidates, ascending, complement of the kept ones
        assert np.all(np.diff(ev) > 0) and ev.min() >= 0 and ev.max() < n
        kept = sorted(set(before[:n].tolist()) - set(before[ev].tolist()))
        np.testing.assert_array_equal(after[:K], kept)
        # prompt positions never enter the candidate list; evicted never come back
        assert before.min() >= lp
        assert not (set(after.tolist()) & seen_evicted)
        seen_evicted |= set(before[ev].tolist())
    # cached count stays within [K+r, K+2r) after each step's eviction
    assert K + r <= gen.size < K + 2 * r


def test_no_eviction_below_budget():
    gen, fired = run_head(300, 256, 64)
    assert fired == [] and gen.size == 300


def test_budget_not_multiple_of_r():
    K, r = 100, 64
    gen, fired = run_head(1000, K, r)
    # first firing step: smallest multiple of r with g - r > K
    assert fired[0][0] == 192 and fired[0][3].size == 192 - 64 - 100
    for g, before, after, ev in fired:
        assert after.size == K + r


def test_zero_budget_keeps_only_the_buffer():
    gen, fired = run_head(256, 0, 64)
    for g, before, after, ev in fired:
        np.testing.assert_array_equal(after, before[-64:])


def load_golden():
    rows, approx = [], None
    with open(GOLDEN) as f:
        for line in f:
            t = line.strip()
            if t.startswith("# per_round_approx"):
                parts = t.split()
                approx = (float(parts[2]), float(parts[4]))
            if not t or t.startswith("#"):
                continue
            K, r, n = (int(x) for x in t.split())
            rows.append((K, r, n))
    return rows, approx


def test_paper_per_round_rate():
    rows, (approx, tol) = load_golden()
    K, r, _ = rows[0]
    assert abs(K / (K + r) - approx) < tol


@pytest.mark.parametrize("E", [1, 3, 15, 39, 57])
def test_survival_matches_paper_closed_form(E):
    """Appendix D / Appendix B: a candidate survives n rounds with ((K)/(K+r))^n.
    Track every candidate of round 1 over E rounds in many independent heads."""
    rows, _ = load_golden()
    assert any(n == E for (_, _, n) in rows) or E == 1
    K, r = 1024, 64
    heads = 48
    survived = 0
    tracked = 0
    for h in range(heads):
        # steady state right before a firing step: K+2r cached, g multiple of r
        g = 8192
        gen = np.arange(g - (K + 2 * r), g, dtype=np.int32)
        cand = set(gen[: K + r].tolist())
        tracked += len(cand)
        for e in range(E):
            new, ev = oracle.evict_head(gen, g, K, r, 2024, 5, h)
            gen = new
            g += r
            gen = np.append(gen, np.arange(g - r, g, dtype=np.int32))
        survived += len(cand & set(gen.tolist()))
    p = (K / (K + r)) ** E
    mean = tracked * p
    # exactly K survive per round, which makes counts less variable than binomial
    assert abs(survived - mean) < 5 * np.sqrt(tracked * p * (1 - p)) + 1, (survived, mean)
