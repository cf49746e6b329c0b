"""Pins of the oracle's selection (Eq. 1 with section 3's uniform scores).

Checked against what the mathematics fixes: a uniform K-subset of N candidates
(brute force over all C(N, K) subsets), per-slot inclusion K/N, pairwise
co-inclusion K(K-1)/(N(N-1)), independence across heads, tie-breaking by the
lower ordinal, and an independent definition (lexicographic sort) of
"the K smallest (key, ordinal)".
"""
import itertools

import numpy as np
import pytest

import oracle


def chi2_stat(obs, exp):
    obs = np.asarray(obs, dtype=np.float64)
    exp = np.asarray(exp, dtype=np.float64)
    return float(((obs - exp) ** 2 / exp).sum())


# 0.999 quantiles of chi-square (scipy computes them; kept as a fallback-free check)
def chi2_crit(dof, q=0.9995):
    from scipy.stats import chi2

    return float(chi2.ppf(q, dof))


def test_select_matches_lexsort_definition():
    rng = np.random.default_rng(0)
    for n, K in [(1, 1), (2, 1), (10, 0), (10, 10), (320, 256), (2112, 2048), (777, 13)]:
        keys = rng.integers(0, 2**32, size=n, dtype=np.uint64).astype(np.uint32)
        got = oracle.select_keep(keys, K)
        order = np.lexsort((np.arange(n), keys))  # primary key: keys, secondary: ordinal
        ref = np.sort(order[:K]).astype(np.int32)
        np.testing.assert_array_equal(got, ref)


def test_select_ties_keep_lower_ordinal():
    keys = np.array([5, 3, 5, 5, 1, 5], dtype=np.uint32)
    # sorted (key, j): (1,4) (3,1) (5,0) (5,2) (5,3) (5,5) -> keep 4 = {0,1,2,4}
    np.testing.assert_array_equal(oracle.select_keep(keys, 4), [0, 1, 2, 4])
    keys = np.zeros(7, dtype=np.uint32)
    np.testing.assert_array_equal(oracle.select_keep(keys, 3), [0, 1, 2])


def test_select_rejects_bad_args():
    with pytest.raises(ValueError):
        oracle.select_keep(np.zeros(3, dtype=np.uint32), 4)


def test_brute_force_uniform_subsets_small_n():
    """N=6, K=4: all 15 subsets equiprobable over independent draws (step varies)."""
    N, K = 6, 4
    subsets = {s: i for i, s in enumerate(itertools.combinations(range(N), K))}
    counts = np.zeros(len(subsets))
    draws = 15000
    for step in range(draws):
        keys = oracle.random_keys(11, 2, 5, step, N)
        counts[subsets[tuple(oracle.select_keep(keys, K))]] += 1
    exp = np.full(len(subsets), draws / len(subsets))
    assert chi2_stat(counts, exp) < chi2_crit(len(subsets) - 1)


def test_inclusion_and_coinclusion_rates():
    N, K = 40, 30
    rounds = 4000
    incl = np.zeros(N)
    pair = 0.0
    for step in range(rounds):
        keep = oracle.select_keep(oracle.random_keys(3, 0, 9, 64 * step, N), K)
        mask = np.zeros(N, dtype=bool)
        mask[keep] = True
        incl += mask
        pair += mask[0] and mask[N - 1]
    # per-slot inclusion K/N (chi-square on the N slot counts, each slot kept ~Bin(rounds, K/N))
    p = K / N
    z = (incl - rounds * p) / np.sqrt(rounds * p * (1 - p))
    assert float((z**2).sum()) < chi2_crit(N)
    # pairwise co-inclusion within a head: K(K-1)/(N(N-1))
    q = K * (K - 1) / (N * (N - 1))
    assert abs(pair / rounds - q) < 5 * np.sqrt(q * (1 - q) / rounds)


def test_heads_draw_independently():
    """Different KV heads (different head_id in the counter) draw independent keep-sets:
    co-inclusion of the same slot across two heads is (K/N)^2."""
    N, K = 50, 25
    rounds = 4000
    both = 0
    for step in range(rounds):
        a = oracle.select_keep(oracle.random_keys(5, 1, 0, step, N), K)
        b = oracle.select_keep(oracle.random_keys(5, 1, 1, step, N), K)
        both += (7 in set(a.tolist())) and (7 in set(b.tolist()))
    q = (K / N) ** 2
    assert abs(both / rounds - q) < 5 * np.sqrt(q * (1 - q) / rounds)
