"""Pins of the oracle's scored comparator (section 2, "Baselines as choices of s":
the SnapKV score -- attention from the last w queries, max-pooled over
neighbouring positions -- and a top-K by that score with the prompt pinned).

Each pin checks the oracle against something other than itself: closed forms
(uniform attention of zero queries), a special case that reduces to a library
softmax, exact invariants (every query's weights sum to one; causality),
hand-worked pooling and selection cases, and a library sort.
"""
import numpy as np
import pytest
from scipy.special import softmax

import oracle
import synth


def _bf16(x):
    return synth.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def _rand_qk(rng, n_q, G, n_k, d=16, scale=1.0):
    q = _bf16(rng.standard_normal((n_q, G, d)) * scale)
    k = _bf16(rng.standard_normal((n_k, d)) * scale)
    return q, k


def test_zero_queries_give_uniform_weights():
    """q = 0: each query spreads weight 1 uniformly over the keys it may see, so
    score_i = G * sum_u [pos_i <= qpos_u] / #{i' : pos_i' <= qpos_u}."""
    G, n_k, d = 3, 11, 8
    q = np.zeros((4, G, d), np.uint16)
    k_pos = np.arange(n_k, dtype=np.int32)
    q_pos = np.array([6, 7, 8, 9], np.int32)
    k = _bf16(np.random.default_rng(0).standard_normal((n_k, d)))
    got = oracle.window_scores(q, q_pos, k, k_pos)
    want = np.zeros(n_k)
    for qp in q_pos:
        vis = k_pos <= qp
        want[vis] += G / vis.sum()
    np.testing.assert_allclose(got, want, rtol=1e-14, atol=0)


def test_single_query_all_visible_is_library_softmax():
    """One query head, every key visible: the score is the softmax of the scaled dot products."""
    rng = np.random.default_rng(1)
    d, n_k = 32, 19
    q, k = _rand_qk(rng, 1, 1, n_k, d)
    scale = 0.37
    qf = synth.bf16_bits_to_f32(q).astype(np.float64)[0, 0]
    kf = synth.bf16_bits_to_f32(k).astype(np.float64)
    want = softmax(scale * (kf @ qf))
    got = oracle.window_scores(q, [100], k, np.arange(n_k), scale)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-15)


def test_default_scale_is_inverse_sqrt_d():
    rng = np.random.default_rng(2)
    q, k = _rand_qk(rng, 2, 2, 9, 64)
    np.testing.assert_allclose(oracle.window_scores(q, [20, 21], k, np.arange(9)),
                               oracle.window_scores(q, [20, 21], k, np.arange(9), 1 / 8.0), rtol=1e-15)


def test_weights_sum_to_queries_times_heads():
    """Every (query, head) softmax sums to one over the keys it sees."""
    rng = np.random.default_rng(3)
    n_q, G, n_k = 6, 4, 40
    q, k = _rand_qk(rng, n_q, G, n_k, 16, 2.0)
    k_pos = np.arange(n_k) + 5
    q_pos = np.arange(n_q) + 38  # the first queries see fewer keys
    s = oracle.window_scores(q, q_pos, k, k_pos)
    assert s.sum() == pytest.approx(n_q * G, rel=1e-13)
    assert (s >= 0).all()


def test_causal_mask():
    """A key after every query gets nothing; a key only the newest query sees gets only its weight."""
    rng = np.random.default_rng(4)
    G, n_k = 2, 12
    q, k = _rand_qk(rng, 3, G, n_k)
    k_pos = np.arange(n_k, dtype=np.int32)
    q_pos = np.array([8, 9, 10], np.int32)
    s = oracle.window_scores(q, q_pos, k, k_pos)
    assert s[11] == 0.0
    last = oracle.window_scores(q[2:], q_pos[2:], k, k_pos)  # the newest query alone
    assert s[10] == pytest.approx(last[10], rel=1e-14)
    # the three queries each contribute independently: the sum over the window is additive
    parts = sum(oracle.window_scores(q[u:u + 1], q_pos[u:u + 1], k, k_pos) for u in range(3))
    np.testing.assert_allclose(s, parts, rtol=1e-13, atol=1e-16)


def test_scale_and_query_doubling_agree():
    """Doubling q (exact in bf16) equals doubling the scale."""
    rng = np.random.default_rng(5)
    q, k = _rand_qk(rng, 3, 2, 25)
    q2 = _bf16(2.0 * synth.bf16_bits_to_f32(q))
    a = oracle.window_scores(q2, [30, 31, 32], k, np.arange(25), 0.3)
    b = oracle.window_scores(q, [30, 31, 32], k, np.arange(25), 0.6)
    np.testing.assert_allclose(a, b, rtol=1e-13, atol=1e-16)


def test_dominant_key_takes_the_weight():
    d, n_k, G, n_q = 16, 10, 3, 4
    k = np.zeros((n_k, d), np.float32)
    k[6, 0] = 4.0
    q = np.zeros((n_q, G, d), np.float32)
    q[:, :, 0] = 4.0
    s = oracle.window_scores(_bf16(q), np.full(n_q, 50), _bf16(k), np.arange(n_k), 1.0)
    # logit 16 against 0: weight e^16 / (e^16 + 9) per query head
    w = np.exp(16.0) / (np.exp(16.0) + 9.0)
    assert s[6] == pytest.approx(n_q * G * w, rel=1e-13)
    assert s[0] == pytest.approx(n_q * G * (1 - w) / 9, rel=1e-12)


def test_max_pool_hand_cases():
    s = [0, 0, 0, 5, 0, 0, 0, 0, 0, 1]
    np.testing.assert_array_equal(oracle.max_pool(s, 3), [5, 5, 5, 5, 5, 5, 5, 1, 1, 1])
    np.testing.assert_array_equal(oracle.max_pool(s, 0), s)
    np.testing.assert_array_equal(oracle.max_pool(s, 1), [0, 0, 5, 5, 5, 0, 0, 0, 1, 1])
    np.testing.assert_array_equal(oracle.max_pool(s, 20), [5] * 10)
    assert oracle.max_pool([], 3).size == 0
    rng = np.random.default_rng(6)
    x = rng.random(50)
    assert (oracle.max_pool(x, 3) >= x).all()


def test_select_top_hand_cases_and_library_sort():
    # ties go to the earlier position
    np.testing.assert_array_equal(oracle.select_top([3, 1, 3, 2, 3], 2), [0, 2])
    np.testing.assert_array_equal(oracle.select_top([3, 1, 3, 2, 3], 4), [0, 2, 3, 4])
    assert oracle.select_top([1, 2], 0).size == 0
    np.testing.assert_array_equal(oracle.select_top([1, 2, 0], 3), [0, 1, 2])
    with pytest.raises(ValueError):
        oracle.select_top([1, 2], 3)
    rng = np.random.default_rng(7)
    for _ in range(20):
        n = int(rng.integers(1, 60))
        s = rng.integers(0, 6, n).astype(np.float64)  # many ties
        K = int(rng.integers(0, n + 1))
        want = np.sort(np.lexsort((np.arange(n), -s))[:K])
        np.testing.assert_array_equal(oracle.select_top(s, K), want)


def test_scored_round_cadence_and_spike():
    """Same trigger as the random policy; a single spike keeps its pooled neighbourhood."""
    K, r = 7, 4
    gen = np.arange(100, 100 + K + 2 * r, dtype=np.int32)  # c = K + 2r at g = 16: fires (16 % 4 == 0)
    n = gen.size - r
    raw = np.zeros(n)
    raw[5] = 1.0
    new, ev = oracle.evict_head_scored(gen, 16, K, r, raw, radius=3)
    np.testing.assert_array_equal(new[:K], gen[2:9])  # candidates 2..8 pooled to 1.0
    np.testing.assert_array_equal(new[K:], gen[n:])   # the buffer is untouched
    np.testing.assert_array_equal(ev, [0, 1, 9, 10])
    same, none = oracle.evict_head_scored(gen, 15, K, r, raw)  # 15 % r != 0: no round
    np.testing.assert_array_equal(same, gen)
    assert none.size == 0


def test_scored_round_with_increasing_scores_is_recency():
    """Scores increasing with position and no pooling keep the K newest candidates: the recency policy."""
    K, r, g = 20, 8, 48
    gen = np.arange(3, 3 + K + 2 * r, dtype=np.int32)
    n = gen.size - r
    new, ev = oracle.evict_head_scored(gen, g, K, r, np.linspace(0.1, 1.0, n), radius=0)
    rec, ev_rec = oracle.evict_head_policy(gen, g, K, r, 0, 0, 0, 1, 0, oracle.POLICY_RECENCY)
    np.testing.assert_array_equal(new, rec)
    np.testing.assert_array_equal(ev, ev_rec)
