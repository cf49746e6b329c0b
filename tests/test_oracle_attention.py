"""Pins of the oracle's fp64 decode attention (section 2, 'Notation'):
closed forms and an independent library softmax attention in fp64."""
import numpy as np
import pytest

import oracle
import synth


def bf16(x):
    return synth.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def f(x):
    return synth.bf16_bits_to_f32(x).astype(np.float64)


def rand_bf16(rng, shape, s=1.0):
    return bf16(rng.standard_normal(shape) * s)


def test_zero_query_gives_mean_of_values():
    rng = np.random.default_rng(1)
    k, v = rand_bf16(rng, (37, 64)), rand_bf16(rng, (37, 64))
    q = bf16(np.zeros((3, 64)))
    out = oracle.attend(q, k, v)
    np.testing.assert_allclose(out, np.broadcast_to(f(v).mean(0), out.shape), rtol=0, atol=1e-12)


def test_single_slot_gives_its_value():
    rng = np.random.default_rng(2)
    q, k, v = rand_bf16(rng, (4, 128)), rand_bf16(rng, (1, 128)), rand_bf16(rng, (1, 128))
    np.testing.assert_allclose(oracle.attend(q, k, v), np.broadcast_to(f(v)[0], (4, 128)), atol=1e-12)


def test_identical_keys_give_mean_of_values():
    rng = np.random.default_rng(3)
    k = np.repeat(rand_bf16(rng, (1, 128)), 50, axis=0)
    v = rand_bf16(rng, (50, 128))
    q = rand_bf16(rng, (2, 128))
    np.testing.assert_allclose(oracle.attend(q, k, v), np.broadcast_to(f(v).mean(0), (2, 128)), atol=1e-12)


def test_planted_key_dominates():
    rng = np.random.default_rng(4)
    d = 128
    q = bf16(np.full((1, d), 1.0))
    k = rand_bf16(rng, (30, d), 0.01)
    k[17] = bf16(np.full(d, 8.0))  # logit gap ~ 8*128/sqrt(128) ~ 90
    v = rand_bf16(rng, (30, d))
    np.testing.assert_allclose(oracle.attend(q, k, v), f(v)[17:18], atol=1e-12)


def test_two_slots_logistic_closed_form():
    d = 64
    rng = np.random.default_rng(5)
    q, k, v = rand_bf16(rng, (1, d)), rand_bf16(rng, (2, d)), rand_bf16(rng, (2, d))
    s = f(k) @ f(q)[0] / np.sqrt(d)
    w = 1.0 / (1.0 + np.exp(s[1] - s[0]))
    np.testing.assert_allclose(oracle.attend(q, k, v)[0], w * f(v)[0] + (1 - w) * f(v)[1], rtol=1e-13, atol=1e-13)


def test_explicit_scale():
    rng = np.random.default_rng(6)
    q, k, v = rand_bf16(rng, (2, 32)), rand_bf16(rng, (9, 32)), rand_bf16(rng, (9, 32))
    a = oracle.attend(q, k, v, scale=0.5)
    s = f(q) @ f(k).T * 0.5
    p = np.exp(s - s.max(1, keepdims=True))
    p /= p.sum(1, keepdims=True)
    np.testing.assert_allclose(a, p @ f(v), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("n,G,d", [(1, 1, 64), (7, 4, 128), (300, 5, 128), (1000, 8, 128)])
def test_matches_library_sdpa_fp64(n, G, d):
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(n + G)
    q, k, v = rand_bf16(rng, (G, d)), rand_bf16(rng, (n, d), 2.0), rand_bf16(rng, (n, d))
    out = oracle.attend(q, k, v)
    tq = torch.from_numpy(f(q)).reshape(1, 1, G, d)
    tk = torch.from_numpy(f(k)).reshape(1, 1, n, d)
    tv = torch.from_numpy(f(v)).reshape(1, 1, n, d)
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv).reshape(G, d).numpy()
    np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)


def test_empty_cache_gives_zero():
    out = oracle.attend(bf16(np.ones((2, 8))), np.zeros((0, 8), np.uint16), np.zeros((0, 8), np.uint16))
    assert np.all(out == 0)
