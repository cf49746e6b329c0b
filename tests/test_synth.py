"""Checks of the shared synthetic-input generator (host side)."""
import numpy as np
import pytest

import synth


def test_bf16_rounding_matches_torch_rne():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(20000).astype(np.float32),
                        np.array([1.0 + 2**-8, 1.0 + 3 * 2**-8, -1.0 - 2**-8, 0.0, -0.0], np.float32)])
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(synth.f32_to_bf16_bits(x), ref)


def test_values_are_standard_normal_like():
    v = synth.bf16_bits_to_f32(synth.kv_rows(1, 0, 0, 0, 0, np.arange(4000), 128)).astype(np.float64)
    assert abs(v.mean()) < 0.01 and abs(v.std() - 1.0) < 0.01
    assert np.abs(v).max() < 6.0


def test_streams_and_positions_differ_and_repeat():
    a = synth.kv_rows(5, 0, 1, 2, 3, [10, 11], 64)
    b = synth.kv_rows(5, 1, 1, 2, 3, [10, 11], 64)
    c = synth.kv_rows(5, 0, 1, 2, 3, [10, 11], 64)
    assert not np.array_equal(a, b)
    assert not np.array_equal(a[0], a[1])
    np.testing.assert_array_equal(a, c)
    np.testing.assert_array_equal(synth.kv_rows(5, 0, 1, 2, 3, [11], 64)[0], a[1])


def test_key_scale_is_lognormal():
    s = synth.key_channel_scale(2, 36, 8, 128).astype(np.float64)
    z = np.log(s)
    assert abs(z.mean()) < 0.02 and abs(z.std() - 0.5) < 0.02


def test_uniform_ints_range_and_repeat():
    a = synth.uniform_ints(5, 1000, 256, 4096)
    assert a.min() >= 256 and a.max() <= 4096
    np.testing.assert_array_equal(a, synth.uniform_ints(5, 1000, 256, 4096))
