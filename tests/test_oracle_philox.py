"""Pins of the oracle's Philox4x32-10 (SC'11) against an independent implementation.

The Random123 known-answer files are not available on this machine, so the
oracle's generator is checked differentially against ATen's header-only
``at::philox_engine`` (BSD source shipped with PyTorch), compiled and run on
the host.  ATen's counter layout: counter = (offset_lo, offset_hi, subseq_lo,
subseq_hi), key = (seed_lo, seed_hi); successive calls return words 0..3.
"""
import os
import subprocess
import tempfile

import numpy as np
import pytest

import oracle

DRIVER = r"""
#include <ATen/core/PhiloxRNGEngine.h>
#include <cstdio>
#include <cstdint>
int main() {
  unsigned long long c0,c1,c2,c3,k0,k1;
  while (scanf("%llu %llu %llu %llu %llu %llu", &c0,&c1,&c2,&c3,&k0,&k1) == 6) {
    uint64_t seed = k0 | (k1 << 32), sub = c2 | (c3 << 32), off = c0 | (c1 << 32);
    at::philox_engine e(seed, sub, off);
    uint32_t a = e(), b = e(), c = e(), d = e();
    printf("%u %u %u %u\n", a, b, c, d);
  }
  return 0;
}
"""


@pytest.fixture(scope="module")
def aten_philox():
    import torch.utils.cpp_extension as ce

    inc = ce.include_paths()[0]
    if not os.path.exists(os.path.join(inc, "ATen", "core", "PhiloxRNGEngine.h")):
        pytest.skip("ATen PhiloxRNGEngine.h not available")
    d = tempfile.mkdtemp(prefix="aten_philox_")
    src = os.path.join(d, "drv.cpp")
    exe = os.path.join(d, "drv")
    with open(src, "w") as f:
        f.write(DRIVER)
    subprocess.check_call(["g++", "-std=c++17", "-O1", "-I" + inc, src, "-o", exe])

    def run(rows):
        inp = "\n".join(" ".join(str(int(x)) for x in r) for r in rows) + "\n"
        out = subprocess.run([exe], input=inp, capture_output=True, text=True, check=True).stdout
        return np.array([[int(t) for t in line.split()] for line in out.strip().splitlines()], dtype=np.uint64)

    return run


def test_philox_matches_aten_edge_and_random(aten_philox):
    rng = np.random.default_rng(1234)
    rows = [[0] * 6, [0xFFFFFFFF] * 6, [1, 0, 0, 0, 0, 0], [0, 0, 0, 0, 1, 0], [0, 0, 0, 1, 0, 0]]
    rows += rng.integers(0, 2**32, size=(300, 6), dtype=np.uint64).tolist()
    ref = aten_philox(rows)
    got = np.array([oracle.philox4x32_10(r[:4], r[4:]) for r in rows], dtype=np.uint64)
    np.testing.assert_array_equal(got, ref)


def test_random_key_counter_layout(aten_philox):
    """The library's mapping: counter (j, step, layer, head_id), key (seed), word 0."""
    seed = 0x0123456789ABCDEF
    cases = [(0, 0, 0, 0), (5, 384, 3, 17), (8255, 32768, 63, 255), (1, 2**31, 255, 4095)]
    rows = [[j, step, layer, hid, seed & 0xFFFFFFFF, seed >> 32] for (j, step, layer, hid) in cases]
    ref = aten_philox(rows)
    for (j, step, layer, hid), r in zip(cases, ref):
        assert oracle.random_key(seed, layer, hid, step, j) == int(r[0])


def test_philox_bits_are_balanced():
    """Each output bit of word 0 over consecutive counters is ~Bernoulli(1/2)."""
    n = 20000
    ks = oracle.random_keys(7, 0, 0, 64, n).astype(np.uint64)
    for bit in range(32):
        p = float(((ks >> np.uint64(bit)) & np.uint64(1)).mean())
        assert abs(p - 0.5) < 5 * 0.5 / np.sqrt(n), (bit, p)
