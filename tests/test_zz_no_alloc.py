"""ra_decode_attn_noalloc: the attention entry point for callers that cannot
hand the library device scratch memory when they call it (for example code
running while another framework owns every device allocation, or inside a
region where cudaMalloc is not allowed).  Its split-K scratch is a fixed
device array inside the library, so the call allocates nothing.

It is called through the C ABI and must give the same result as ra_decode_attn
on two calls in a row -- bit for bit, since it runs the same kernel with the same
split and merge order; only the scratch differs -- and that result is itself within
the attention tolerance of the fp64 oracle elsewhere.  The shared array keeps the
previous call's contents, which must not leak into the next result: before the
compared calls, a call on a context of another shape leaves its own partial
records and counters behind.
This file sorts last so that a stop-at-first-failure run has already run every
other test; it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest

from conftest import cuda_available
from ra_testlib import MAX_ABS, MEAN_REL, Runner, bf16_to_f64

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]


def _close(a_bits, b_bits):
    a, b = bf16_to_f64(a_bits), bf16_to_f64(b_bits)
    err = np.abs(a - b)
    assert err.max() < MAX_ABS and err.sum() / np.abs(b).sum() < MEAN_REL


def test_noalloc_matches_decode_attn_on_two_calls():
    import torch

    import paper_2609_03430_gb300 as ra
    import synth

    run = Runner(L=2, H=40, KVH=8, prompt_lens=[33, 0, 300], K=96, r=32, eseed=3, dseed=8)
    for _ in range(200):  # several evictions per sequence
        run.step()
    lib = ra.lib()
    stream = torch.cuda.current_stream().cuda_stream
    # another shape first (G = 8, long split heads): its partials and counters stay in the array
    other = Runner(L=1, H=16, KVH=2, prompt_lens=[2500, 1200], K=256, r=64, eseed=4, dseed=9)
    for _ in range(3):
        other.step()
    qo = other.up(np.stack([synth.q_rows(9, 0, b, np.arange(16), 7, 128) for b in range(2)]))
    oo = torch.zeros((2, 16, 128), dtype=torch.int16, device="cuda")
    assert lib.ra_decode_attn_noalloc(other.ctx, 0, qo.data_ptr(), oo.data_ptr(), ctypes.c_float(0.0), stream) == 0
    torch.cuda.synchronize()
    other.close()
    for layer in range(run.L):
        for call in range(2):
            q = np.stack([synth.q_rows(8, layer, b, np.arange(run.H), 1000 + call, 128) for b in range(run.B)])
            tq = run.up(q)
            ref = torch.zeros((run.B, run.H, 128), dtype=torch.int16, device="cuda")
            got = torch.full((run.B, run.H, 128), -1, dtype=torch.int16, device="cuda")
            assert lib.ra_decode_attn(run.ctx, layer, tq.data_ptr(), ref.data_ptr(), ctypes.c_float(0.0), stream) == 0
            rc = lib.ra_decode_attn_noalloc(run.ctx, layer, tq.data_ptr(), got.data_ptr(), ctypes.c_float(0.0), stream)
            assert rc == 0, ra.ra_last_error(run.ctx)
            torch.cuda.synchronize()
            assert torch.equal(got, ref), f"layer {layer} call {call}"
            _close(got.cpu().numpy(), ref.cpu().numpy())
    run.close()


def test_noalloc_rejects_layers_beyond_its_scratch():
    import torch

    import paper_2609_03430_gb300 as ra

    # 512 sequences x 4 KV heads x G=8: the partial records alone exceed the fixed 8 MiB array
    cache = ra.RandomAttentionCache(1, 32, 4, 128, [1] * 512, 8, 4, 0)
    q = torch.zeros((512, 32, 128), dtype=torch.int16, device="cuda")
    out = torch.zeros_like(q)
    rc = ra.lib().ra_decode_attn_noalloc(cache.ctx, 0, q.data_ptr(), out.data_ptr(), ctypes.c_float(0.0),
                                         torch.cuda.current_stream().cuda_stream)
    assert rc == ra.RA_ERR_CAPACITY
    assert "scratch" in ra.ra_last_error(cache.ctx)
    cache.close()
