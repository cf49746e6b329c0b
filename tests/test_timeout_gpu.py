"""Failure detection on the device: every mbarrier wait of the pipelines is bounded, and a wait
that runs out flags RA_ERR_DEVICE_TIMEOUT in the context's error word instead of hanging.

The failure is made safely: ra_debug_timeout_probe launches one CTA whose barrier is armed for
bytes that nothing ever sends, with a 1 ms limit on its wait; it touches no memory beyond its own
shared memory and the error word.  The test checks that ra_check_device reports the timeout
exactly once, and that the same context then runs decode steps through an eviction correctly
(bit-exact survivors, attention within tolerance of the oracle).
"""
import ctypes

import pytest

from conftest import cuda_available
from ra_testlib import Runner

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]


def test_bounded_wait_timeout_is_reported_once_and_the_context_stays_usable():
    import torch

    import paper_2609_03430_gb300 as ra

    run = Runner(L=2, H=16, KVH=4, prompt_lens=[40, 7], K=32, r=16, eseed=5, dseed=6)
    for _ in range(70):  # the first eviction fires at g = 64
        run.step(check_attn_layers=(1,))
    run.check_state()
    lib = ra.lib()
    stream = torch.cuda.current_stream().cuda_stream
    assert lib.ra_check_device(run.ctx, stream) == ra.RA_OK
    assert lib.ra_debug_timeout_probe(run.ctx, ctypes.c_uint64(1_000_000), stream) == ra.RA_OK
    assert lib.ra_check_device(run.ctx, stream) == ra.RA_ERR_DEVICE_TIMEOUT
    assert "bounded wait" in ra.ra_last_error(run.ctx)
    assert lib.ra_check_device(run.ctx, stream) == ra.RA_OK  # reported once
    # limits outside [1 us, 100 ms] are refused on the host
    assert lib.ra_debug_timeout_probe(run.ctx, ctypes.c_uint64(10), stream) == ra.RA_ERR_INVALID_ARG
    assert lib.ra_debug_timeout_probe(run.ctx, ctypes.c_uint64(10**9), stream) == ra.RA_ERR_INVALID_ARG
    fired = 0
    for _ in range(40):  # more steps, with evictions, on the same context
        fired += sum(run.step(check_attn_layers=(0, 1)).values())
    assert fired > 0
    run.check_state()
    run.close()  # ra_check_device: nothing new flagged
