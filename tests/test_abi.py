"""The C-ABI library loads, exports every symbol include/ra.h declares, and its
host-side validation works without a GPU (no compute calls here)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def ra():
    from paper_2609_03430_gb300 import _build

    _build.build()
    import paper_2609_03430_gb300 as ra

    ra.lib()
    return ra


def declared_functions():
    text = open(os.path.join(ROOT, "include", "ra.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:[\w\s\*]+?)\b(ra_\w+)\s*\(", text, flags=re.M)))


def test_every_declared_symbol_is_exported(ra):
    names = declared_functions()
    assert len(names) >= 20, names
    for n in names:
        assert hasattr(ra.lib(), n), n
        assert n in ra.SIGNATURES, f"binding lacks {n}"


def test_binding_has_no_undeclared_symbols(ra):
    assert set(ra.SIGNATURES) == set(declared_functions())


def test_create_validation_is_host_only(ra):
    L = ra.lib()
    ctx = ctypes.c_void_p()
    cases = [
        ((0, 32, 8, 128, 10, 64, 64, 0), ra.RA_ERR_INVALID_ARG),   # layers
        ((1, 30, 8, 128, 10, 64, 64, 0), ra.RA_ERR_INVALID_ARG),   # q_heads not a multiple
        ((1, 72, 8, 128, 10, 64, 64, 0), ra.RA_ERR_UNSUPPORTED),   # G = 9
        ((1, 32, 8, 64, 10, 64, 64, 0), ra.RA_ERR_UNSUPPORTED),    # head_dim
        ((1, 32, 8, 128, -1, 64, 64, 0), ra.RA_ERR_INVALID_ARG),   # prompt
        ((1, 32, 8, 128, 10, -1, 64, 0), ra.RA_ERR_INVALID_ARG),   # K
        ((1, 32, 8, 128, 10, 64, 0, 0), ra.RA_ERR_INVALID_ARG),    # r
        ((1, 32, 8, 128, 10, 40000, 64, 0), ra.RA_ERR_UNSUPPORTED),  # K + r too large for select
    ]
    for args, code in cases:
        assert L.ra_create(ctypes.byref(ctx), *args) == code, args
        assert ra.ra_last_error(None)
    assert L.ra_create(ctypes.byref(ctx), 2, 32, 8, 128, 10, 64, 64, 0) == ra.RA_OK
    assert ra.ra_device_bytes(ctx) > 0
    # unbound context: every device call is a state error, detected before any CUDA call
    assert L.ra_append_kv(ctx, 0, None, None, None) == ra.RA_ERR_STATE
    assert L.ra_evict(ctx, 0, None, None) == ra.RA_ERR_STATE
    assert L.ra_decode_attn(ctx, 0, None, None, ctypes.c_float(0), None) == ra.RA_ERR_STATE
    assert L.ra_debug_timeout_probe(ctx, ctypes.c_uint64(1000000), None) == ra.RA_ERR_STATE
    assert L.ra_bind(ctx, None, 0, None) == ra.RA_ERR_INVALID_ARG
    assert ra.ra_get_counters(ctx, 0, 1) == (0, 0, 0)
    ra.ra_destroy(ctx)


def test_device_bytes_cover_the_caches(ra):
    # config-2 shape: 36 layers, 16 seqs, 8 KV heads, prompt 512, K 2048, r 64
    ctx = ra.ra_create_batched(36, 32, 8, 128, [512] * 16, 2048, 64, 2)
    # prompts in pages of 192 positions: 512 -> 3 pages
    rows = 36 * 16 * 8 * 3 * 192 + (36 + 1) * 16 * 8 * (2048 + 128)
    assert ra.ra_device_bytes(ctx) >= 2 * rows * 256 + (36 + 1) * 16 * 8 * (2048 + 128) * 4
    assert ra.ra_device_bytes(ctx) < 2 * rows * 256 * 1.01 + (64 << 20)
    ra.ra_destroy(ctx)


def test_scored_policy_sizes_its_buffers_before_bind(ra):
    """The scored policy adds the query window (L*B*KVH*r*G rows), the scores (L*B*KVH*(K+2r) fp32)
    and the pass-1 statistics to the arena; it must be chosen before binding; r*G is capped at 512."""
    L, B, H, KVH, K, r = 4, 3, 32, 8, 256, 64
    ctx = ra.ra_create_batched(L, H, KVH, 128, [100, 0, 700], K, r, 0)
    base = ra.ra_device_bytes(ctx)
    ra.ra_set_policy(ctx, ra.RA_POLICY_SNAPKV)
    grown = ra.ra_device_bytes(ctx)
    window = L * B * KVH * r * (H // KVH) * 256
    scores = L * B * KVH * (K + 2 * r) * 4
    assert grown >= base + window + scores
    assert grown < base + window + scores + (64 << 20)
    ra.ra_set_policy(ctx, ra.RA_POLICY_RANDOM)  # the buffers stay: switching back is allowed
    assert ra.ra_device_bytes(ctx) == grown
    with pytest.raises(ra.RAError) as e:
        ra.ra_set_policy(ctx, 5)
    assert e.value.code == ra.RA_ERR_INVALID_ARG
    ra.ra_destroy(ctx)
    big = ra.ra_create_batched(1, 64, 8, 128, [10], 64, 128, 0)  # r * G = 1024
    with pytest.raises(ra.RAError) as e:
        ra.ra_set_policy(big, ra.RA_POLICY_SNAPKV)
    assert e.value.code == ra.RA_ERR_UNSUPPORTED
    lib = ra.lib()
    assert lib.ra_restore_queries(big, 0, None, ctypes.c_float(0), None) == ra.RA_ERR_STATE  # unbound
    n = ctypes.c_int(0)
    assert lib.ra_get_scores(big, 0, 0, 0, None, 0, ctypes.byref(n), None) == ra.RA_ERR_STATE
    ra.ra_destroy(big)


def test_compaction_mode_validation(ra):
    ctx = ra.ra_create_batched(2, 8, 2, 128, [10], 64, 16, 0)
    ra.ra_set_compaction(ctx, ra.RA_COMPACT_HOLEFILL)
    with pytest.raises(ra.RAError) as e:
        ra.ra_set_policy(ctx, ra.RA_POLICY_SNAPKV)  # pooling needs time-ordered slots
    assert e.value.code == ra.RA_ERR_UNSUPPORTED
    ra.ra_set_compaction(ctx, ra.RA_COMPACT_ORDERED)
    ra.ra_set_policy(ctx, ra.RA_POLICY_SNAPKV)
    with pytest.raises(ra.RAError) as e:
        ra.ra_set_compaction(ctx, ra.RA_COMPACT_HOLEFILL)
    assert e.value.code == ra.RA_ERR_UNSUPPORTED
    with pytest.raises(ra.RAError) as e:
        ra.ra_set_compaction(ctx, 3)
    assert e.value.code == ra.RA_ERR_INVALID_ARG
    ra.ra_destroy(ctx)


def test_no_cpu_fallback_in_product_package():
    """The product package never imports the oracle (test infrastructure)."""
    pkg = os.path.join(ROOT, "paper_2609_03430_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                src = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in src and "from oracle" not in src and "ra_oracle" not in src, f


def test_prompt_pool_sizing_and_admission_validation(ra):
    """The prompt pool is set before binding (pages of 192 positions); admission is refused on
    unbound contexts, and the pool can only grow past what the creation prompts use."""
    L = ra.lib()
    ctx = ra.ra_create_batched(2, 8, 2, 128, [100, 300, 0], 64, 16, 0)
    base = ra.ra_device_bytes(ctx)
    ra.ra_set_prompt_pool(ctx, 4000, 3 * 4000)  # room for three 4000-token prompts
    grown = ra.ra_device_bytes(ctx)
    pages = -(-12000 // 192)
    assert grown >= base + 2 * 2 * 2 * (pages - 3) * 192 * 256  # K and V, 2 layers, 2 heads, extra pages
    ra.ra_set_prompt_pool(ctx, 0, 0)  # never below the creation prompts
    assert ra.ra_device_bytes(ctx) == base
    assert L.ra_admit(ctx, 0, 10, None, None, 10, None) == ra.RA_ERR_STATE  # unbound
    with pytest.raises(ra.RAError) as e:
        ra.ra_set_prompt_pool(ctx, -1, 0)
    assert e.value.code == ra.RA_ERR_INVALID_ARG
    ra.ra_destroy(ctx)
