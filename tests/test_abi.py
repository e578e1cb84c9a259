"""The C-ABI library loads, exports every entry point include/kvq.h declares,
and validates arguments on the host (no GPU needed: nothing here launches)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def kvq():
    from paper_2609_04263_gb300 import build, kvq as K
    build.build()
    K.lib()
    return K


def _declared():
    src = open(os.path.join(ROOT, "include", "kvq.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(kvq_[a-z_]+)\s*\(", src)))


def test_exports_every_declared_symbol(kvq):
    names = _declared()
    assert len(names) >= 12
    so = ctypes.CDLL(kvq.LIB_PATH)
    for n in names:
        assert hasattr(so, n), f"{n} declared in kvq.h but not exported"


def test_binding_names_match_header(kvq):
    for n in _declared():
        assert hasattr(kvq, n), f"binding lacks {n}"


def test_abi_version(kvq):
    assert kvq.kvq_abi_version() == 1


def _desc(kvq, **kw):
    base = dict(fmt=kvq.KVQ_FMT_AFFINE, key_bits=4, value_bits=4, group_size=32,
                residual_tokens=0, sink_tokens=0, norm_iters=8, batch=4, kv_heads=4,
                q_heads=32, head_dim=64, max_tokens=2304, dtype=kvq.KVQ_BF16)
    base.update(kw)
    return kvq.kvq_cache_desc(**base)


def test_cache_bytes_accounts_for_every_plane(kvq):
    d = _desc(kvq)
    n = kvq.kvq_cache_bytes(d)
    B, H, T, D = 4, 4, 2304, 64
    codes = B * H * T * D * 4 // 8
    meta = B * H * T * (D // 32) * 2
    ws = B * 32 * 32 * (D + 2) * 4
    assert n >= 2 * codes + 4 * meta + ws
    assert n <= 2 * codes + 4 * meta + ws + 16 * 256


@pytest.mark.parametrize("kw,status", [
    (dict(fmt=9), 1), (dict(dtype=7), 1), (dict(batch=0), 2),
    (dict(q_heads=30), 2), (dict(head_dim=96), 4), (dict(key_bits=3), 4),
    (dict(group_size=48), 2), (dict(group_size=128), 2),
    (dict(fmt=4, group_size=128, head_dim=256), 4),
])
def test_descriptor_validation(kvq, kw, status):
    d = _desc(kvq, **kw)
    assert kvq.lib().kvq_cache_bytes(ctypes.byref(d)) == 0
    assert kvq.kvq_last_error() != ""
    with pytest.raises(kvq.KvqError) as ei:
        kvq.kvq_create_cache(d, 1 << 20, 1 << 40)
    assert ei.value.status == status


def test_create_view_and_host_validation(kvq):
    d = _desc(kvq, max_tokens=100)
    n = kvq.kvq_cache_bytes(d)
    fake = 1 << 32                         # never dereferenced on the host
    with pytest.raises(kvq.KvqError) as ei:
        kvq.kvq_create_cache(d, fake, n - 1)
    assert ei.value.status == kvq.KVQ_ERR_CAPACITY
    with pytest.raises(kvq.KvqError):
        kvq.kvq_create_cache(d, fake + 16, n)          # misaligned
    h = kvq.kvq_create_cache(d, fake, n)
    try:
        assert kvq.kvq_cache_tokens(h) == 0
        v = kvq.kvq_cache_view(h)
        ptrs = [v.ptr[i] for i in range(kvq.NUM_PLANES) if v.ptr[i]]
        assert all(fake <= p < fake + n and p % 256 == 0 for p in ptrs)
        assert v.dims[0][2] == 128 and v.dims[0][3] == 32 and v.elem_bytes[0] == 1  # rows padded to 64
        # capacity and argument errors are caught before any launch
        with pytest.raises(kvq.KvqError) as ei:
            kvq.kvq_append_pack(h, 1 << 33, 1 << 33, 101, 0)
        assert ei.value.status == kvq.KVQ_ERR_CAPACITY
        with pytest.raises(kvq.KvqError):
            kvq.kvq_append_pack(h, 0, 0, 4, 0)
        with pytest.raises(kvq.KvqError) as ei:
            kvq.kvq_attend_decode(h, 1 << 33, 32, 0.125, 1 << 33, 0)
        assert ei.value.status == kvq.KVQ_ERR_SHAPE        # nothing cached yet
        with pytest.raises(kvq.KvqError) as ei:
            kvq.kvq_attend_prefill(h, 1 << 33, 1, 16, 0.125, 1 << 33, 0)
        assert ei.value.status == kvq.KVQ_ERR_SHAPE        # wrong head count
        assert kvq.kvq_cache_tokens(h) == 0
    finally:
        kvq.kvq_destroy_cache(h)
    assert kvq.kvq_cache_tokens(None) == -1


def test_project_validation(kvq):
    P = 1 << 33
    cases = [
        dict(d_in=100),            # bf16 needs d_in % 64 == 0
        dict(head_dim=80),
        dict(r_q=12),              # bf16 rank must be a multiple of 8
        dict(r_q=80),
        dict(heads=(30, 4)),
        dict(dtype=5),
    ]
    for c in cases:
        hq, hkv = c.get("heads", (32, 4))
        with pytest.raises(kvq.KvqError):
            kvq.kvq_project_lora(P, 1, 4, c.get("d_in", 2048), P, P, P, c.get("r_q", 16), P, P,
                                 16, P, P, 16, 2.0, hq, hkv, c.get("head_dim", 64), 0, None, 1e4,
                                 c.get("dtype", kvq.KVQ_BF16), P, P, P, 0)


def test_append_index_range_is_checked_on_the_host(kvq):
    """Appends whose elements a kernel could not index in 32 bits, or whose
    batch x kv heads exceed the grid's y range, are refused before any launch."""
    fake = 1 << 32
    # batch x kv heads above 65535
    d = _desc(kvq, batch=65536, kv_heads=1, q_heads=1, max_tokens=64)
    h = kvq.kvq_create_cache(d, fake, kvq.kvq_cache_bytes(d))
    try:
        with pytest.raises(kvq.KvqError) as ei:
            kvq.kvq_append_pack(h, 1 << 33, 1 << 33, 1, 0)
        assert ei.value.status == kvq.KVQ_ERR_SHAPE
        assert kvq.kvq_cache_tokens(h) == 0
    finally:
        kvq.kvq_destroy_cache(h)
    # B Hkv (L + G) D / 4 at 2^31: 64 x 8 x (2^17 + 32) x 256 / 4 > 2^31
    d = _desc(kvq, batch=64, kv_heads=8, q_heads=8, head_dim=256, max_tokens=1 << 17)
    h = kvq.kvq_create_cache(d, fake, kvq.kvq_cache_bytes(d))
    try:
        with pytest.raises(kvq.KvqError) as ei:
            kvq.kvq_append_pack(h, 1 << 33, 1 << 33, 1 << 17, 0)
        assert ei.value.status == kvq.KVQ_ERR_SHAPE
        assert kvq.kvq_cache_tokens(h) == 0
    finally:
        kvq.kvq_destroy_cache(h)


def test_project_append_shape_rules_on_the_host(kvq):
    """The fused projection-and-append states which caches it covers and
    refuses the others (and capacity overflows) before any launch."""
    fake = 1 << 32
    P = 1 << 33
    d = _desc(kvq, max_tokens=64)                       # affine 4-bit, G 32, bf16
    h = kvq.kvq_create_cache(d, fake, kvq.kvq_cache_bytes(d))
    try:
        assert kvq.kvq_project_append_supported(h, 32, 2048, 16, 16, 16)
        assert not kvq.kvq_project_append_supported(h, 2, 2048, 16, 16, 16)   # decode rows
        assert not kvq.kvq_project_append_supported(h, 32, 100, 16, 16, 16)   # d_in
        assert not kvq.kvq_project_append_supported(h, 32, 2048, 12, 16, 16)  # rank
        with pytest.raises(kvq.KvqError) as ei:
            kvq.kvq_project_append(h, P, 65, 2048, P, P, P, 16, P, P, 16, P, P, 16, 2.0, 1e4, P, 0)
        assert ei.value.status == kvq.KVQ_ERR_CAPACITY
        with pytest.raises(kvq.KvqError) as ei:
            kvq.kvq_project_append(h, P, 2, 2048, P, P, P, 16, P, P, 16, P, P, 16, 2.0, 1e4, P, 0)
        assert ei.value.status == kvq.KVQ_ERR_UNSUPPORTED
        assert kvq.kvq_cache_tokens(h) == 0
    finally:
        kvq.kvq_destroy_cache(h)
    for kw in (dict(fmt=kvq.KVQ_FMT_KIVI, residual_tokens=32), dict(group_size=64),
               dict(dtype=kvq.KVQ_F32)):
        d = _desc(kvq, max_tokens=64, **kw)
        h = kvq.kvq_create_cache(d, fake, kvq.kvq_cache_bytes(d))
        try:
            assert not kvq.kvq_project_append_supported(h, 32, 2048, 16, 16, 16)
        finally:
            kvq.kvq_destroy_cache(h)
    assert kvq.kvq_project_append_supported(None, 32, 2048, 16, 16, 16) is False


def test_backward_host_rules(kvq):
    """The straight-through backward refuses, before any launch: queries
    beyond the cached tokens, KVarN caches, too small a workspace; the
    adapter backward's workspace is the pre-RoPE gradient plus two rank-wide
    buffers per adapter."""
    fake = 1 << 32
    P = 1 << 33
    d = _desc(kvq, max_tokens=64)
    h = kvq.kvq_create_cache(d, fake, kvq.kvq_cache_bytes(d))
    try:
        assert kvq.kvq_attend_backward_workspace(h, 1, d.q_heads) == 0     # nothing cached
        with pytest.raises(kvq.KvqError) as ei:
            kvq.kvq_attend_backward(h, P, P, 1, d.q_heads, 0.125, P, P, P, P, 1 << 30, 0)
        assert ei.value.status == kvq.KVQ_ERR_SHAPE
    finally:
        kvq.kvq_destroy_cache(h)
    d = _desc(kvq, max_tokens=256, fmt=kvq.KVQ_FMT_KVARN, group_size=64, sink_tokens=16)
    h = kvq.kvq_create_cache(d, fake, kvq.kvq_cache_bytes(d))
    try:
        with pytest.raises(kvq.KvqError) as ei:
            kvq.kvq_attend_backward(h, P, P, 1, d.q_heads, 0.125, P, P, P, P, 1 << 30, 0)
        assert ei.value.status == kvq.KVQ_ERR_UNSUPPORTED
    finally:
        kvq.kvq_destroy_cache(h)
    B, L, Hq, Hkv, D, r = 2, 100, 8, 2, 64, (16, 0, 8)

    def a256(n):
        return (n + 255) // 256 * 256
    d_in = 256
    want = (a256(B * L * (Hq + 2 * Hkv) * D * 4) + sum(2 * a256(B * L * x * 4) for x in r)
            + a256(d_in * (Hq + 2 * Hkv) * D * 2))
    assert kvq.kvq_lora_backward_workspace(B, L, d_in, Hq, Hkv, D, *r) == want
    with pytest.raises(kvq.KvqError) as ei:
        kvq.kvq_lora_backward(P, B, L, 256, P, P, P, 16, None, None, 0, P, P, 8, 2.0, Hq, Hkv, D,
                              0, 1e4, kvq.KVQ_BF16, P, P, P, L, P, P, None, None, P, P, None,
                              P, want - 1, 0)
    assert ei.value.status == kvq.KVQ_ERR_CAPACITY
    with pytest.raises(kvq.KvqError) as ei:                 # kv_rows < L
        kvq.kvq_lora_backward(P, B, L, 256, P, P, P, 16, None, None, 0, P, P, 8, 2.0, Hq, Hkv, D,
                              0, 1e4, kvq.KVQ_BF16, P, P, P, L - 1, P, P, None, None, P, P, None,
                              P, want, 0)
    assert ei.value.status == kvq.KVQ_ERR_SHAPE


def test_ragged_and_paged_layout_rules(kvq):
    """Ragged and paged layouts are built for bf16 affine / symmetric caches
    (G 32, equal 2- or 4-bit keys and values, head_dim 64 or 128); a paged
    cache sizes its planes by the pool, starts with every page free, and
    refuses appends beyond max_tokens before any launch."""
    fake = 1 << 32
    P = 1 << 33
    base = dict(batch=3, kv_heads=2, q_heads=8, head_dim=64, max_tokens=500)
    for kw in (dict(fmt=kvq.KVQ_FMT_KVARN, group_size=64, sink_tokens=16), dict(dtype=kvq.KVQ_F32),
               dict(key_bits=2), dict(group_size=64), dict(head_dim=256)):
        d = _desc(kvq, **{**base, **kw, "layout": kvq.KVQ_LAYOUT_RAGGED})
        with pytest.raises(kvq.KvqError):
            kvq.kvq_cache_bytes(d)
    d = _desc(kvq, **base, layout=kvq.KVQ_LAYOUT_PAGED, num_pages=0)
    with pytest.raises(kvq.KvqError):                       # a pool needs pages
        kvq.kvq_cache_bytes(d)
    d = _desc(kvq, **base, layout=kvq.KVQ_LAYOUT_PAGED, num_pages=5)
    n = kvq.kvq_cache_bytes(d)
    h = kvq.kvq_create_cache(d, fake, n)
    try:
        assert kvq.kvq_free_pages(h) == 5
        assert kvq.kvq_seq_pages(h, 0) == []
        assert kvq.kvq_seq_tokens(h, 2) == 0 and kvq.kvq_seq_tokens(h, 3) == -1
        v = kvq.kvq_cache_view(h)
        assert v.dims[0][0] == 1 and v.dims[0][2] == 5 * kvq.KVQ_PAGE_TOKENS    # the pool
        with pytest.raises(kvq.KvqError) as ei:                    # beyond max_tokens
            kvq.kvq_append_pack_ragged(h, P, P, 600, [600, 0, 0], 0)
        assert ei.value.status == kvq.KVQ_ERR_CAPACITY
        with pytest.raises(kvq.KvqError) as ei:                    # more pages than the pool
            kvq.kvq_append_pack_ragged(h, P, P, 500, [500, 500, 500], 0)
        assert ei.value.status == kvq.KVQ_ERR_CAPACITY
        with pytest.raises(kvq.KvqError) as ei:                    # a count above L
            kvq.kvq_append_pack_ragged(h, P, P, 4, [5, 0, 0], 0)
        assert ei.value.status == kvq.KVQ_ERR_ARG
        assert kvq.kvq_free_pages(h) == 5                           # nothing was taken
    finally:
        kvq.kvq_destroy_cache(h)
    # a ragged cache of the same shape holds B x max_tokens rows and no pool
    d = _desc(kvq, **base, layout=kvq.KVQ_LAYOUT_RAGGED)
    h = kvq.kvq_create_cache(d, fake, kvq.kvq_cache_bytes(d))
    try:
        assert kvq.kvq_free_pages(h) == -1
        v = kvq.kvq_cache_view(h)
        assert v.dims[0][0] == 3 and v.dims[0][2] == 512
    finally:
        kvq.kvq_destroy_cache(h)
