"""Pins of the oracle's physical incremental cache (Section 3.1) for each format.

Invariants that any correct implementation has: chunked appends give the same
bytes as one append, full-precision windows hold the input bit for bit, the
KIVI split point follows its closed form, a format with everything held at
full precision reconstructs the input exactly, and per-channel key groups sit
on an exact grid when the input does.
"""
import numpy as np
import pytest

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth

AFFINE, SYM, KIVI, KVARN, FLOAT = O.FMT_AFFINE, O.FMT_SYMMETRIC, O.FMT_KIVI, O.FMT_KVARN, O.FMT_FLOAT


def _cache(fmt, **kw):
    base = dict(key_bits=4, value_bits=4, group_size=32, batch=2, kv_heads=2,
                head_dim=64, max_tokens=400, act="bf16")
    if fmt == KIVI:
        base.update(key_bits=2, value_bits=2, residual_tokens=64)
    if fmt == KVARN:
        base.update(key_bits=4, value_bits=2, group_size=16, sink_tokens=24,
                    norm_iters=8, head_dim=64)
    if fmt == SYM:
        base.update(key_bits=2, value_bits=2)
    base.update(kw)
    return O.OracleCache(fmt, **base)


def _kv(c, T, seed=0):
    shp = (c.B, c.H, T, c.D)
    k = O.round_to(synth.kv_states(shp, seed=seed, stream=0), "bf16")
    v = O.round_to(synth.kv_states(shp, seed=seed, stream=1), "bf16")
    return k, v


def _live_planes(c):
    """The planes restricted to the rows that hold live tokens."""
    P, T, G = c.planes, c.T, c.G
    out = {}
    for name, arr in P.items():
        if c.fmt == KIVI and name.endswith("_full"):
            ring = c.R + G
            tq = O.kivi_quantized_prefix(T, c.R, G)
            out[name] = np.stack([arr[:, :, t % ring] for t in range(tq, T)], 2)
        elif c.fmt == KIVI and name == "k_scale" or c.fmt == KIVI and name == "k_zero":
            out[name] = arr[:, :, :O.kivi_quantized_prefix(T, c.R, G) // G]
        elif c.fmt == KIVI:
            out[name] = arr[:, :, :O.kivi_quantized_prefix(T, c.R, G)]
        elif c.fmt == KVARN and name.endswith("_pend"):
            nb = O.kvarn_blocks(T, c.S, G)
            out[name] = np.stack([arr[:, :, (t - c.S) % G]
                                  for t in range(c.S + nb * G, T)] or
                                 [np.zeros(arr.shape[:2] + arr.shape[3:])], 2)
        elif c.fmt == KVARN and name.endswith("_col"):
            out[name] = arr[:, :, :O.kvarn_blocks(T, c.S, G)]
        elif c.fmt == KVARN and name.endswith("_full"):
            out[name] = arr[:, :, :min(T, c.S)]
        elif c.fmt == KVARN:
            out[name] = arr[:, :, :O.kvarn_blocks(T, c.S, G) * G]
        else:
            out[name] = arr[:, :, :T]
    return out


@pytest.mark.parametrize("fmt", [FLOAT, AFFINE, SYM, KIVI, KVARN])
@pytest.mark.parametrize("chunks", [[300], [128, 128, 44], [1] * 7 + [293], [37, 1, 100, 162]])
def test_chunking_invariance(fmt, chunks):
    """The cache after T tokens is a function of T only (Section 3.1 appends
    in 128-token chunks during evaluation; any split gives the same bytes)."""
    T = sum(chunks)
    ref = _cache(fmt)
    k, v = _kv(ref, T)
    ref.append(k, v)
    c = _cache(fmt)
    t = 0
    for n in chunks:
        c.append(k[:, :, t:t + n], v[:, :, t:t + n])
        t += n
    a, b = _live_planes(ref), _live_planes(c)
    assert a.keys() == b.keys()
    for name in a:
        assert np.array_equal(a[name].view(np.uint8), b[name].view(np.uint8)), name


@pytest.mark.parametrize("T", [0, 31, 32, 63, 64, 65, 95, 96, 97, 200])
def test_kivi_split_closed_form(T):
    R, G = 64, 32
    tq = O.kivi_quantized_prefix(T, R, G)
    assert tq % G == 0 and tq <= max(T - R, 0)
    assert T - tq < R + G                  # residual never exceeds R + G - 1
    if T >= R:
        assert T - tq >= R                  # and keeps at least R tokens


def test_kivi_residual_holds_input_bitwise():
    c = _cache(KIVI)
    k, v = _kv(c, 250)
    c.append(k[:, :, :100], v[:, :, :100])
    c.append(k[:, :, 100:], v[:, :, 100:])
    kh, vh = c.reconstruct()
    tq = O.kivi_quantized_prefix(250, 64, 32)
    assert np.array_equal(kh[:, :, tq:], k[:, :, tq:].astype(np.float64))
    assert np.array_equal(vh[:, :, tq:], v[:, :, tq:].astype(np.float64))
    # and the quantized prefix differs from the input (it is really coded)
    assert not np.array_equal(kh[:, :, :tq], k[:, :, :tq].astype(np.float64))


def test_kivi_window_covering_everything_is_float_attention():
    c = _cache(KIVI, residual_tokens=400)
    f = _cache(FLOAT)
    k, v = _kv(c, 300)
    c.append(k, v)
    f.append(k, v)
    q = synth.queries((2, 4, 5, 64))
    assert np.array_equal(O.attend(c, q), O.attend(f, q))


def test_kivi_keys_are_per_channel_groups():
    """Keys on an exact per-channel grid (each channel its own power-of-two
    step and offset over a 32-token block) are recovered exactly, while the
    per-token value quantizer of the same data is not exact."""
    c = _cache(KIVI, residual_tokens=0, batch=1, kv_heads=1)
    rng = np.random.default_rng(3)
    D = 64
    step = 2.0 ** rng.integers(-4, 0, D)
    off = rng.integers(-8, 8, D) * 0.25
    k = np.zeros((1, 1, 64, D), np.float32)
    for blk in range(2):
        codes = rng.integers(0, 4, (32, D))
        codes[0], codes[1] = 0, 3
        k[0, 0, blk * 32:(blk + 1) * 32] = off + codes * step
    c.append(k, k)
    kh, vh = c.reconstruct()
    assert np.array_equal(kh, k.astype(np.float64))
    assert not np.array_equal(vh, k.astype(np.float64))


def test_kvarn_sinks_and_pending_hold_input_bitwise():
    c = _cache(KVARN)
    k, v = _kv(c, 24 + 16 * 3 + 5)
    c.append(k, v)
    kh, vh = c.reconstruct()
    T = k.shape[2]
    nb = O.kvarn_blocks(T, 24, 16)
    assert nb == 3
    full = list(range(24)) + list(range(24 + nb * 16, T))
    assert np.array_equal(kh[:, :, full], k[:, :, full].astype(np.float64))
    assert np.array_equal(vh[:, :, full], v[:, :, full].astype(np.float64))
    # quantized blocks reconstruct close to the input (4-bit keys, 2-bit values)
    blk = slice(24, 24 + nb * 16)
    rel_k = np.linalg.norm(kh[:, :, blk] - k[:, :, blk]) / np.linalg.norm(k[:, :, blk])
    rel_v = np.linalg.norm(vh[:, :, blk] - v[:, :, blk]) / np.linalg.norm(v[:, :, blk])
    assert rel_k < 0.12 and rel_v < 0.45


@pytest.mark.parametrize("fmt,bits,tol", [(AFFINE, 4, 0.12), (AFFINE, 2, 0.6),
                                          (SYM, 2, 0.8), (SYM, 4, 0.25), (AFFINE, 8, 0.01)])
def test_reconstruction_error_by_bits(fmt, bits, tol):
    c = _cache(fmt, key_bits=bits, value_bits=bits)
    k, v = _kv(c, 96)
    c.append(k, v)
    kh, _ = c.reconstruct()
    rel = np.linalg.norm(kh - k) / np.linalg.norm(k)
    assert rel < tol


def test_capacity_is_enforced():
    c = _cache(AFFINE, max_tokens=64)
    k, v = _kv(c, 65)
    with pytest.raises(ValueError):
        c.append(k, v)
