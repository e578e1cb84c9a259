"""Pins of the oracle's projection (Section 3, Eq. 1 and Eq. lora), RoPE, and
attention over the reconstruction (Section 3.3)."""
import math
import os

import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _param_rows():
    rows = []
    with open(os.path.join(GOLD, "adapter_params.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                parts = line.split()
                rows.append((parts[0], *map(int, parts[1:5]), parts[5], int(parts[6]),
                             float(parts[7])))
    return rows


@pytest.mark.parametrize("row", _param_rows())
def test_adapter_parameter_counts_match_paper(row):
    model, layers, d_in, q_out, kv_out, place, r, millions = row
    outs = {"Q": q_out, "K": kv_out, "V": kv_out}
    total = layers * sum(O.adapter_params(d_in, outs[p], r) for p in place)
    assert round(total / 1e6, 3) == millions


def test_gemma_adapter_storage_figure():
    """Section 3.4: 21.889M fp32 parameters are 87.6 MB, 1.46% of 6.0 GB."""
    mb = 21.889e6 * 4 / 1e6
    assert round(mb, 1) == 87.6 and round(100 * mb / 6000, 2) == 1.46


def _layer(seed=0, rank=4, B=2, L=5, d_in=48, Hq=4, Hkv=2, D=8):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((B, L, d_in))
    w = rng.standard_normal(((Hq + 2 * Hkv) * D, d_in)) * 0.1
    outs = {"q": Hq * D, "k": Hkv * D, "v": Hkv * D}
    lora = {p: (rng.standard_normal((rank, d_in)) * 0.1,
                rng.standard_normal((outs[p], rank)) * 0.1) for p in "qkv"}
    return x, w, lora, Hq, Hkv, D


def test_lora_zero_b_is_base_projection():
    x, w, lora, Hq, Hkv, D = _layer()
    zero = {p: (a, np.zeros_like(b)) for p, (a, b) in lora.items()}
    none = {p: None for p in "qkv"}
    a = O.project_lora(x, w, zero, 2.0, Hq, Hkv, D, 3, 10000.0)
    b = O.project_lora(x, w, none, 2.0, Hq, Hkv, D, 3, 10000.0)
    for u, v in zip(a, b):
        assert np.array_equal(u, v)


def test_explicit_branch_equals_merged_weight():
    """(alpha/r)(x A^T) B^T == x ((alpha/r) B A)^T: the dense merge W' of Eq. lora."""
    x, w, lora, Hq, Hkv, D = _layer(rank=6)
    alpha_over_r = 2.0
    merged = w.copy()
    lo = 0
    for p, n in (("q", Hq * D), ("k", Hkv * D), ("v", Hkv * D)):
        a, b = lora[p]
        merged[lo:lo + n] += alpha_over_r * b @ a
        lo += n
    none = {p: None for p in "qkv"}
    u = O.project_lora(x, w, lora, alpha_over_r, Hq, Hkv, D, 0, 500000.0)
    v = O.project_lora(x, merged, none, alpha_over_r, Hq, Hkv, D, 0, 500000.0)
    for s, t in zip(u, v):
        assert np.allclose(s, t, rtol=1e-12, atol=1e-12)


def test_projection_layout_is_head_major():
    """Output [B, H, L, D]: head h, position l, channel d comes from row h*D+d."""
    x, w, lora, Hq, Hkv, D = _layer()
    none = {p: None for p in "qkv"}
    q, k, v = O.project_lora(x, w, none, 2.0, Hq, Hkv, D, 0, 0.0)
    assert q.shape == (2, Hq, 5, D) and k.shape == (2, Hkv, 5, D)
    assert np.isclose(q[1, 3, 4, 5], x[1, 4] @ w[3 * D + 5])
    assert np.isclose(k[0, 1, 2, 7], x[0, 2] @ w[(Hq + 1) * D + 7])
    assert np.isclose(v[1, 0, 0, 0], x[1, 0] @ w[(Hq + Hkv) * D])


def test_rope_identity_at_zero_and_norm_preserving():
    rng = np.random.default_rng(0)
    y = rng.standard_normal((1, 2, 6, 64))
    assert np.array_equal(O.rope_rotate_half(y, np.zeros(6), 10000.0), y)
    z = O.rope_rotate_half(y, np.arange(100, 106), 10000.0)
    pair = lambda t: t[..., :32] ** 2 + t[..., 32:] ** 2
    assert np.allclose(pair(z), pair(y))


def test_rope_relative_position():
    """<R_m q, R_n k> depends on m - n only."""
    rng = np.random.default_rng(1)
    q = rng.standard_normal((1, 1, 1, 128))
    k = rng.standard_normal((1, 1, 1, 128))
    dots = []
    for m in (5, 105, 4005):
        qm = O.rope_rotate_half(q, np.array([m]), 500000.0)
        kn = O.rope_rotate_half(k, np.array([m - 3]), 500000.0)
        dots.append(float((qm * kn).sum()))
    assert np.allclose(dots, dots[0], rtol=1e-9)


def test_rope_quarter_turn():
    """Frequency 0 has theta = 1: position pi/2 ... use the D=2 case, where
    a single pair rotates by pos radians."""
    y = np.array([[[[1.0, 0.0]]]])
    z = O.rope_rotate_half(y, np.array([math.pi / 2]), 10000.0)
    assert np.allclose(z[..., 0], 0.0, atol=1e-15) and np.allclose(z[..., 1], 1.0)


@pytest.mark.parametrize("base,thetas", [
    # base^(-2i/D) for D = 8, i = 0..3, written out by hand
    (10000.0, (1.0, 0.1, 0.01, 0.001)),
    (100.0, (1.0, 0.31622776601683794, 0.1, 0.031622776601683794)),   # 100^(-1/4) = 1/sqrt(10)
])
def test_rope_frequency_schedule_hand_worked(base, thetas):
    """The frequency of channel pair i at D = 8 and its pairing partner.

    Rotate-half pairs channel i with channel i + D/2 = i + 4; at position 3 the
    pair turns by 3 theta_i.  A unit vector on channel i must land on
    (cos 3 theta_i) e_i + (sin 3 theta_i) e_(i+4), and one on channel i + 4 on
    -(sin 3 theta_i) e_i + (cos 3 theta_i) e_(i+4).  A schedule of base^(-i/D),
    an interleaved pairing (2i, 2i + 1) or a flipped sign fails here, which the
    invariants (identity at 0, norm, relative position) cannot see."""
    for i, th in enumerate(thetas):
        c, s = math.cos(3 * th), math.sin(3 * th)
        e = np.zeros((1, 1, 1, 8))
        e[..., i] = 1.0
        want = np.zeros(8)
        want[i], want[i + 4] = c, s
        got = O.rope_rotate_half(e, np.array([3]), base)[0, 0, 0]
        assert np.allclose(got, want, rtol=0, atol=1e-15), (i, got, want)
        e = np.zeros((1, 1, 1, 8))
        e[..., i + 4] = 1.0
        want = np.zeros(8)
        want[i], want[i + 4] = -s, c
        got = O.rope_rotate_half(e, np.array([3]), base)[0, 0, 0]
        assert np.allclose(got, want, rtol=0, atol=1e-15), (i + 4, got, want)


def test_rope_second_pair_at_position_one():
    """D = 4, base 10000, position 1: pair (1, 3) turns by 10000^(-1/2) = 0.01 rad
    and pair (0, 2) by 1 rad."""
    y = np.array([[[[0.0, 2.0, 0.0, 0.0]]]])
    z = O.rope_rotate_half(y, np.array([1]), 10000.0)[0, 0, 0]
    assert np.allclose(z, [0.0, 2.0 * math.cos(0.01), 0.0, 2.0 * math.sin(0.01)],
                       rtol=0, atol=1e-15)
    y = np.array([[[[1.0, 0.0, 0.0, 0.0]]]])
    z = O.rope_rotate_half(y, np.array([1]), 10000.0)[0, 0, 0]
    assert np.allclose(z, [math.cos(1.0), 0.0, math.sin(1.0), 0.0], rtol=0, atol=1e-15)


def _sdpa_ref(q, k, v, q_pos, scale):
    """torch's scaled_dot_product_attention in fp64 (library routine)."""
    g = q.shape[1] // k.shape[1]
    kt = torch.from_numpy(np.repeat(k, g, axis=1))
    vt = torch.from_numpy(np.repeat(v, g, axis=1))
    T = k.shape[2]
    mask = torch.from_numpy(np.arange(T)[None, :] <= np.asarray(q_pos)[:, None])
    return torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q), kt, vt, attn_mask=mask, scale=scale).numpy()


@pytest.mark.parametrize("L,T,Hq,Hkv", [(1, 7, 8, 1), (5, 5, 4, 4), (3, 9, 4, 2), (16, 40, 2, 2)])
def test_attention_against_torch_sdpa(L, T, Hq, Hkv):
    rng = np.random.default_rng(L * 100 + T)
    q = rng.standard_normal((2, Hq, L, 16))
    k = rng.standard_normal((2, Hkv, T, 16))
    v = rng.standard_normal((2, Hkv, T, 16))
    pos = np.arange(T - L, T)
    got = O.attention(q, k, v, pos, 0.25)
    assert np.allclose(got, _sdpa_ref(q, k, v, pos, 0.25), rtol=1e-12, atol=1e-12)


def test_attention_special_cases():
    rng = np.random.default_rng(2)
    v = rng.standard_normal((1, 1, 4, 8))
    k = rng.standard_normal((1, 1, 4, 8))
    q = rng.standard_normal((1, 2, 4, 8))
    o = O.attention(q, k, v, np.arange(4), 0.3)
    # the first query sees only key 0: output is v_0 exactly
    assert np.allclose(o[0, :, 0], v[0, 0, 0])
    # identical keys: uniform weights, output is the mean of the visible values
    kk = np.repeat(k[:, :, :1], 4, axis=2)
    o = O.attention(q, kk, v, np.arange(4), 0.3)
    for l in range(4):
        assert np.allclose(o[0, :, l], v[0, 0, :l + 1].mean(0))


def test_float_cache_attention_is_textbook_attention():
    """FLOAT format: attention over the cache equals plain causal attention."""
    c = O.OracleCache(O.FMT_FLOAT, 16, 16, 32, 1, 2, 32, 64, act="f32")
    rng = np.random.default_rng(4)
    k = rng.standard_normal((1, 2, 20, 32)).astype(np.float32)
    v = rng.standard_normal((1, 2, 20, 32)).astype(np.float32)
    c.append(k[:, :, :12], v[:, :, :12])
    c.append(k[:, :, 12:], v[:, :, 12:])
    q = rng.standard_normal((1, 4, 8, 32))
    got = O.attend(c, q)
    ref = _sdpa_ref(q, k.astype(np.float64), v.astype(np.float64), np.arange(12, 20),
                    1 / math.sqrt(32))
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-12)
