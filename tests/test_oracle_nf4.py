"""Pins of the oracle's NF4 base-weight dequantization (the 4-bit NormalFloat
data type of QLoRA, which the paper cites for its frozen NF4 bases; Sections 2,
3.4 and 4)."""
import os

import numpy as np
import pytest

from oracle import kvq_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "nf4_levels.txt")


def _published():
    with open(GOLDEN) as f:
        return np.array([float(l) for l in f if l.strip() and not l.startswith("#")])


def test_levels_match_the_published_table():
    """The published levels are the same construction evaluated in fp32 with
    the probability offset written to seven digits: they agree to about one
    unit of fp32 rounding (the largest difference is 1.1e-7, at level 13)."""
    got = O.nf4_levels()
    ref = _published()
    assert got.shape == (16,)
    # (plausible mistakes move a level far more: the offset taken as 1/32
    # moves one by 2.7e-3; 8 quantiles on each half has no exact zero)
    assert np.max(np.abs(got - ref)) < 2e-7


def test_level_structure():
    v = O.nf4_levels()
    assert np.all(np.diff(v) > 0)
    assert v[0] == -1.0 and v[15] == 1.0 and v[7] == 0.0
    assert (v > 0).sum() == 8 and (v < 0).sum() == 7     # asymmetric: zero is exact


def test_dequant_nibble_order_and_blocks():
    # row 0: byte 0 = 0xF0 -> input 0 is level 0 (-1), input 1 is level 15 (+1);
    # byte 1 = 0x87 -> input 2 is level 7 (0), input 3 is level 8
    codes = np.full((2, 64), 0x77, dtype=np.uint8)       # 128 inputs: two blocks
    codes[0, 0] = 0xF0
    codes[0, 1] = 0x87
    codes[1, 32:] = 0xFF                                  # second block of row 1: all +1
    absmax = np.array([[2.0, 0.5], [3.0, 0.25]])
    w = O.nf4_dequant(codes, absmax)
    lv = O.nf4_levels()
    assert w.shape == (2, 128)
    assert w[0, 0] == -2.0 and w[0, 1] == 2.0 and w[0, 2] == 0.0
    assert np.isclose(w[0, 3], 2.0 * lv[8], rtol=0, atol=1e-9)
    assert np.all(w[0, 4:64] == 0.0) and np.all(w[0, 64:] == 0.0)
    assert np.all(w[1, :64] == 0.0) and np.all(w[1, 64:] == 0.25)


def test_projection_over_a_known_base():
    """All codes 15 (level +1): W is the absmax of each block broadcast, so
    x W^T is the block sums of x weighted by the absmax values."""
    rng = np.random.default_rng(3)
    Hq, Hkv, D, d_in = 2, 1, 64, 128
    n = (Hq + 2 * Hkv) * D
    codes = np.full((n, d_in // 2), 0xFF, dtype=np.uint8)
    absmax = rng.uniform(0.01, 0.1, size=(n, d_in // 64))
    x = rng.standard_normal((1, 3, d_in))
    none = {p: None for p in "qkv"}
    q, k, v = O.project_lora_nf4(x, codes, absmax, none, 2.0, Hq, Hkv, D)
    bsum = x.reshape(1, 3, 2, 64).sum(-1)                  # [1, 3, 2 blocks]
    y = bsum @ absmax.T                                    # [1, 3, n]
    assert np.allclose(q[0, 1, 2], y[0, 2, D:2 * D], rtol=1e-12, atol=1e-12)
    assert np.allclose(v[0, 0, 0], y[0, 0, (Hq + Hkv) * D:], rtol=1e-12, atol=1e-12)
