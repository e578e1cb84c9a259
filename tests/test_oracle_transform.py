"""Pins of the oracle's KVarN pieces: the fixed normalised Hadamard transform
and dual-axis variance normalisation (Sections 2 and 3.1)."""
import math

import numpy as np
import pytest
import scipy.linalg

from oracle import kvq_oracle as O


@pytest.mark.parametrize("D", [2, 8, 64, 128, 256])
def test_fwht_equals_sylvester_matrix(D):
    """Against scipy's Sylvester-construction Hadamard matrix (library)."""
    rng = np.random.default_rng(D)
    x = rng.standard_normal((16, D)).astype(np.float32)
    ref = x.astype(np.float64) @ scipy.linalg.hadamard(D).T / math.sqrt(D)
    got = O.fwht_f32(x)
    assert got.dtype == np.float32
    assert np.max(np.abs(got - ref)) <= 1e-5 * np.max(np.abs(ref))
    assert np.allclose(O.hadamard_matrix(D), scipy.linalg.hadamard(D) / math.sqrt(D))


@pytest.mark.parametrize("D", [64, 256])
def test_fwht_orthogonal_and_norm_preserving(D):
    rng = np.random.default_rng(7)
    x = rng.standard_normal((32, D)).astype(np.float32)
    y = O.fwht_f32(x)
    assert np.allclose(np.linalg.norm(y, axis=1), np.linalg.norm(x, axis=1), rtol=1e-5)
    assert np.max(np.abs(O.fwht_f32(y) - x)) < 1e-5
    H = O.hadamard_matrix(D)
    assert np.allclose(H @ H, np.eye(D), atol=1e-12)


def test_fwht_power_of_two_scale_is_exact():
    """With D = 256 the normalisation 1/16 is exact, so integer inputs give
    exact dyadic outputs: e_0 maps to the constant 1/16 vector."""
    e0 = np.zeros((1, 256), np.float32)
    e0[0, 0] = 1
    assert np.all(O.fwht_f32(e0) == np.float32(1 / 16))


def test_tree_sum_order():
    """The stride-halving tree: ((a0+a2)+(a1+a3)) for n = 4, checked on values
    where a different order rounds differently."""
    a = np.array([1.0, 2.0 ** -24, -1.0, 2.0 ** -24], np.float32)
    # (1 + -1) + (2^-24 + 2^-24) = 2^-23 exactly
    assert O.tree_sum_f32(a) == np.float32(2.0 ** -23)
    b = np.array([1.0, 2.0 ** -24, 2.0 ** -24, -1.0], np.float32)
    # (1 + 2^-24) + (2^-24 - 1) = 1 + (-1 + 2^-24) = 2^-24 (1 + 2^-24 rounds to 1)
    assert O.tree_sum_f32(b) == np.float32(2.0 ** -24)


def test_davn_normalises_both_axes():
    rng = np.random.default_rng(11)
    y = (rng.standard_normal((64, 256)) * np.exp(rng.normal(0, 1, (64, 1)))
         * np.exp(rng.normal(0, 1, (1, 256)))).astype(np.float32)
    out, r, c = O.davn_f32(y, 8)
    row_rms = np.sqrt((out.astype(np.float64) ** 2).mean(1))
    col_rms = np.sqrt((out.astype(np.float64) ** 2).mean(0))
    assert np.max(np.abs(col_rms - 1)) < 1e-5     # the last step is on columns
    assert np.max(np.abs(row_rms - 1)) < 0.05
    # the scales reproduce the input
    rec = r.astype(np.float64)[:, None] * c.astype(np.float64)[None, :] * out
    assert np.max(np.abs(rec - y) / (np.abs(y) + 1e-6)) < 1e-4


def test_davn_zero_iterations_is_identity():
    y = np.random.default_rng(0).standard_normal((64, 64)).astype(np.float32)
    out, r, c = O.davn_f32(y, 0)
    assert np.array_equal(out, y) and np.all(r == 1) and np.all(c == 1)


@pytest.mark.parametrize("bits", [2, 4])
def test_kvarn_reduces_to_affine_without_rotation_and_normalisation(bits):
    """Special case: no rotation and zero normalisation iterations leaves the
    plain grouped affine quantizer of Eq. (affine), bit for bit."""
    x = np.random.default_rng(5).standard_normal((64, 256)).astype(np.float32)
    c, s, m, r, cc = O.kvarn_block_quant(x, bits, 64, 0, rotate=False)
    c2, s2, m2 = O.affine_quant(x.reshape(64, 4, 64), bits)
    assert np.array_equal(c, c2.reshape(64, 256))
    assert np.array_equal(s.view(np.uint16), s2.view(np.uint16))
    assert np.array_equal(m.view(np.uint16), m2.view(np.uint16))
    assert np.all(r == 1) and np.all(cc == 1)


def test_kvarn_block_error_scales_with_row_col_scales():
    """Reconstruction error of a block stays within r_i c_j (s/2 + metadata
    rounding) plus fp16 rounding of r and c."""
    rng = np.random.default_rng(9)
    x = (rng.standard_normal((64, 256)) * np.exp(rng.normal(0, 0.5, (1, 256)))).astype(np.float32)
    for bits in (2, 4):
        c, s, m, r, cc = O.kvarn_block_quant(x, bits, 64, 8)
        xh = O.kvarn_block_dequant(c, s, m, r, cc, 64)
        # error measured in the rotated domain, where the grid lives
        y = O.fwht_f32(x).astype(np.float64)
        yh = xh @ O.hadamard_matrix(256)
        rc = r.astype(np.float64)[:, None] * cc.astype(np.float64)[None, :]
        s_full = np.repeat(s.astype(np.float64), 64, axis=1)
        amp = np.abs(yh / rc)
        bound = rc * (s_full * 0.5 + 4e-3 * (amp + 4.0)) + 2e-3 * np.abs(yh)
        assert np.all(np.abs(y - yh) <= bound)
        # and the inverse rotation preserves the error norm
        assert np.isclose(np.linalg.norm(x - xh), np.linalg.norm(y - yh), rtol=1e-4)


def test_fwht_stage_order_is_fixed():
    """Stages run h = 1 first: for (1, 2^-24, -1, 2^-24) output 0 is
    ((1 + 2^-24) + (-1 + 2^-24)) / 2 = 2^-25; running h = 2 first would give
    ((1 - 1) + (2^-24 + 2^-24)) / 2 = 2^-24."""
    x = np.array([[1.0, 2.0 ** -24, -1.0, 2.0 ** -24]], np.float32)
    assert O.fwht_f32(x)[0, 0] == np.float32(2.0 ** -25)
