"""Pins of the oracle's quantizers and bit packing (Section 3.1, Eq. affine).

Each pin is independent of the oracle's own code: hand-worked groups, exact
code-grid recovery, closed-form error bounds, and brute force over all codes.
"""
import os

import numpy as np
import pytest

from oracle import kvq_oracle as O

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _read_examples():
    rows = []
    with open(os.path.join(GOLD, "quant_examples.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            kind, bits, x, codes, by, s16, m16 = line.split()
            rows.append((kind, int(bits), [float(v) for v in x.split(",")],
                         [int(v) for v in codes.split(",")],
                         [int(v, 16) for v in by.split(",")], int(s16, 16),
                         None if m16 == "-" else int(m16, 16)))
    return rows


@pytest.mark.parametrize("row", _read_examples())
def test_hand_worked_groups(row):
    kind, bits, x, codes, by, s16, m16 = row
    x = np.array([x], dtype=np.float32)
    if kind == "affine":
        c, s, m = O.affine_quant(x, bits)
        assert int(m.view(np.uint16)[0]) == m16
    else:
        c, s = O.symmetric_quant(x, bits)
    assert c[0].tolist() == codes
    assert int(s.view(np.uint16)[0]) == s16
    packed = O.pack_codes(c, bits)
    assert packed[0].tolist() == by


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_pack_roundtrip(bits):
    rng = np.random.default_rng(0)
    c = rng.integers(0, 2 ** bits, size=(3, 5, 64), dtype=np.uint8)
    p = O.pack_codes(c, bits)
    assert p.shape == (3, 5, 64 * bits // 8)
    assert np.array_equal(O.unpack_codes(p, bits), c)


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_affine_exact_grid_recovery(bits):
    """mn and s fp16-exact powers of two, x = mn + k s, max k = 2^b - 1:
    the codes are k and the reconstruction is x exactly."""
    rng = np.random.default_rng(1)
    qmax = 2 ** bits - 1
    for trial in range(50):
        e = int(rng.integers(-6, 3))
        s = 2.0 ** e
        mn = float(rng.integers(-40, 40)) * 2.0 ** -2
        k = rng.integers(0, qmax + 1, size=32)
        k[0], k[1] = 0, qmax
        rng.shuffle(k)
        x = (mn + k * s).astype(np.float32)[None]
        c, s16, m16 = O.affine_quant(x, bits)
        assert np.array_equal(c[0], k)
        assert float(s16[0]) == s and float(m16[0]) == mn
        assert np.array_equal(O.affine_dequant(c, s16, m16)[0], x[0].astype(np.float64))


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_symmetric_exact_grid_recovery(bits):
    rng = np.random.default_rng(2)
    qmax = 2 ** (bits - 1) - 1
    for trial in range(50):
        s = 2.0 ** int(rng.integers(-6, 3))
        q = rng.integers(-qmax, qmax + 1, size=32)
        q[0] = qmax if trial % 2 else -qmax
        x = (q * s).astype(np.float32)[None]
        u, s16 = O.symmetric_quant(x, bits)
        assert np.array_equal(u[0].astype(int) - 2 ** (bits - 1), q)
        assert float(s16[0]) == s
        assert np.array_equal(O.symmetric_dequant(u, s16, bits)[0], x[0].astype(np.float64))


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_affine_roundtrip_bound_and_brute_force(bits):
    """|x - x_hat| <= s/2 + |mn - m16| + c |s - s16| (with the fp32 s, mn),
    and every code is the nearest grid point of the fp32 grid."""
    rng = np.random.default_rng(3)
    x = (rng.standard_normal((400, 32)) * rng.uniform(0.01, 30, (400, 1))
         + rng.normal(0, 3, (400, 1))).astype(np.float32)
    c, s16, m16 = O.affine_quant(x, bits)
    x64 = x.astype(np.float64)
    mn = x.min(1).astype(np.float64)
    mx = x.max(1).astype(np.float64)
    s = np.maximum((mx - mn) / (2 ** bits - 1), 1e-8)
    xh = O.affine_dequant(c, s16, m16)
    bound = (s / 2)[:, None] + np.abs(mn - m16.astype(np.float64))[:, None] \
        + c * np.abs(s - s16.astype(np.float64))[:, None]
    assert np.all(np.abs(x64 - xh) <= bound * (1 + 1e-5) + 1e-30)
    # brute force: the chosen code minimises |(x - mn)/s - k| over all k
    grid = np.arange(2 ** bits)[None, None, :]
    dist = np.abs((x64 - mn[:, None])[..., None] / s[:, None, None] - grid)
    best = dist.min(-1)
    chosen = np.take_along_axis(dist, c[..., None].astype(np.int64), -1)[..., 0]
    assert np.all(chosen <= best + 1e-5)
    # 8-bit error bound: range / 510 plus fp16 metadata rounding
    if bits == 8:
        rel = np.abs(x64 - xh).max(1) / np.maximum(mx - mn, 1e-30)
        assert np.all(rel <= 1 / 510 + 2e-3)


def test_round_half_to_even():
    # (x - mn)/s lands exactly on k + 0.5 for k = 0..6: codes must be even
    s = 1.0
    x = np.array([[0.0, 0.5, 1.5, 2.5, 3.5, 4.5, 5.5, 6.5, 15.0]], np.float32)
    c, _, _ = O.affine_quant(x, 4)
    assert c[0].tolist() == [0, 0, 2, 2, 4, 4, 6, 6, 15]


def test_degenerate_and_negative_zero():
    x = np.full((1, 32), -0.0, np.float32)
    c, s16, m16 = O.affine_quant(x, 4)
    assert not c.any()
    assert int(s16.view(np.uint16)[0]) == 0          # fp16(1e-8) underflows
    assert int(m16.view(np.uint16)[0]) == 0          # -0 stored as +0
    u, s16 = O.symmetric_quant(np.zeros((1, 32), np.float32), 2)
    assert np.all(u == 2)
    assert np.all(O.symmetric_dequant(u, s16, 2) == 0)


@pytest.mark.parametrize("bits", [2, 4])
def test_symmetric_bound(bits):
    rng = np.random.default_rng(4)
    x = rng.standard_normal((300, 32)).astype(np.float32) * 3
    u, s16 = O.symmetric_quant(x, bits)
    qmax = 2 ** (bits - 1) - 1
    s = np.maximum(np.abs(x.astype(np.float64)).max(1) / qmax, 1e-8)
    q = u.astype(np.float64) - 2 ** (bits - 1)
    err = np.abs(x - O.symmetric_dequant(u, s16, bits))
    bound = (s / 2)[:, None] + np.abs(q) * np.abs(s - s16.astype(np.float64))[:, None]
    assert np.all(err <= bound * (1 + 1e-5))
    # codes 0 never used: the symmetric range is [-qmax, qmax]
    assert u.min() >= 1
