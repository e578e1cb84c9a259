"""The fast code quotient of the pack kernels, checked in IEEE fp32 on the host.

A code is rint of the fp32-rounded quotient a / s (round half to even both
times).  The kernels form q = RN(a * RN(1 / s)) and keep rint(q) only when q
lies farther than 2^-14 from the half-integer between its neighbouring
integers and |q| < 64; otherwise they form the IEEE quotient.  This test
replays that decision with numpy's fp32 arithmetic (correctly rounded, like
the kernels' __frcp_rn and __fmul_rn) on random and adversarial inputs and
checks that whenever the fast path is taken it agrees with rint(RN(a / s)).
"""
import numpy as np

GUARD = np.float32(2.0 ** -14)


def fast_ok_and_code(a, s):
    inv = np.float32(1.0) / s                     # RN(1 / s)
    q = a * inv                                   # RN(a * inv)
    d = np.abs(q - (np.floor(q) + np.float32(0.5)))
    ok = (d > GUARD) & (np.abs(q) < np.float32(64.0))
    return ok, np.rint(q)


def exact_code(a, s):
    return np.rint(a / s)                         # RN(a / s), then half to even


def _check(a, s):
    a = a.astype(np.float32)
    s = s.astype(np.float32)
    ok, fast = fast_ok_and_code(a, s)
    exact = exact_code(a, s)
    bad = ok & (fast != exact)
    assert not bad.any(), (a[bad][:5], s[bad][:5])
    return ok.mean()


def test_random_groups():
    rng = np.random.default_rng(0)
    n = 2_000_000
    # affine: s = max((mx - mn) / (2^b - 1), 1e-8), a = x - mn in [0, mx - mn]
    for levels in (3, 15, 255):
        span = np.exp(rng.uniform(-20, 12, n)).astype(np.float32)
        s = np.maximum(span / np.float32(levels), np.float32(1e-8))
        a = (rng.uniform(0, 1, n) * span).astype(np.float32)
        frac = _check(a, s)
        if levels < 64:
            assert frac > 0.99                    # 2- and 4-bit codes: the fast path
        # (8-bit codes above 64 take the IEEE quotient: correct, only slower)
    # symmetric: a = x in [-amax, amax], s = amax / qmax
    for qmax in (1, 7, 127):
        amax = np.exp(rng.uniform(-20, 12, n)).astype(np.float32)
        s = np.maximum(amax / np.float32(qmax), np.float32(1e-8))
        a = (rng.uniform(-1, 1, n) * amax).astype(np.float32)
        _check(a, s)


def test_bf16_grids_and_exact_ties():
    # bf16 inputs put many quotients on or next to a half-integer
    rng = np.random.default_rng(1)
    n = 1_000_000
    bf = lambda x: (x.astype(np.float32).view(np.uint32) & np.uint32(0xFFFF0000)).view(np.float32)
    x = bf(rng.standard_normal((n, 2)).astype(np.float32))
    mn, mx = np.minimum(x[:, 0], x[:, 1]), np.maximum(x[:, 0], x[:, 1])
    for levels in (3, 15):
        s = np.maximum((mx - mn) / np.float32(levels), np.float32(1e-8))
        t = bf(rng.uniform(0, 1, n).astype(np.float32) * (mx - mn) + mn)
        _check(t - mn, s)
    # exact ties and their neighbours: a = (k + 1/2) s, then one to four ulps off
    k = rng.integers(0, 15, n).astype(np.float32)
    s = np.exp(rng.uniform(-10, 5, n)).astype(np.float32)
    a = (k + np.float32(0.5)) * s
    for ulps in range(-4, 5):
        _check(np.nextafter(a, np.float32(np.inf) if ulps > 0 else np.float32(-np.inf))
               if ulps else a, s)
        a_shift = a.copy()
        for _ in range(abs(ulps)):
            a_shift = np.nextafter(a_shift, np.float32(np.inf) if ulps > 0 else np.float32(0))
        _check(a_shift, s)


def test_special_values_take_the_exact_path():
    s = np.array([1.0, 1e-8, 3.0, 1.0], np.float32)
    a = np.array([np.nan, 1.0, np.inf, 1e9], np.float32)
    with np.errstate(invalid="ignore"):           # inf - inf on the way, as on the GPU
        ok, _ = fast_ok_and_code(a, s)
    assert not ok.any()                           # NaN, out of range: IEEE quotient
