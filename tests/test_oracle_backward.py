"""Pins of the oracle's straight-through backward (Section 3.3: appended
states enter attention as x_hat + x - stopgrad(x)).

The gradients come from PyTorch autograd through torch restatements of the
oracle's attention and projection; these pins tie those restatements to the
numpy functions the forward tests pin, check the gradients against central
finite differences of the numpy forward, and check the straight-through
identity itself."""
import math

import numpy as np

from oracle import kvq_oracle as O


def _rng(seed):
    return np.random.default_rng(seed)


def test_attention_backward_matches_finite_differences_of_the_forward():
    rng = _rng(0)
    B, Hq, Hkv, L, T, D = 1, 4, 2, 3, 6, 8
    q = rng.standard_normal((B, Hq, L, D))
    k = rng.standard_normal((B, Hkv, T, D))
    v = rng.standard_normal((B, Hkv, T, D))
    dout = rng.standard_normal((B, Hq, L, D))
    pos = np.arange(T - L, T)
    scale = 1 / math.sqrt(D)
    dq, dk, dv = O.attention_backward(q, k, v, pos, scale, dout)
    f = lambda q_, k_, v_: float((O.attention(q_, k_, v_, pos, scale) * dout).sum())
    eps = 1e-6
    for arr, grad, which in ((q, dq, 0), (k, dk, 1), (v, dv, 2)):
        for idx in [(0, 0, 0, 0), (0, 1, 2, 5), (0, arr.shape[1] - 1, arr.shape[2] - 1, 7)]:
            plus, minus = arr.copy(), arr.copy()
            plus[idx] += eps
            minus[idx] -= eps
            args_p = [q, k, v]
            args_m = [q, k, v]
            args_p[which], args_m[which] = plus, minus
            fd = (f(*args_p) - f(*args_m)) / (2 * eps)
            assert abs(fd - grad[idx]) < 1e-6 * max(1.0, abs(fd)), (which, idx, fd, grad[idx])


def test_masked_keys_get_no_gradient():
    """Keys after the last query's position are invisible: zero gradient."""
    rng = _rng(1)
    q = rng.standard_normal((1, 2, 2, 4))
    k = rng.standard_normal((1, 1, 7, 4))
    v = rng.standard_normal((1, 1, 7, 4))
    _, dk, dv = O.attention_backward(q, k, v, np.array([2, 3]), 0.5, rng.standard_normal(q.shape))
    assert np.all(dk[:, :, 4:] == 0) and np.all(dv[:, :, 4:] == 0)
    assert np.any(dk[:, :, :4] != 0) and np.any(dv[:, :, :4] != 0)


def test_lora_backward_matches_finite_differences_of_the_projection():
    rng = _rng(2)
    B, L, d_in, Hq, Hkv, D, r = 1, 3, 16, 2, 1, 8, 4
    x = rng.standard_normal((B, L, d_in))
    w = 0.1 * rng.standard_normal(((Hq + 2 * Hkv) * D, d_in))
    lora = {p: (0.1 * rng.standard_normal((r, d_in)),
                0.1 * rng.standard_normal(((Hq if p == "q" else Hkv) * D, r))) for p in "qkv"}
    dq = rng.standard_normal((B, Hq, L, D))
    dk = rng.standard_normal((B, Hkv, L, D))
    dv = rng.standard_normal((B, Hkv, L, D))
    grads = O.lora_backward(x, w, lora, 2.0, Hq, Hkv, D, dq, dk, dv, pos0=5, rope_base=100.0)

    def f(lr):
        q, k, v = O.project_lora(x, w, lr, 2.0, Hq, Hkv, D, pos0=5, rope_base=100.0)
        return float((q * dq).sum() + (k * dk).sum() + (v * dv).sum())
    eps = 1e-6
    for p in "qkv":
        for m in (0, 1):
            for idx in [(0, 0), (r - 1, 3) if m == 0 else (D - 1, r - 1)]:
                lp = {k_: tuple(t.copy() for t in v_) for k_, v_ in lora.items()}
                lm = {k_: tuple(t.copy() for t in v_) for k_, v_ in lora.items()}
                lp[p][m][idx] += eps
                lm[p][m][idx] -= eps
                fd = (f(lp) - f(lm)) / (2 * eps)
                got = grads[p][m][idx]
                assert abs(fd - got) < 1e-6 * max(1.0, abs(fd)), (p, m, idx, fd, got)


def test_straight_through_identity_on_a_coded_cache():
    """x_hat + x - stopgrad(x): the gradient reaching the appended keys and
    values is the gradient at their reconstruction, unchanged, although the
    forward uses the reconstruction (an affine 2-bit cache here)."""
    import torch
    rng = _rng(3)
    B, H, Hq, T, D = 1, 1, 2, 40, 32
    k = rng.standard_normal((B, H, T, D)).astype(np.float32)
    v = rng.standard_normal((B, H, T, D)).astype(np.float32)
    c = O.OracleCache(O.FMT_AFFINE, 2, 2, 32, B, H, D, T, act="f32")
    c.append(k, v)
    kh, vh = c.reconstruct()
    assert np.abs(kh - k).max() > 1e-2                       # the coding changed the values
    q = rng.standard_normal((B, Hq, T, D))
    dout = rng.standard_normal((B, Hq, T, D))
    pos = np.arange(T)
    _, dk_hat, dv_hat = O.attention_backward(q, kh, vh, pos, 0.2, dout)
    # the STE expression itself, through autograd
    tk = torch.tensor(k.astype(np.float64), requires_grad=True)
    tv = torch.tensor(v.astype(np.float64), requires_grad=True)
    kst = torch.as_tensor(kh) + tk - tk.detach()
    vst = torch.as_tensor(vh) + tv - tv.detach()
    o = O._attention_torch(torch.as_tensor(q), kst, vst, pos, 0.2)
    assert np.allclose(o.detach().numpy(), O.attention(q, kh, vh, pos, 0.2), rtol=1e-12, atol=1e-12)
    (o * torch.as_tensor(dout)).sum().backward()
    assert np.array_equal(tk.grad.numpy(), dk_hat) and np.array_equal(tv.grad.numpy(), dv_hat)
