"""Straight-through backward (Section 3.3: appended states enter attention as
x_hat + x - stopgrad(x)) against the oracle's fp64 autograd.

kvq_attend_backward: dq, and dk, dv at the stored reconstruction (which the
estimator passes unchanged to the coded keys and values), for the L newest
queries over every cached token.  kvq_lora_backward: the rank-r factors'
gradients from the projection's output gradients.  The oracle takes the
reconstruction from its own cache fed the same keys and values, so both
sides differentiate the same function.

Tolerance: fp32 accumulation over at most g L or B L terms against fp64, per
(sequence, head) slice (attention) or per matrix (adapters): max-abs
difference within 1e-3 of the slice's largest oracle value."""
import math

import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu
from tests.helpers import ACT, FORMATS, gpu_cache, kv_pair, oracle_cache

pytestmark = pytest.mark.gpu

TOL = 1e-3


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def _close(got, ref, what, axes=(2, 3)):
    got = np.asarray(got, dtype=np.float64)
    err = np.abs(got - ref).max(axis=axes)
    rel = err / np.maximum(np.abs(ref).max(axis=axes), 1e-30)
    assert rel.max() <= TOL, f"{what}: worst relative error {rel.max():.2e}"


def _filled(spec, act, B, Hkv, Hq, D, T0, L, seed):
    """Caches on both sides holding T0 earlier tokens, then the L new ones."""
    gc = gpu_cache(spec, B, Hkv, Hq, D, T0 + L + 8, act)
    oc = oracle_cache(spec, B, Hkv, D, T0 + L + 8, act)
    for n, st in ((T0, 0), (L, 1)):
        if n == 0:
            continue
        k, v, nk, nv = kv_pair(B, Hkv, n, D, act, seed=seed, stream=st)
        gc.append(k, v)
        oc.append(nk, nv)
    return gc, oc


# fmt, act, B, Hkv, Hq, D, earlier tokens T0, new tokens L
CASES = [
    ("affine4", "bf16", 2, 2, 8, 64, 0, 150),      # L = T, ragged
    ("sym2", "bf16", 1, 4, 16, 64, 37, 64),        # a prefix, GQA 4
    ("kivi2", "bf16", 2, 2, 4, 128, 100, 90),      # coded blocks and the residual window
    ("float", "f32", 1, 2, 2, 64, 10, 33),         # the unquantized control
    ("affine8", "bf16", 1, 1, 16, 128, 0, 70),     # GQA 16: 1120 stacked rows
    ("kivi_r0", "f32", 1, 1, 2, 64, 0, 100),
    ("affine4", "bf16", 1, 1, 1, 256, 5, 40),      # head_dim 256
]


@pytest.mark.parametrize("fmt,act,B,Hkv,Hq,D,T0,L", CASES)
def test_attend_backward_parity(fmt, act, B, Hkv, Hq, D, T0, L):
    spec = FORMATS[fmt]
    gc, oc = _filled(spec, act, B, Hkv, Hq, D, T0, L, seed=D + L)
    T = T0 + L
    rng = np.random.default_rng(L)
    q = torch.from_numpy(rng.standard_normal((B, Hq, L, D)).astype(np.float32)).to(ACT[act])
    do = torch.from_numpy(rng.standard_normal((B, Hq, L, D)).astype(np.float32)).to(ACT[act])
    scale = 1.0 / math.sqrt(D)
    dq, dk, dv = gc.attend_backward(q.cuda(), do.cuda(), scale=scale)
    torch.cuda.synchronize()
    kh, vh = oc.reconstruct()
    rq, rk, rv = O.attention_backward(q.float().numpy(), kh, vh, np.arange(T - L, T), scale,
                                      do.float().numpy())
    _close(dq.cpu().numpy(), rq, "dq")
    _close(dk.cpu().numpy(), rk, "dk")
    _close(dv.cpu().numpy(), rv, "dv")


def test_attend_backward_pair_by_pair_workspace():
    """A workspace for one (sequence, kv head) pair runs the pairs one pass
    at a time and gives the same gradients as one pass over all pairs."""
    from paper_2609_04263_gb300 import kvq
    B, Hkv, Hq, D, L = 2, 3, 6, 64, 96
    gc, _ = _filled(FORMATS["affine4"], "bf16", B, Hkv, Hq, D, 20, L, seed=5)
    rng = np.random.default_rng(9)
    q = torch.from_numpy(rng.standard_normal((B, Hq, L, D)).astype(np.float32)).bfloat16().cuda()
    do = torch.from_numpy(rng.standard_normal((B, Hq, L, D)).astype(np.float32)).bfloat16().cuda()
    per = kvq.kvq_attend_backward_workspace(gc.handle, L, Hq)
    one = gc.attend_backward(q, do, workspace=torch.empty(per, dtype=torch.uint8, device="cuda"))
    alls = gc.attend_backward(q, do)
    torch.cuda.synchronize()
    for a, b in zip(one, alls):
        assert torch.equal(a, b)


def _adapters(wl_kw, ranks, seed, act):
    wl = synth.Workload(name="t", dtype="bf16", layers=1, batch=1, prefill=8, decode=0, fmt=1,
                        key_bits=4, value_bits=4, group_size=32, rank=8, outlier_frac=0.01,
                        rope_base=10000.0, **wl_kw)
    w, _ = synth.layer_weights(wl, 0, seed=seed)
    lora = {}
    for i, p in enumerate("qkv"):
        if ranks[i]:
            _, lr = synth.layer_weights(wl, 1 + i, seed=seed, rank=ranks[i])
            lora[p] = lr[p]
        else:
            lora[p] = None
    dt = ACT[act]
    tw = torch.from_numpy(w).to(dt)
    tl = {p: None if v is None else tuple(torch.from_numpy(t).to(dt) for t in v)
          for p, v in lora.items()}
    return tw, tl


# act, B, L, d_in, Hq, Hkv, D, ranks, kv_rows - L, pos0, rope base
LORA_CASES = [
    ("bf16", 2, 70, 256, 8, 2, 64, (16, 16, 16), 0, 3, 10000.0),
    ("bf16", 1, 40, 512, 4, 4, 128, (8, 0, 24), 25, 100, 500000.0),   # d_k rows beyond L
    ("f32", 3, 17, 128, 2, 1, 64, (8, 8, 8), 0, 0, 0.0),              # no RoPE
    ("bf16", 2, 300, 1024, 8, 2, 128, (16, 16, 16), 0, 0, 500000.0),  # d_x on tensor cores: ragged row tile, 4 column tiles
    ("bf16", 1, 33, 192, 4, 2, 64, (8, 8, 8), 0, 0, 10000.0),        # d_in not a multiple of 128: the SIMT d_x
]


@pytest.mark.parametrize("act,B,L,d_in,Hq,Hkv,D,ranks,extra,pos0,base", LORA_CASES)
def test_lora_backward_parity(act, B, L, d_in, Hq, Hkv, D, ranks, extra, pos0, base):
    from paper_2609_04263_gb300 import api
    tw, tl = _adapters(dict(d_in=d_in, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=D), ranks, L, act)
    rng = np.random.default_rng(L + d_in)
    x = torch.from_numpy(synth.hidden_states((B, L, d_in), outlier_frac=0.01, seed=L)).to(ACT[act])
    dq = rng.standard_normal((B, Hq, L, D)).astype(np.float32)
    dk = rng.standard_normal((B, Hkv, L + extra, D)).astype(np.float32)
    dv = rng.standard_normal((B, Hkv, L + extra, D)).astype(np.float32)
    dev = {p: None if v is None else tuple(t.cuda() for t in v) for p, v in tl.items()}
    grads, dx = api.lora_backward(x.cuda(), tw.cuda(), dev, 2.0, Hq, Hkv, D,
                                  torch.from_numpy(dq).cuda(), torch.from_numpy(dk).cuda(),
                                  torch.from_numpy(dv).cuda(), pos0=pos0, rope_base=base,
                                  want_dx=True)
    torch.cuda.synchronize()
    nl = {p: None if v is None else tuple(t.float().numpy() for t in v) for p, v in tl.items()}
    ref = O.lora_backward(x.float().numpy(), tw.float().numpy(), nl, 2.0, Hq, Hkv, D, dq,
                          dk[:, :, extra:], dv[:, :, extra:], pos0=pos0, rope_base=base)
    for p in "qkv":
        if ref[p] is None:
            assert grads[p] is None
            continue
        for name, g, r in zip(("dA", "dB"), grads[p], ref[p]):
            _close(g.cpu().numpy()[None, None], r[None, None], f"{name}_{p}")
    # d_x against the oracle's input gradient (autograd through the projection)
    xt = torch.tensor(x.float().numpy().astype(np.float64), requires_grad=True)
    f64 = lambda a: torch.as_tensor(np.asarray(a, dtype=np.float64))
    lt = {p: None if v is None else tuple(f64(t) for t in v) for p, v in nl.items()}
    outs = O._project_torch(xt, f64(tw.float().numpy()), lt, 2.0, Hq, Hkv, D, pos0, base)
    sum((o * f64(g)).sum() for o, g in zip(outs, (dq, dk[:, :, extra:], dv[:, :, extra:]))).backward()
    _close(dx.cpu().numpy()[None], xt.grad.numpy()[None], "d_x", axes=(2, 3))


def test_ste_chain_through_a_coded_cache():
    """The training step the estimator serves: project (bf16), code the new
    keys and values into a 2-bit KIVI cache, attend, then backward through
    attention and into all three adapters.  The oracle differentiates the
    same reconstruction (its cache fed the projection's k, v) and the same
    projection in fp64."""
    from paper_2609_04263_gb300 import api
    B, L, d_in, Hq, Hkv, D = 2, 160, 512, 8, 2, 64
    ranks = (16, 16, 16)
    tw, tl = _adapters(dict(d_in=d_in, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=D), ranks, 1, "bf16")
    x = torch.from_numpy(synth.hidden_states((B, L, d_in), outlier_frac=0.01, seed=4)).bfloat16()
    dev = {p: tuple(t.cuda() for t in v) for p, v in tl.items()}
    spec = FORMATS["kivi2"]
    gc = gpu_cache(spec, B, Hkv, Hq, D, L, "bf16")
    oc = oracle_cache(spec, B, Hkv, D, L, "bf16")
    q, k, v = api.project_lora(x.cuda(), tw.cuda(), dev, 2.0, Hq, Hkv, D, rope_base=10000.0)
    gc.append(k, v)
    oc.append(k.float().cpu().numpy(), v.float().cpu().numpy())
    out = gc.attend_prefill(q)
    rng = np.random.default_rng(2)
    do = torch.from_numpy(rng.standard_normal(out.shape).astype(np.float32)).bfloat16()
    dq, dk, dv = gc.attend_backward(q, do.cuda())
    grads, _ = api.lora_backward(x.cuda(), tw.cuda(), dev, 2.0, Hq, Hkv, D, dq, dk, dv,
                                 rope_base=10000.0)
    torch.cuda.synchronize()
    kh, vh = oc.reconstruct()
    scale = 1.0 / math.sqrt(D)
    rq, rk, rv = O.attention_backward(q.float().cpu().numpy(), kh, vh, np.arange(L), scale,
                                      do.float().numpy())
    nl = {p: tuple(t.float().numpy() for t in v) for p, v in tl.items()}
    ref = O.lora_backward(x.float().numpy(), tw.float().numpy(), nl, 2.0, Hq, Hkv, D, rq, rk, rv,
                          rope_base=10000.0)
    for p in "qkv":
        for name, g, r in zip(("dA", "dB"), grads[p], ref[p]):
            _close(g.cpu().numpy()[None, None], r[None, None], f"{name}_{p}")
