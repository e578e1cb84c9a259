"""Parity at the workloads' full sizes, in the launch configuration bench.py
times (same shapes, same calls, decode steps replayed from a captured graph).

For every workload (single layer of each model shape, layer 0 weights):
  * projection: contiguous segments of rows at the start of the first
    sequence and the end of the last, against the oracle's fp64 projection;
  * prefill append: the packed planes of sampled (sequence, kv head) pairs bit
    for bit, against oracle caches fed the same projected k, v;
  * prefill attention: sampled queries of every query head of those kv heads;
  * decode: all decode steps of the workload; the planes at the end bit for
    bit and the attention output of the first and last step.
Outputs are bf16 (fp32 for the single-layer workload); the attention bound is
max-abs 2e-2 beyond the output's own rounding (bf16 holds |o| ~ 8 to 0.03).
"""
import math

import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def _act_tol(act):
    return (1e-4, 2.0 ** -23) if act == "f32" else (2e-2, 2.0 ** -8)


def _check_attention(got, ref, act, what):
    atol, rtol = _act_tol(act)
    err = np.abs(got - ref)
    bound = atol + rtol * np.abs(ref)
    worst = float((err - bound).max())
    assert worst <= 0, f"{what}: max-abs {err.max():.3e} exceeds the bound by {worst:.3e}"


def _planes_subset(cache, b, h):
    """GPU planes of one (sequence, kv head), shaped like a 1x1 oracle cache."""
    out = {}
    for name, t in cache.planes().items():
        if not isinstance(t, torch.Tensor) or name == "workspace":
            continue
        a = t[b:b + 1, h:h + 1]
        a = a.float().cpu().numpy() if a.dtype == torch.bfloat16 else a.cpu().numpy()
        out[name] = a
    return out


def _compare_subset(cache, b, h, oc):
    from tests.helpers import live
    gp = _planes_subset(cache, b, h)
    for name, ref in oc.planes.items():
        if ref.size == 0:
            continue
        got = gp[name]
        if name in ("k_row", "v_row"):
            got = got.reshape(1, 1, -1)
        a, r = live(name, got, oc), live(name, ref, oc)
        assert a.shape == r.shape, name
        if a.dtype == np.float16:
            same = np.array_equal(a.view(np.uint16), r.view(np.uint16))
        elif a.dtype == np.float32:
            same = np.array_equal(a, r.astype(np.float32))
        else:
            same = np.array_equal(a, r)
        assert same, f"plane {name} of (b={b}, h={h}) differs from the oracle"


@pytest.mark.parametrize("name", list(synth.WORKLOADS))
def test_full_size_layer(name):
    from paper_2609_04263_gb300 import api
    wl = synth.WORKLOADS[name]
    act = wl.dtype
    dt = torch.bfloat16 if act == "bf16" else torch.float32
    B, P, Dn, D = wl.batch, wl.prefill, wl.decode, wl.head_dim
    Hq, Hkv, g = wl.n_q_heads, wl.n_kv_heads, wl.n_q_heads // wl.n_kv_heads
    dev = "cuda"
    w, lora = synth.layer_weights(wl, 0)
    tw = torch.from_numpy(w).to(dt)
    tl = {p: tuple(torch.from_numpy(t).to(dt) for t in lora[p]) for p in "qkv"}
    nw = tw.float().numpy()
    nl = {p: tuple(t.float().numpy() for t in tl[p]) for p in "qkv"}
    dw, dl = tw.to(dev), {p: tuple(t.to(dev) for t in tl[p]) for p in "qkv"}
    x_pre = torch.from_numpy(synth.hidden_states((B, P, wl.d_in), wl.hidden, wl.outlier_frac)).to(dt)
    x_dec = torch.from_numpy(synth.hidden_states((B, Dn, wl.d_in), wl.hidden, wl.outlier_frac,
                                                 stream=1)).to(dt)
    desc = api.make_desc(wl.fmt, wl.key_bits, wl.value_bits, wl.group_size, B, Hkv, Hq, D,
                         wl.max_tokens, dt, residual_tokens=wl.residual_tokens,
                         sink_tokens=wl.sink_tokens, norm_iters=wl.norm_iters)
    cache = api.Cache(desc)
    args = (wl.alpha_over_r, Hq, Hkv, D)

    # ---- prefill projection (sampled row segments) ----
    q, k, v = api.project_lora(x_pre.to(dev), dw, dl, *args, rope_base=wl.rope_base,
                               pos_cache=cache)
    torch.cuda.synchronize()
    ptol = 1e-5 if act == "f32" else 1e-2
    for b, lo in ((0, 0), (B - 1, P - 64)):
        seg = x_pre[b:b + 1, lo:lo + 64].float().numpy()
        ref = O.project_lora(seg, nw, nl, *args, pos0=lo, rope_base=wl.rope_base)
        for got_t, ref_t in zip((q, k, v), ref):
            got = got_t[b:b + 1, :, lo:lo + 64].float().cpu().numpy()
            rel = np.abs(got - ref_t).max() / np.abs(ref_t).max()
            assert rel <= ptol, f"projection rows {lo}..{lo + 63} of sequence {b}: {rel:.2e}"

    # ---- prefill append and attention ----
    cache.append(k, v)
    o = cache.attend_prefill(q)
    torch.cuda.synchronize()
    samples = [(0, 0), (B - 1, Hkv - 1)]
    spec = dict(fmt=wl.fmt, key_bits=wl.key_bits, value_bits=wl.value_bits,
                group_size=wl.group_size, residual_tokens=wl.residual_tokens,
                sink_tokens=wl.sink_tokens, norm_iters=wl.norm_iters)
    ocs = {}
    for b, h in samples:
        oc = O.OracleCache(batch=1, kv_heads=1, head_dim=D, max_tokens=wl.max_tokens, act=act,
                           **spec)
        oc.append(k[b:b + 1, h:h + 1].float().cpu().numpy(),
                  v[b:b + 1, h:h + 1].float().cpu().numpy())
        _compare_subset(cache, b, h, oc)
        ocs[(b, h)] = oc
        kh, vh = oc.reconstruct()
        ls = sorted({0, 1, 63, P // 2, P - 17, P - 1} | set(range(P - 16, P)))
        heads = list(range(h * g, (h + 1) * g))
        qs = q[b:b + 1, heads][:, :, ls].float().cpu().numpy()
        ref = O.attention(qs, kh, vh, np.array(ls), 1.0 / math.sqrt(D))
        got = o[b:b + 1, heads][:, :, ls].float().cpu().numpy()
        _check_attention(got, ref, act, f"prefill attention (b={b}, kv head {h})")

    # ---- decode: the bench's captured step, replayed Dn times ----
    xs = torch.empty(B, 1, wl.d_in, dtype=dt, device=dev)
    outs = tuple(torch.empty(B, hh, 1, D, dtype=dt, device=dev) for hh in (Hq, Hkv, Hkv))
    od = torch.empty(B, Hq, 1, D, dtype=dt, device=dev)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        api.project_lora(xs, dw, dl, *args, rope_base=wl.rope_base, out=outs, pos_cache=cache)
        cache.append(outs[1], outs[2])
        cache.attend_decode(outs[0], out=od)
    x_dec_dev = x_dec.to(dev)
    for s in range(Dn):
        xs.copy_(x_dec_dev[:, s:s + 1])
        graph.replay()
        torch.cuda.synchronize()
        kk = outs[1].float().cpu().numpy()
        vv = outs[2].float().cpu().numpy()
        for (b, h), oc in ocs.items():
            oc.append(kk[b:b + 1, h:h + 1], vv[b:b + 1, h:h + 1])
        if s in (0, Dn - 1):
            if s == 0:     # decode projection rows against the oracle
                ref = O.project_lora(x_dec[:, 0:1].float().numpy(), nw, nl, *args, pos0=P,
                                     rope_base=wl.rope_base)
                for got_t, ref_t in zip(outs, ref):
                    rel = np.abs(got_t.float().cpu().numpy() - ref_t).max() / np.abs(ref_t).max()
                    assert rel <= ptol, f"decode projection: {rel:.2e}"
            for (b, h), oc in ocs.items():
                heads = list(range(h * g, (h + 1) * g))
                qd = outs[0][b:b + 1, heads].float().cpu().numpy()
                ref = O.attend(oc, qd)
                got = od[b:b + 1, heads].float().cpu().numpy()
                _check_attention(got, ref, act, f"decode step {s} (b={b}, kv head {h})")
    assert cache.sync() == wl.max_tokens
    for (b, h), oc in ocs.items():
        _compare_subset(cache, b, h, oc)
