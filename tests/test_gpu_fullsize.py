"""Parity at the workloads' full sizes, in the launch configuration bench.py
times (same shapes, same calls, decode steps replayed from a captured graph).

For every workload (single layer of each model shape, layer 0 weights):
  * projection: contiguous segments of rows at the start of the first
    sequence and the end of the last, against the oracle's fp64 projection;
  * prefill append: the packed planes of sampled (sequence, kv head) pairs bit
    for bit, against oracle caches fed the same projected k, v; where the
    fused projection-and-append covers the cache (the bench's prefill path),
    its whole cache and queries bit for bit against the separate calls';
  * prefill attention: sampled queries of every query head of those kv heads;
  * decode: all decode steps of the workload through kvq_decode_step (the
    fused single-kernel step where the library takes it, as the bench does),
    replayed from one captured graph; the step's q, k, v and attention output
    at the first and last step against the oracle, and at the end the planes
    bit for bit against oracle caches fed the steps' own keys and values.
Projections are checked per (sequence, head) against the oracle rounded to
the activation dtype (relative 1e-2 for bf16, 1e-5 for fp32).  Attention
outputs must be a rounding of a value within max-abs 2e-2 (bf16) or 1e-4
(fp32) of the fp64 oracle.
"""
import math

import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu
from tests.helpers import check_attention, check_projection

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


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


# which decode path bench.py's kvq_decode_step takes on each workload
FUSED = {"single_layer_f32": False, "tinyllama_affine4": True, "tinyllama_sym2": True,
         "llama8b_kivi": False, "gemma12b_kvarn": False}


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
    assert cache.decode_step_fused(wl.d_in, dl) == FUSED[name]

    # ---- prefill projection (sampled row segments, every head) ----
    q, k, v = api.project_lora(x_pre.to(dev), dw, dl, *args, rope_base=wl.rope_base,
                               pos_cache=cache)
    torch.cuda.synchronize()
    for b, lo in ((0, 0), (B - 1, P - 64)):
        seg = x_pre[b:b + 1, lo:lo + 64].float().numpy()
        ref = O.project_lora(seg, nw, nl, *args, pos0=lo, rope_base=wl.rope_base)
        for got_t, ref_t, pn in zip((q, k, v), ref, "qkv"):
            got = got_t[b:b + 1, :, lo:lo + 64].float().cpu().numpy()
            check_projection(got, ref_t, act, f"prefill {pn} rows {lo}..{lo + 63} of sequence {b}")

    # ---- prefill append and attention ----
    cache.append(k, v)
    if cache.project_append_supported(P, wl.d_in, dl):
        # bench.py's prefill takes the fused projection-and-append here: its
        # cache and queries must be the separate calls', bit for bit
        fused = api.Cache(desc)
        q_f = fused.project_append(x_pre.to(dev), dw, dl, wl.alpha_over_r, wl.rope_base)
        torch.cuda.synchronize()
        assert torch.equal(q_f.view(torch.int16), q.view(torch.int16))
        assert fused.sync() == P
        gp, fp = cache.planes(), fused.planes()
        for name, t in gp.items():          # rows of the P stored tokens
            if isinstance(t, torch.Tensor) and name != "workspace":
                assert torch.equal(t[:, :, :P].contiguous().view(torch.uint8),
                                   fp[name][:, :, :P].contiguous().view(torch.uint8)), name
        del fused, q_f
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
        check_attention(got, ref, act, f"prefill attention (b={b}, kv head {h})")

    # ---- decode: bench.py's captured kvq_decode_step, replayed Dn times ----
    xs = torch.empty(B, 1, wl.d_in, dtype=dt, device=dev)
    outs = tuple(torch.empty(B, hh, 1, D, dtype=dt, device=dev) for hh in (Hq, Hkv, Hkv))
    od = torch.empty(B, Hq, 1, D, dtype=dt, device=dev)
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        cache.decode_step(xs, dw, dl, wl.alpha_over_r, wl.rope_base, qkv=outs, out=od)
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
            # the step's own q, k, v against the oracle projection, per head
            ref = O.project_lora(x_dec[:, s:s + 1].float().numpy(), nw, nl, *args, pos0=P + s,
                                 rope_base=wl.rope_base)
            for got_t, ref_t, pn in zip(outs, ref, "qkv"):
                check_projection(got_t.float().cpu().numpy(), ref_t, act,
                                  f"decode step {s} projection {pn}")
            for (b, h), oc in ocs.items():
                heads = list(range(h * g, (h + 1) * g))
                qd = outs[0][b:b + 1, heads].float().cpu().numpy()
                ref = O.attend(oc, qd)
                got = od[b:b + 1, heads].float().cpu().numpy()
                check_attention(got, ref, act, f"decode step {s} (b={b}, kv head {h})")
    assert cache.sync() == wl.max_tokens
    # the planes the decode steps wrote, against oracle caches fed the steps' own k, v
    for (b, h), oc in ocs.items():
        _compare_subset(cache, b, h, oc)
