"""kvq_decode_step (projection of the new token, append, decode attention; one
cooperative kernel for bf16 affine/symmetric caches) gives the same results as
the three separate calls, step after step and when replayed from a captured
graph, and both match the oracle."""
import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu
from tests.helpers import FORMATS, compare_planes, oracle_cache

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


CASES = [
    ("affine4", 4, 512, 32, 4, 64, 16),     # fused path
    ("sym2", 8, 256, 16, 2, 64, 64),        # fused path, rank 64
    ("affine2", 3, 256, 8, 2, 128, 8),      # fused path, D = 128
    ("kivi2", 2, 256, 8, 2, 128, 16),       # general path (three calls)
    ("affine4_g128", 2, 256, 4, 2, 256, 16),  # general path
]


@pytest.mark.parametrize("fmt_name,B,d_in,Hq,Hkv,D,r", CASES)
@pytest.mark.parametrize("graphed", [False, True])
def test_decode_step_matches_separate_calls(fmt_name, B, d_in, Hq, Hkv, D, r, graphed):
    from paper_2609_04263_gb300 import api
    spec = FORMATS[fmt_name]
    prefill, steps = 100, 12
    Tmax = prefill + steps
    wl = synth.Workload(name="t", dtype="bf16", layers=1, d_in=d_in, n_q_heads=Hq,
                        n_kv_heads=Hkv, head_dim=D, rope_base=10000.0, batch=B, prefill=0,
                        decode=0, fmt=1, key_bits=4, value_bits=4, group_size=32, rank=r,
                        outlier_frac=0.01)
    w, lora = synth.layer_weights(wl, 0)
    bf = torch.bfloat16
    tw = torch.from_numpy(w).to(bf).cuda()
    tl = {p: tuple(torch.from_numpy(t).to(bf).cuda() for t in lora[p]) for p in "qkv"}
    x = torch.from_numpy(synth.hidden_states((B, prefill + steps, d_in), outlier_frac=0.01,
                                             seed=7)).to(bf).cuda()
    kw = dict(spec)
    fmt = kw.pop("fmt")

    def mk():
        return api.Cache(api.make_desc(fmt, kw["key_bits"], kw["value_bits"], kw["group_size"], B,
                                       Hkv, Hq, D, Tmax, bf,
                                       residual_tokens=kw.get("residual_tokens", 0)))
    fused, ref = mk(), mk()
    oc = oracle_cache(spec, B, Hkv, D, Tmax, "bf16")
    for c in (fused, ref):
        q, k, v = api.project_lora(x[:, :prefill].contiguous(), tw, tl, 2.0, Hq, Hkv, D,
                                   rope_base=10000.0, pos_cache=c)
        c.append(k, v)
        c.attend_prefill(q)
    oc.append(k.float().cpu().numpy(), v.float().cpu().numpy())
    xs = torch.empty(B, 1, d_in, dtype=bf, device="cuda")
    qkv = tuple(torch.empty(B, h, 1, D, dtype=bf, device="cuda") for h in (Hq, Hkv, Hkv))
    out = torch.empty(B, Hq, 1, D, dtype=bf, device="cuda")
    graph = None
    if graphed:
        torch.cuda.synchronize()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=side):
            fused.decode_step(xs, tw, tl, 2.0, 10000.0, qkv=qkv, out=out)
        fused.sync()
    for s in range(steps):
        xs.copy_(x[:, prefill + s:prefill + s + 1])
        if graphed:
            graph.replay()
        else:
            fused.decode_step(xs, tw, tl, 2.0, 10000.0, qkv=qkv, out=out)
        q2, k2, v2 = api.project_lora(xs, tw, tl, 2.0, Hq, Hkv, D, rope_base=10000.0,
                                      pos_cache=ref)
        ref.append(k2, v2)
        o2 = ref.attend_decode(q2)
        torch.cuda.synchronize()
        for a_, b_ in zip(qkv, (q2, k2, v2)):
            assert torch.equal(a_, b_)
        assert (out.float() - o2.float()).abs().max().item() <= 2e-3
        oc.append(k2.float().cpu().numpy(), v2.float().cpu().numpy())
        refo = O.attend(oc, q2.float().cpu().numpy())
        assert np.abs(out.float().cpu().numpy() - refo).max() <= 2e-2
    assert fused.sync() == Tmax
    compare_planes(fused, oc)
    compare_planes(ref, oc)
