"""kvq_decode_step (projection of the new token, append, decode attention; one
cooperative kernel for bf16 affine/symmetric caches) against the three
separate calls, step after step and replayed from a captured graph, and both
against the oracle.

The fused kernel sums the projection (and its rank-r branch) in its own
order and precision, so its q/k/v may differ from the separate calls' in the
last bits; each path's q/k/v is checked against the oracle projection per
(sequence, head), each path's packed
planes are checked bit for bit against an oracle cache fed that path's own
keys and values, and each path's attention against the oracle: the bf16
output must be a rounding of a value within max-abs 2e-2 of the fp64 oracle
(the d_in 2048 cases give outputs of magnitude 4-8, where one bf16 step is
0.03)."""
import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu
from tests.helpers import FORMATS, check_attention, check_projection, compare_planes, oracle_cache

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


# fmt, B, d_in, Hq, Hkv, D, rank, prefill, fused expected
CASES = [
    ("affine4", 4, 512, 32, 4, 64, 16, 100, True),
    ("affine4", 4, 2048, 32, 4, 64, 16, 300, True),   # 1024-channel projection units
    ("sym2", 8, 2048, 32, 4, 64, 64, 130, True),      # the same at rank 64
    ("affine2", 2, 1536, 8, 2, 128, 16, 100, True),   # 512-channel units (1536 % 1024 != 0)
    ("sym2", 8, 256, 16, 2, 64, 64, 100, True),      # rank 64
    ("affine2", 3, 256, 8, 2, 128, 8, 100, True),    # D = 128
    ("sym4", 12, 256, 8, 2, 64, 8, 70, True),        # B > 8: second MMA row block
    ("sym4", 16, 256, 16, 8, 64, 8, 600, True),      # one split of 10 chunks: refills
    ("affine4", 16, 256, 16, 16, 64, 8, 40, True),   # more split items than CTAs
    ("kivi2", 2, 256, 8, 2, 128, 16, 100, False),    # three calls
    ("affine4_g128", 2, 256, 4, 2, 256, 16, 100, False),
]


@pytest.mark.parametrize("fmt_name,B,d_in,Hq,Hkv,D,r,prefill,fused_expected", CASES)
@pytest.mark.parametrize("graphed", [False, True])
def test_decode_step_matches_separate_calls(fmt_name, B, d_in, Hq, Hkv, D, r, prefill,
                                            fused_expected, graphed):
    from paper_2609_04263_gb300 import api
    spec = FORMATS[fmt_name]
    steps = 12
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
    nw = tw.float().cpu().numpy()
    nl = {p: tuple(t.float().cpu().numpy() for t in tl[p]) for p in "qkv"}
    kw = dict(spec)
    fmt = kw.pop("fmt")

    def mk():
        return api.Cache(api.make_desc(fmt, kw["key_bits"], kw["value_bits"], kw["group_size"], B,
                                       Hkv, Hq, D, Tmax, bf,
                                       residual_tokens=kw.get("residual_tokens", 0)))
    fused, ref = mk(), mk()
    assert fused.decode_step_fused(d_in, tl) == fused_expected
    oc_f = oracle_cache(spec, B, Hkv, D, Tmax, "bf16")
    oc_r = oracle_cache(spec, B, Hkv, D, Tmax, "bf16")
    for c in (fused, ref):
        q, k, v = api.project_lora(x[:, :prefill].contiguous(), tw, tl, 2.0, Hq, Hkv, D,
                                   rope_base=10000.0, pos_cache=c)
        c.append(k, v)
        c.attend_prefill(q)
    for oc in (oc_f, oc_r):
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
        # each path's q, k, v against the oracle projection, per head
        ref_p = O.project_lora(xs.float().cpu().numpy(), nw, nl, 2.0, Hq, Hkv, D,
                               pos0=prefill + s, rope_base=10000.0)
        for a_, b_, r_, name in zip(qkv, (q2, k2, v2), ref_p, "qkv"):
            check_projection(a_.float().cpu().numpy(), r_, "bf16", f"step {s} fused {name}")
            check_projection(b_.float().cpu().numpy(), r_, "bf16", f"step {s} separate {name}")
        oc_f.append(qkv[1].float().cpu().numpy(), qkv[2].float().cpu().numpy())
        oc_r.append(k2.float().cpu().numpy(), v2.float().cpu().numpy())
        ref_f = O.attend(oc_f, qkv[0].float().cpu().numpy())
        ref_r = O.attend(oc_r, q2.float().cpu().numpy())
        check_attention(out.float().cpu().numpy(), ref_f, "bf16", f"step {s}: fused attention")
        check_attention(o2.float().cpu().numpy(), ref_r, "bf16", f"step {s}: separate attention")
    assert fused.sync() == Tmax
    compare_planes(fused, oc_f)
    compare_planes(ref, oc_r)
    assert fused.sync() == Tmax


def test_decode_step_capacity_refused():
    """A step on a full cache is refused on the host and changes nothing."""
    from paper_2609_04263_gb300 import api, kvq
    B, d_in, Hq, Hkv, D, r = 2, 256, 8, 2, 64, 8
    wl = synth.Workload(name="t", dtype="bf16", layers=1, d_in=d_in, n_q_heads=Hq,
                        n_kv_heads=Hkv, head_dim=D, rope_base=10000.0, batch=B, prefill=0,
                        decode=0, fmt=1, key_bits=4, value_bits=4, group_size=32, rank=r)
    w, lora = synth.layer_weights(wl, 0)
    bf = torch.bfloat16
    tw = torch.from_numpy(w).to(bf).cuda()
    tl = {p: tuple(torch.from_numpy(t).to(bf).cuda() for t in lora[p]) for p in "qkv"}
    c = api.Cache(api.make_desc(O.FMT_AFFINE, 4, 4, 32, B, Hkv, Hq, D, 3, bf))
    xs = torch.from_numpy(synth.hidden_states((B, 1, d_in), seed=3)).to(bf).cuda()
    for _ in range(3):
        c.decode_step(xs, tw, tl, 2.0, 10000.0)
    assert c.sync() == 3
    before = {k: v.clone() for k, v in c.planes().items() if isinstance(v, torch.Tensor)}
    with pytest.raises(kvq.KvqError):
        c.decode_step(xs, tw, tl, 2.0, 10000.0)
    assert c.sync() == 3
    after = c.planes()
    for k, v in before.items():
        if k != "workspace":
            assert torch.equal(v.contiguous().view(torch.uint8),
                               after[k].contiguous().view(torch.uint8)), k
