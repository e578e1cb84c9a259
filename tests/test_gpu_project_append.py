"""kvq_project_append (the Q/K/V projection fused with the append of the new
keys and values, Section 3 Eq. (1) and Eq. (lora), then Section 3.1) against
the two separate calls and the oracle.

The fused kernel codes the keys and values the projection would have stored
(rotated, rounded to bf16) straight into the cache, so its planes must be
bit for bit those of an oracle cache fed the separate projection's k and v,
chunk after chunk, and its queries bit for bit the separate call's."""
import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu
from tests.helpers import (FORMATS, check_attention, check_projection, compare_planes, gpu_cache,
                           oracle_cache)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


# fmt, B, chunks, d_in, Hq, Hkv, D, ranks (q, k, v), rope base
CASES = [
    ("affine4", 2, [100, 60], 512, 8, 2, 64, (16, 16, 16), 10000.0),
    ("sym2", 1, [200], 256, 16, 4, 64, (64, 0, 8), 10000.0),
    ("affine8", 3, [40, 33], 256, 4, 2, 128, (8, 8, 8), 500000.0),
    ("affine2", 2, [130], 384, 8, 2, 128, (0, 16, 32), 0.0),
    ("sym4", 1, [17, 300], 256, 4, 4, 64, (16, 16, 16), 10000.0),
    # the TinyLlama-shaped prefill: 4 x 2048 rows, d_in 2048, 32 / 4 heads
    ("affine4", 4, [2048], 2048, 32, 4, 64, (16, 16, 16), 10000.0),
]


def _weights(B, T, d_in, Hq, Hkv, D, ranks, seed):
    wl = synth.Workload(name="t", dtype="bf16", layers=1, d_in=d_in, n_q_heads=Hq,
                        n_kv_heads=Hkv, head_dim=D, rope_base=10000.0, batch=B, prefill=T,
                        decode=0, fmt=1, key_bits=4, value_bits=4, group_size=32, rank=8,
                        outlier_frac=0.01)
    w, _ = synth.layer_weights(wl, 0, seed=seed)
    lora = {}
    for i, p in enumerate("qkv"):
        if ranks[i]:
            _, lr = synth.layer_weights(wl, 1 + i, seed=seed, rank=ranks[i])
            lora[p] = lr[p]
        else:
            lora[p] = None
    bf = torch.bfloat16
    tw = torch.from_numpy(w).to(bf).cuda()
    tl = {p: None if v is None else tuple(torch.from_numpy(t).to(bf).cuda() for t in v)
          for p, v in lora.items()}
    x = torch.from_numpy(synth.hidden_states((B, T, d_in), outlier_frac=0.01, seed=seed)).to(bf)
    return x.cuda(), tw, tl


@pytest.mark.parametrize("fmt_name,B,chunks,d_in,Hq,Hkv,D,ranks,base", CASES)
def test_project_append_matches_separate_calls(fmt_name, B, chunks, d_in, Hq, Hkv, D, ranks, base):
    from paper_2609_04263_gb300 import api
    spec = FORMATS[fmt_name]
    T = sum(chunks)
    x, tw, tl = _weights(B, T, d_in, Hq, Hkv, D, ranks, seed=len(chunks) * 7 + D)
    fused = gpu_cache(spec, B, Hkv, Hq, D, T + 4, "bf16")
    ref = gpu_cache(spec, B, Hkv, Hq, D, T + 4, "bf16")
    oc = oracle_cache(spec, B, Hkv, D, T + 4, "bf16")
    nl = {p: None if v is None else tuple(t.float().cpu().numpy() for t in v) for p, v in tl.items()}
    lo = 0
    for n in chunks:
        xs = x[:, lo:lo + n].contiguous()
        assert fused.project_append_supported(n, d_in, tl)
        q_f = fused.project_append(xs, tw, tl, 2.0, base)
        q_r, k_r, v_r = api.project_lora(xs, tw, tl, 2.0, Hq, Hkv, D, rope_base=base, pos_cache=ref)
        ref.append(k_r, v_r)
        torch.cuda.synchronize()
        assert torch.equal(q_f.view(torch.int16), q_r.view(torch.int16)), "queries differ"
        oc.append(k_r.float().cpu().numpy(), v_r.float().cpu().numpy())
        if lo == 0:   # the projection itself against the oracle, per head
            refp = O.project_lora(xs.float().cpu().numpy(), tw.float().cpu().numpy(), nl, 2.0,
                                  Hq, Hkv, D, pos0=0, rope_base=base)
            for got, r_, name in zip((q_r, k_r, v_r), refp, "qkv"):
                check_projection(got.float().cpu().numpy(), r_, "bf16", name)
        lo += n
    assert fused.sync() == T
    compare_planes(fused, oc)
    # prefill attention of the last chunk over the fused cache, against the oracle
    n = chunks[-1]
    o = fused.attend_prefill(q_f)
    ref_o = O.attend(oc, q_f.float().cpu().numpy())
    check_attention(o.float().cpu().numpy(), ref_o, "bf16", "attention over the fused append")


def test_project_append_replayed_capacity_refusal():
    """A captured fused call replayed on a full cache writes nothing and
    leaves the token count (the device refuses it like an append)."""
    B, n, d_in, Hq, Hkv, D = 1, 32, 256, 4, 2, 64
    x, tw, tl = _weights(B, n, d_in, Hq, Hkv, D, (8, 8, 8), seed=3)
    c = gpu_cache(FORMATS["affine4"], B, Hkv, Hq, D, 2 * n, "bf16")
    q = torch.empty(B, Hq, n, D, dtype=torch.bfloat16, device="cuda")
    c.project_append(x, tw, tl, 2.0, 10000.0, q=q)   # eager first call: the cache is set up
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        c.project_append(x, tw, tl, 2.0, 10000.0, q=q)
    assert c.sync() == n                         # capture does not execute
    g.replay()
    torch.cuda.synchronize()
    assert c.sync() == 2 * n
    before = {k: v.clone() for k, v in c.planes().items() if isinstance(v, torch.Tensor)}
    g.replay()                                   # a third append would overflow
    torch.cuda.synchronize()
    from paper_2609_04263_gb300 import kvq
    with pytest.raises(kvq.KvqError) as ei:
        c.sync()
    assert ei.value.status == kvq.KVQ_ERR_CAPACITY
    assert c.tokens == 2 * n
    after = c.planes()
    for k, v in before.items():
        if k != "workspace":
            assert torch.equal(v.contiguous().view(torch.uint8), after[k].contiguous().view(torch.uint8)), k
