"""A decode step (projection with positions from the cache, append, decode
attention) captured once in a CUDA graph and replayed: the device-resident
token count advances on every replay, the planes match the oracle fed the
same projected k/v, and an overflowing replay is refused on the device."""
import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu
from tests.helpers import check_projection, compare_planes

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def _layer(B, d_in, Hq, Hkv, D, r):
    wl = synth.Workload(name="g", dtype="bf16", layers=1, d_in=d_in, n_q_heads=Hq,
                        n_kv_heads=Hkv, head_dim=D, rope_base=10000.0, batch=B, prefill=0,
                        decode=0, fmt=1, key_bits=4, value_bits=4, group_size=32, rank=r,
                        outlier_frac=0.01)
    w, lora = synth.layer_weights(wl, 0)
    bf = torch.bfloat16
    tw = torch.from_numpy(w).to(bf)
    tl = {p: tuple(torch.from_numpy(t).to(bf) for t in lora[p]) for p in "qkv"}
    return tw, tl


@pytest.mark.parametrize("fmt_name", ["affine4", "kivi2"])
def test_captured_decode_step_replays(fmt_name):
    from paper_2609_04263_gb300 import api
    from tests.helpers import FORMATS, oracle_cache
    spec = dict(FORMATS[fmt_name])
    B, d_in, Hq, Hkv, D, r = 2, 256, 8, 2, 64, 16
    prefill, steps = 70, 40
    Tmax = prefill + steps
    tw, tl = _layer(B, d_in, Hq, Hkv, D, r)
    w, lora = tw.cuda(), {p: tuple(t.cuda() for t in v) for p, v in tl.items()}
    nl = {p: tuple(t.float().numpy() for t in v) for p, v in tl.items()}
    x_all = torch.from_numpy(synth.hidden_states((B, prefill + steps, d_in), outlier_frac=0.01,
                                                 seed=4)).to(torch.bfloat16)
    fmt = spec.pop("fmt")
    desc = api.make_desc(fmt, spec["key_bits"], spec["value_bits"], spec["group_size"], B, Hkv,
                         Hq, D, Tmax, torch.bfloat16,
                         residual_tokens=spec.get("residual_tokens", 0))
    cache = api.Cache(desc)
    oc = oracle_cache(FORMATS[fmt_name], B, Hkv, D, Tmax, "bf16")
    # prefill, eager
    xp = x_all[:, :prefill].contiguous().cuda()
    q, k, v = api.project_lora(xp, w, lora, 2.0, Hq, Hkv, D, rope_base=10000.0,
                               pos_cache=cache)
    cache.append(k, v)
    cache.attend_prefill(q)
    oc.append(k.float().cpu().numpy(), v.float().cpu().numpy())
    # capture one decode step
    xs = torch.empty(B, 1, d_in, dtype=torch.bfloat16, device="cuda")
    outs = tuple(torch.empty(B, h, 1, D, dtype=torch.bfloat16, device="cuda")
                 for h in (Hq, Hkv, Hkv))
    o = torch.empty(B, Hq, 1, D, dtype=torch.bfloat16, device="cuda")
    side = torch.cuda.Stream()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        api.project_lora(xs, w, lora, 2.0, Hq, Hkv, D, rope_base=10000.0, out=outs,
                         pos_cache=cache)
        cache.append(outs[1], outs[2])
        cache.attend_decode(outs[0], out=o)
    # capture does not execute: the host mirror advanced once, the device did not
    assert cache.sync() == prefill
    for s in range(steps):
        xs.copy_(x_all[:, prefill + s:prefill + s + 1])
        g.replay()
        torch.cuda.synchronize()
        # oracle: same projected k/v, positions continue the cache
        ref = O.project_lora(x_all[:, prefill + s:prefill + s + 1].float().numpy(),
                             tw.float().numpy(), nl, 2.0, Hq, Hkv, D, pos0=prefill + s,
                             rope_base=10000.0)
        for got_t, ref_t, name in zip(outs, ref, "qkv"):
            check_projection(got_t.float().cpu().numpy(), ref_t, "bf16", f"step {s} {name}")
        oc.append(outs[1].float().cpu().numpy(), outs[2].float().cpu().numpy())
        ref_o = O.attend(oc, outs[0].float().cpu().numpy())
        assert np.abs(o.float().cpu().numpy() - ref_o).max() <= 2e-2
    assert cache.sync() == Tmax
    compare_planes(cache, oc)
    # one more replay would overflow: refused on the device, nothing written
    before = {n: t.clone() for n, t in cache.planes().items() if isinstance(t, torch.Tensor)}
    g.replay()
    from paper_2609_04263_gb300 import kvq
    with pytest.raises(kvq.KvqError) as ei:
        cache.sync()
    assert ei.value.status == kvq.KVQ_ERR_CAPACITY
    assert cache.tokens == Tmax
    after = cache.planes()
    for n, t in before.items():
        if n != "workspace":
            # bit patterns: rows past the stored tokens hold whatever the
            # allocator left there, NaN included
            assert torch.equal(t.contiguous().view(torch.uint8),
                               after[n].contiguous().view(torch.uint8)), n
