"""Projection over a frozen NF4 base (kvq_project_lora_nf4; Sections 3.4 and 4,
the NF4 Gemma and Llama-3.1 bases with explicit adapters) against the oracle,
which dequantizes the same codes with its own NF4 levels and projects in fp64.

Tolerance per (sequence, head), as for every bf16 projection: max-abs
difference from the oracle rounded to bf16 over the head's largest oracle
value, 1e-2.  The kernel rounds each dequantized weight to bf16 (relative
error 2^-9 per weight) before the tensor-core product."""
import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu
from tests.helpers import check_projection

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def _case(B, L, d_in, Hq, Hkv, D, ranks, seed=0):
    wl = synth.Workload(name="t", dtype="bf16", layers=1, d_in=d_in, n_q_heads=Hq,
                        n_kv_heads=Hkv, head_dim=D, rope_base=10000.0, batch=B, prefill=L,
                        decode=0, fmt=1, key_bits=4, value_bits=4, group_size=32, rank=8,
                        outlier_frac=0.01)
    codes, absmax = synth.nf4_base(wl, 0, seed=seed)
    lora = {}
    for i, p in enumerate("qkv"):
        if ranks[i]:
            _, lr = synth.layer_weights(wl, 1 + i, seed=seed, rank=ranks[i])
            lora[p] = lr[p]
        else:
            lora[p] = None
    bf = torch.bfloat16
    x = torch.from_numpy(synth.hidden_states((B, L, d_in), outlier_frac=0.01, seed=seed)).to(bf)
    tl = {p: None if v is None else tuple(torch.from_numpy(t).to(bf) for t in v) for p, v in lora.items()}
    nl = {p: None if v is None else tuple(t.float().numpy() for t in v) for p, v in tl.items()}
    dev = (x.cuda(), torch.from_numpy(codes).cuda(), torch.from_numpy(absmax).cuda(),
           {p: None if v is None else tuple(t.cuda() for t in v) for p, v in tl.items()})
    return dev, (x.float().numpy(), codes, absmax, nl)


# B, L, d_in, Hq, Hkv, D, ranks (q, k, v), pos0, rope base
CASES = [
    (2, 37, 512, 8, 2, 64, (16, 16, 16), 5, 10000.0),          # ragged row tile
    (1, 1, 4096, 32, 8, 128, (16, 16, 16), 8200, 500000.0),    # one decode row
    (16, 1, 4096, 32, 8, 128, (16, 16, 16), 8200, 500000.0),   # the 8B-shaped decode step
    (4, 300, 4096, 32, 8, 128, (16, 16, 16), 0, 500000.0),     # 8B-shaped prefill rows
    (3, 50, 2048, 32, 4, 64, (24, 0, 40), 0, 10000.0),         # part-filled rank tiles, no K adapter
    (2, 64, 256, 4, 4, 64, (0, 0, 0), 0, 0.0),                 # no adapters, no RoPE
]


@pytest.mark.parametrize("B,L,d_in,Hq,Hkv,D,ranks,pos0,base", CASES)
def test_project_nf4_parity(B, L, d_in, Hq, Hkv, D, ranks, pos0, base):
    from paper_2609_04263_gb300 import api
    (tx, tc, ta, tl), (nx, codes, absmax, nl) = _case(B, L, d_in, Hq, Hkv, D, ranks)
    got = api.project_lora_nf4(tx, tc, ta, tl, 2.0, Hq, Hkv, D, pos0=pos0, rope_base=base)
    ref = O.project_lora_nf4(nx, codes, absmax, nl, 2.0, Hq, Hkv, D, pos0=pos0, rope_base=base)
    for name, g, r in zip("qkv", got, ref):
        check_projection(g.float().cpu().numpy(), r, "bf16", name)


def test_project_nf4_full_llama8b_prefill_sampled_rows():
    """The whole 8B-shaped prefill (16 x 8192 rows, the bench's workload with an
    NF4 base); rows at the start of the first sequence and the end of the last
    against the oracle."""
    from paper_2609_04263_gb300 import api
    wl = synth.WORKLOADS["llama8b_kivi"]
    B, L, D = wl.batch, wl.prefill, wl.head_dim
    codes, absmax = synth.nf4_base(wl, 0)
    _, lora = synth.layer_weights(wl, 0)
    bf = torch.bfloat16
    x = torch.from_numpy(synth.hidden_states((B, L, wl.d_in), wl.hidden, wl.outlier_frac)).to(bf)
    tl = {p: tuple(torch.from_numpy(t).to(bf) for t in lora[p]) for p in "qkv"}
    nl = {p: tuple(t.float().numpy() for t in tl[p]) for p in "qkv"}
    q, k, v = api.project_lora_nf4(x.cuda(), torch.from_numpy(codes).cuda(),
                                   torch.from_numpy(absmax).cuda(),
                                   {p: tuple(t.cuda() for t in tl[p]) for p in "qkv"},
                                   wl.alpha_over_r, wl.n_q_heads, wl.n_kv_heads, D,
                                   rope_base=wl.rope_base)
    torch.cuda.synchronize()
    for b, lo in ((0, 0), (B - 1, L - 64)):
        seg = x[b:b + 1, lo:lo + 64].float().numpy()
        ref = O.project_lora_nf4(seg, codes, absmax, nl, wl.alpha_over_r, wl.n_q_heads,
                                 wl.n_kv_heads, D, pos0=lo, rope_base=wl.rope_base)
        for got_t, ref_t, name in zip((q, k, v), ref, "qkv"):
            check_projection(got_t[b:b + 1, :, lo:lo + 64].float().cpu().numpy(), ref_t, "bf16",
                             f"{name} rows {lo}.. of sequence {b}")
