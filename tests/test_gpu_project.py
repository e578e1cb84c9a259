"""Projection parity: GPU Q/K/V with explicit LoRA branches and RoPE against
the oracle's fp64 projection (Section 3, Eq. 1 and Eq. lora), same seeded
inputs.  Tolerance, per (sequence, head): max-abs difference from the oracle
rounded to the activation dtype over that head's max-abs oracle value, 1e-2
(bf16), 1e-5 (fp32)."""
import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu
from tests.helpers import ACT, check_projection

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def _case(act, B, L, d_in, Hq, Hkv, D, ranks, outlier=0.01, seed=0):
    wl = synth.Workload(name="t", dtype=act, layers=1, d_in=d_in, n_q_heads=Hq,
                        n_kv_heads=Hkv, head_dim=D, rope_base=10000.0, batch=B, prefill=L,
                        decode=0, fmt=1, key_bits=4, value_bits=4, group_size=32, rank=8,
                        outlier_frac=outlier)
    x = synth.hidden_states((B, L, d_in), outlier_frac=outlier, seed=seed)
    w, _ = synth.layer_weights(wl, 0, seed=seed)
    lora = {}
    for i, p in enumerate("qkv"):
        r = ranks[i]
        if r == 0:
            lora[p] = None
            continue
        _, lr = synth.layer_weights(wl, 1 + i, seed=seed, rank=r)
        lora[p] = lr[p]
    dt = ACT[act]
    tx = torch.from_numpy(x).to(dt)
    tw = torch.from_numpy(w).to(dt)
    tl = {p: None if v is None else tuple(torch.from_numpy(t).to(dt) for t in v)
          for p, v in lora.items()}
    nx = tx.float().numpy()
    nw = tw.float().numpy()
    nl = {p: None if v is None else tuple(t.float().numpy() for t in v) for p, v in tl.items()}
    return (tx.cuda(), tw.cuda(), {p: None if v is None else tuple(t.cuda() for t in v)
                                   for p, v in tl.items()}), (nx, nw, nl)


CASES = [
    ("bf16", 2, 37, 512, 8, 2, 64, (16, 16, 16), 5, 10000.0),
    ("bf16", 1, 130, 256, 4, 2, 128, (64, 0, 8), 0, 500000.0),
    ("bf16", 3, 5, 384, 2, 2, 256, (0, 32, 32), 900, 10000.0),
    ("bf16", 4, 1, 512, 8, 2, 64, (16, 16, 16), 2048, 10000.0),
    # decode shapes of the weight-streaming kernel: 8B-like (16 rows, 4096
    # channels, ranges spanning projections), 12B-like (a ragged last stage,
    # D = 256), a two-chunk last stage with 8- and 64-rank factors and one
    # CTA per pair-tile, and 24/8/40-rank factors (part-filled U tiles)
    ("bf16", 16, 1, 4096, 32, 8, 128, (16, 16, 16), 8200, 500000.0),
    ("bf16", 4, 1, 3840, 16, 8, 256, (32, 32, 32), 8700, 10000.0),
    ("bf16", 1, 1, 2112, 4, 1, 64, (8, 0, 64), 3, 10000.0),
    ("bf16", 2, 4, 1024, 6, 2, 64, (24, 8, 40), 0, 10000.0),
    # d_in above the streaming kernel's range: the per-tile decode kernel
    ("bf16", 3, 1, 4160, 4, 2, 64, (16, 0, 8), 11, 10000.0),
    ("bf16", 1, 64, 256, 4, 4, 64, (0, 0, 0), 0, 0.0),
    ("f32", 1, 96, 256, 4, 4, 64, (8, 8, 8), 0, 10000.0),
    ("f32", 1, 1, 256, 4, 4, 64, (8, 8, 8), 511, 10000.0),
]


@pytest.mark.parametrize("act,B,L,d_in,Hq,Hkv,D,ranks,pos0,base", CASES)
def test_project_parity(act, B, L, d_in, Hq, Hkv, D, ranks, pos0, base):
    from paper_2609_04263_gb300 import api
    (tx, tw, tl), (nx, nw, nl) = _case(act, B, L, d_in, Hq, Hkv, D, ranks)
    got = api.project_lora(tx, tw, tl, 2.0, Hq, Hkv, D, pos0=pos0, rope_base=base)
    ref = O.project_lora(nx, nw, nl, 2.0, Hq, Hkv, D, pos0=pos0, rope_base=base)
    for name, g, r in zip("qkv", got, ref):
        check_projection(g.float().cpu().numpy(), r, act, name)
