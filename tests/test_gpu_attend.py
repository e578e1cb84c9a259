"""Attention parity: GPU decode and prefill attention over the packed cache
against the oracle's fp64 attention over the reconstruction (Sections
3.2-3.3), on the same seeded inputs.  The cache planes are first checked bit
for bit, so both sides attend over the same stored state.  Tolerance:
max-abs 1e-4 (fp32) and 2e-2 (bf16)."""
import math

import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth
from tests.gpu_common import require_gpu
from tests.helpers import ACT, FORMATS, compare_planes, gpu_cache, kv_pair, oracle_cache

pytestmark = pytest.mark.gpu
TOL = {"f32": 1e-4, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def _fill(name, act, B, H, Hq, D, chunks, Tmax):
    spec = FORMATS[name]
    oc = oracle_cache(spec, B, H, D, Tmax, act)
    gc = gpu_cache(spec, B, H, Hq, D, Tmax, act)
    for i, n in enumerate(chunks):
        kt, vt, kn, vn = kv_pair(B, H, n, D, act, seed=5, stream=i)
        gc.append(kt, vt)
        oc.append(kn, vn)
    torch.cuda.synchronize()
    compare_planes(gc, oc)
    return gc, oc


def _q(B, Hq, L, D, act, stream):
    q = torch.from_numpy(synth.queries((B, Hq, L, D), seed=9, stream=stream)).to(ACT[act])
    return q.cuda(), q.float().numpy()


DECODE = [
    ("affine4", "bf16", 2, 2, 16, 64, [300, 1]),
    ("affine4", "f32", 1, 4, 4, 64, [512, 1]),
    ("affine2", "bf16", 1, 2, 8, 128, [257]),
    ("sym2", "bf16", 2, 2, 16, 64, [1000, 25]),
    ("sym4", "bf16", 1, 1, 1, 64, [33]),
    ("float", "bf16", 1, 2, 4, 64, [100]),
    ("float", "f32", 1, 2, 2, 256, [70]),
    ("affine4_g128", "bf16", 1, 2, 4, 256, [200]),
    ("kivi2", "bf16", 2, 2, 8, 128, [300, 1, 1]),
    ("kivi_r0", "bf16", 1, 2, 4, 64, [95]),
    ("kvarn", "bf16", 1, 2, 4, 256, [128 + 64 * 2 + 9]),
    ("kvarn_small", "bf16", 2, 2, 4, 64, [40 + 32 * 3 + 31, 1]),
    ("kvarn_small", "f32", 1, 1, 2, 64, [20]),      # sinks only
    ("affine4", "bf16", 1, 1, 16, 128, [777]),      # GQA group 16
    ("sym2", "bf16", 3, 2, 6, 64, [65]),            # odd group, ragged chunk
    ("kivi2", "bf16", 1, 1, 8, 64, [1000, 7]),      # chunks straddle the residual edge
    ("affine2", "bf16", 2, 4, 8, 64, [4095, 1]),
    # shapes large enough for the streaming decode (>= 16 blocks of 32 tokens
    # per CTA); many short heads put up to 8 heads in one ring stage
    ("affine4", "bf16", 160, 16, 32, 64, [20]),
    ("sym2", "bf16", 100, 16, 32, 64, [40]),         # two blocks per head, the second partial
    ("kivi2", "bf16", 160, 16, 64, 128, [31]),       # residual only: nothing coded
    ("kivi2", "bf16", 8, 8, 32, 128, [1297, 3]),     # heads spanning several CTAs
    ("affine2", "bf16", 4, 8, 64, 128, [2500]),      # GQA 8, D 128
    # KVarN long enough for the streaming kernel over the coded tokens (the
    # sinks and staged tokens go through the split kernel, then one combine)
    ("kvarn", "bf16", 8, 8, 16, 256, [1500]),
    ("kvarn_small", "bf16", 16, 8, 32, 64, [700, 1]),
    # 8-bit caches (the paper's 2/4/8-bit operating points)
    ("affine8", "bf16", 2, 2, 8, 64, [300, 1]),
    ("affine8", "f32", 1, 2, 2, 64, [129]),
    ("sym8", "bf16", 1, 2, 8, 128, [517]),
    ("affine8_g64", "bf16", 2, 1, 4, 128, [1000, 3]),
    ("kivi_k8", "bf16", 1, 2, 8, 128, [400, 1]),
]


@pytest.mark.parametrize("name,act,B,H,Hq,D,chunks", DECODE)
def test_decode_parity(name, act, B, H, Hq, D, chunks):
    T = sum(chunks)
    gc, oc = _fill(name, act, B, H, Hq, D, chunks, T + 8)
    qt, qn = _q(B, Hq, 1, D, act, 0)
    got = gc.attend_decode(qt).float().cpu().numpy()
    ref = O.attend(oc, qn)
    err = np.abs(got - ref).max()
    assert err <= TOL[act], f"max-abs {err}"


PREFILL = [
    ("affine4", "bf16", 2, 2, 16, 64, [0], 300),
    ("affine4", "bf16", 1, 2, 16, 64, [200], 129),
    ("affine4", "f32", 1, 4, 4, 64, [0], 512),
    ("sym2", "bf16", 1, 2, 16, 64, [64], 100),
    ("float", "bf16", 1, 2, 4, 128, [10], 50),
    ("affine2", "bf16", 1, 2, 2, 256, [0], 97),
    ("kivi2", "bf16", 1, 2, 8, 128, [100], 250),
    ("kivi_r0", "bf16", 1, 1, 4, 64, [0], 70),
    ("kvarn", "bf16", 1, 2, 4, 256, [100], 200),
    ("kvarn_small", "bf16", 1, 2, 2, 64, [0], 150),
    ("affine4", "bf16", 1, 1, 16, 64, [0], 130),     # GQA 16: 8 queries per CTA
    ("sym4", "bf16", 2, 1, 6, 128, [37], 90),        # group 6 does not divide the rows
    ("affine4", "bf16", 1, 1, 2, 256, [50], 333),
    # head_dim 128 on the 256-row tensor-core kernel: several 64-token KV
    # tiles, GQA 1 (the two query tiles at different positions), 4 and 16
    # (16 queries per CTA), a KIVI residual window inside the last tiles, a
    # prefill shorter than one tile
    ("affine4", "bf16", 2, 2, 8, 128, [300], 700),
    ("kivi2", "bf16", 1, 2, 8, 128, [0], 1000),
    ("kivi2", "bf16", 2, 1, 1, 128, [64], 333),
    ("sym2", "bf16", 1, 1, 16, 128, [0], 200),
    ("affine2", "bf16", 1, 2, 4, 128, [0], 40),
    ("sym4", "bf16", 1, 2, 8, 128, [500], 129),
    # 8-bit caches
    ("affine8", "bf16", 1, 2, 8, 64, [100], 300),
    ("affine8", "f32", 1, 1, 2, 64, [0], 97),
    ("sym8", "bf16", 2, 1, 4, 128, [64], 200),
    ("affine8_g64", "bf16", 1, 2, 4, 256, [0], 130),
    ("kivi_k8", "bf16", 1, 2, 8, 128, [200], 180),
]


@pytest.mark.parametrize("name,act,B,H,Hq,D,before,L", PREFILL)
def test_prefill_parity(name, act, B, H, Hq, D, before, L):
    before = [n for n in before if n]
    Tmax = sum(before) + L + 8
    gc, oc = _fill(name, act, B, H, Hq, D, before + [L], Tmax)
    qt, qn = _q(B, Hq, L, D, act, 1)
    got = gc.attend_prefill(qt).float().cpu().numpy()
    ref = O.attend(oc, qn)
    err = np.abs(got - ref).max()
    assert err <= TOL[act], f"max-abs {err}"


def test_decode_split_equals_single_tile_reference():
    """Many splits over a long cache merge to the same output as the oracle."""
    gc, oc = _fill("affine4", "bf16", 1, 1, 8, 64, [2048], 2100)
    qt, qn = _q(1, 8, 1, 64, "bf16", 3)
    got = gc.attend_decode(qt).float().cpu().numpy()
    assert np.abs(got - O.attend(oc, qn)).max() <= 2e-2


def test_attend_wrong_heads_rejected():
    from paper_2609_04263_gb300 import kvq
    gc, _ = _fill("affine4", "bf16", 1, 2, 4, 64, [10], 20)
    qt, _ = _q(1, 2, 1, 64, "bf16", 0)
    with pytest.raises(kvq.KvqError):
        gc.attend_decode(qt)
