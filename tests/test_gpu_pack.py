"""Quantize-and-pack parity: the GPU planes equal the oracle's bit for bit
(codes, fp16 scales/offsets, KVarN row/column scales, full-precision windows)
for every format, on the same seeded inputs, across chunked appends."""
import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from tests.gpu_common import require_gpu
from tests.helpers import FORMATS, compare_planes, gpu_cache, kv_pair, oracle_cache

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


CASES = [
    ("affine4", "bf16", 2, 3, 64, [200, 1, 55, 129]),
    ("affine2", "bf16", 2, 2, 128, [300, 7]),
    ("affine8_g64", "f32", 1, 2, 128, [77, 64]),
    ("affine4_g128", "bf16", 1, 2, 256, [150, 3]),
    ("sym2", "bf16", 2, 2, 64, [256, 3]),
    ("sym4", "f32", 1, 4, 64, [100, 1, 1]),
    # the smallest groups: one and two lanes per group
    ("sym4_g8", "bf16", 2, 3, 64, [90, 1, 17]),
    ("affine2_g16", "bf16", 1, 2, 128, [65, 2]),
    ("float", "bf16", 2, 2, 64, [50, 13]),
    ("float", "f32", 1, 2, 128, [9, 1]),
    ("kivi2", "bf16", 2, 2, 128, [300, 1, 1, 40, 33]),
    ("kivi_r0", "bf16", 1, 2, 64, [31, 1, 64, 5]),
    # KIVI blocks of 64 tokens: the flush kernel for other group sizes
    ("kivi_g64", "bf16", 2, 2, 128, [200, 1, 70]),
    ("kivi2", "bf16", 1, 2, 256, [170, 2]),
    # 4- and 8-bit KIVI keys in 32-token blocks (the compile-time flush)
    ("kivi_k4", "bf16", 2, 2, 128, [150, 1, 40]),
    ("kivi_k8", "bf16", 1, 2, 64, [100, 3]),
    ("kvarn_small", "bf16", 1, 2, 64, [70, 1, 1, 100]),
    ("kvarn", "bf16", 1, 2, 256, [330, 60]),
    ("kvarn_small", "f32", 1, 1, 128, [45, 64]),
]


@pytest.mark.parametrize("name,act,B,H,D,chunks", CASES)
def test_pack_parity(name, act, B, H, D, chunks):
    spec = FORMATS[name]
    T = sum(chunks)
    Tmax = T + 17
    oc = oracle_cache(spec, B, H, D, Tmax, act)
    gc = gpu_cache(spec, B, H, H, D, Tmax, act)
    t = 0
    for i, n in enumerate(chunks):
        kt, vt, kn, vn = kv_pair(B, H, n, D, act, seed=11, stream=i)
        gc.append(kt, vt)
        oc.append(kn, vn)
        t += n
        if i in (0, len(chunks) - 1):
            torch.cuda.synchronize()
            compare_planes(gc, oc)


@pytest.mark.parametrize("name", ["affine4", "affine2", "sym2", "sym4", "kivi_r0"])
def test_pack_edge_values(name):
    """Constant groups (scale floor), -0.0, exact .5 ties and large magnitudes."""
    spec = FORMATS[name]
    B, H, L, D = 1, 2, 64, 64
    k = np.random.default_rng(0).standard_normal((B, H, L, D)).astype(np.float32)
    k[:, :, 0] = 0.75                         # constant groups
    k[:, :, 1] = -0.0                         # negative zero
    k[:, :, 2, :32] = np.arange(32) * 0.5     # grid with ties
    k[:, :, 3] *= 3000.0                      # large values (fp16-safe scales)
    k[:, :, 4, :32] = 1e-30                   # tiny values: s floors at 1e-8
    # quotients exactly on a half-integer (scale 1): ties to even, for 4-bit
    # affine (0 .. 15), 2-bit affine (0 .. 3) and 4-bit symmetric (-7 .. 7)
    k[:, :, 5, :32] = np.concatenate([[0.0, 15.0], np.arange(15) + 0.5, np.arange(15) + 0.25])
    k[:, :, 6, :32] = np.concatenate([[0.0, 3.0], np.tile([0.5, 1.5, 2.5], 10)])
    k[:, :, 7, :32] = np.concatenate([[-7.0, 7.0, 0.0, 0.0], np.arange(-7, 7) + 0.5,
                                      np.arange(-7, 7) + 0.5])
    v = k[:, :, ::-1].copy()
    kt = torch.from_numpy(k).to(torch.bfloat16)
    vt = torch.from_numpy(v).to(torch.bfloat16)
    oc = oracle_cache(spec, B, H, D, 128, "bf16")
    gc = gpu_cache(spec, B, H, H, D, 128, "bf16")
    oc.append(kt.float().numpy(), vt.float().numpy())
    gc.append(kt.cuda(), vt.cuda())
    torch.cuda.synchronize()
    compare_planes(gc, oc)


def test_empty_append_is_noop():
    spec = FORMATS["affine4"]
    gc = gpu_cache(spec, 1, 1, 1, 64, 32, "bf16")
    e = torch.empty(1, 1, 0, 64, dtype=torch.bfloat16, device="cuda")
    gc.append(e, e)
    assert gc.tokens == 0


def test_capacity_error_leaves_cache_unchanged():
    from paper_2609_04263_gb300 import kvq
    spec = FORMATS["affine4"]
    gc = gpu_cache(spec, 1, 1, 1, 64, 40, "bf16")
    kt, vt, _, _ = kv_pair(1, 1, 32, 64, "bf16")
    gc.append(kt, vt)
    kt, vt, _, _ = kv_pair(1, 1, 9, 64, "bf16", stream=1)
    with pytest.raises(kvq.KvqError) as ei:
        gc.append(kt, vt)
    assert ei.value.status == kvq.KVQ_ERR_CAPACITY and gc.tokens == 32
