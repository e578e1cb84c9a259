"""The allocation-free decode entry point (kvq_attend_decode_noalloc).

Callers that cannot allocate device memory (plugin hosts that hand an op only
its tensors, allocation-free serving loops, processes whose pool reserves all
free HBM) use this variant: its split-K partials live in the library's static
device scratch instead of the cache's workspace.  It launches the same
kernels on the same inputs as kvq_attend_decode with only the partials'
address changed, so its output must be bit for bit the same, call after call
(the scratch keeps the previous call's contents), and it must refuse shapes
whose partials do not fit the scratch.

The caches below reach every kernel that writes or reads the partials: the
persistent streaming decode (a long affine cache), the split kernel with its
in-kernel merge (short caches), the KVarN tensor-core kernel with its sink
kernel, whose last CTA merges (a long KVarN cache), and the fp32 generic kernel
with its combine.  Calls on different caches are interleaved so that rows another path
left in the scratch are there when the next one runs.

Collected last so that a failure here cannot hide the other GPU tests.
"""
import math

import numpy as np
import pytest
import torch

from tests.gpu_common import require_gpu
from tests.helpers import FORMATS, gpu_cache, kv_pair

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def _decode_both(gc, q):
    from paper_2609_04263_gb300 import kvq
    stream = torch.cuda.current_stream().cuda_stream
    scale = 1.0 / math.sqrt(q.shape[-1])
    ref = torch.empty_like(q)
    got = torch.empty_like(q)
    kvq.kvq_attend_decode(gc.handle, q.data_ptr(), q.shape[1], scale, ref.data_ptr(), stream)
    kvq.kvq_attend_decode_noalloc(gc.handle, q.data_ptr(), q.shape[1], scale, got.data_ptr(),
                                  stream)
    torch.cuda.synchronize()
    return got, ref


def _same_bits(got, ref, what):
    a = got.contiguous().view(torch.int16 if got.element_size() == 2 else torch.int32)
    b = ref.contiguous().view(torch.int16 if ref.element_size() == 2 else torch.int32)
    n = int((a != b).sum())
    err = float((got.float() - ref.float()).abs().max())
    assert n == 0, f"{what}: {n} outputs differ from kvq_attend_decode (max-abs {err:.3e})"


def _filled(spec, B, H, Hq, D, T, act, seed):
    c = gpu_cache(spec, B, H, Hq, D, T + 8, act)
    k, v, _, _ = kv_pair(B, H, T, D, act, seed=seed)
    c.append(k, v)
    g = torch.Generator(device="cuda").manual_seed(seed)
    q = torch.randn(B, Hq, 1, D, device="cuda", generator=g).to(k.dtype)
    return c, q


def test_matches_existing_entry_point_on_consecutive_calls():
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    # B x Hkv = 16 sequences x heads; 16 x T / 32 blocks >= 16 per SM takes
    # the persistent streaming kernel
    t_stream = 16 * sms * 32 // 16 + 200
    cases = {
        "streaming (affine 4-bit, long)": _filled(FORMATS["affine4"], 4, 4, 32, 64, t_stream,
                                                  "bf16", 1),
        "split kernel (affine 4-bit, short)": _filled(FORMATS["affine4"], 2, 2, 16, 64, 1000,
                                                      "bf16", 2),
        "split kernel (symmetric 2-bit, D 128)": _filled(FORMATS["sym2"], 1, 4, 8, 128, 40,
                                                         "bf16", 3),
        # 2 x 2 heads, up to 60 CTAs: 4 x coded / 32 >= 16 x 60 needs 7680 coded tokens
        "KVarN tensor-core kernel + sinks with the merge": _filled(FORMATS["kvarn_small"], 2, 2, 8,
                                                              64, 7800, "bf16", 4),
        "generic fp32 kernel + combine": _filled(FORMATS["affine4"], 2, 2, 4, 64, 300, "f32", 5),
    }
    # two rounds in a row over all paths: each call finds the other paths'
    # partials (or its own from the previous round) in the static scratch
    for rnd in range(2):
        for what, (c, q) in cases.items():
            got, ref = _decode_both(c, q)
            _same_bits(got, ref, f"round {rnd}: {what}")
            assert torch.isfinite(got.float()).all()


def test_rejects_partials_beyond_the_static_scratch():
    from paper_2609_04263_gb300 import kvq
    # 16 x 64 q heads x 32 splits x 258 floats > 1,048,576
    big = gpu_cache(FORMATS["affine4"], 16, 8, 64, 256, 8, "bf16")
    k, v, _, _ = kv_pair(16, 8, 4, 256, "bf16")
    big.append(k, v)
    q = torch.zeros(16, 64, 1, 256, dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(q)
    with pytest.raises(kvq.KvqError) as ei:
        kvq.kvq_attend_decode_noalloc(big.handle, q.data_ptr(), 64, 0.0625, out.data_ptr(),
                                      torch.cuda.current_stream().cuda_stream)
    assert ei.value.status == kvq.KVQ_ERR_CAPACITY
    assert "static scratch" in kvq.kvq_last_error()
