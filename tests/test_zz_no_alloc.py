"""The allocation-free decode entry point (kvq_attend_decode_noalloc).

Callers that cannot allocate device memory (plugin hosts that hand an op only
its tensors, allocation-free serving loops, processes whose pool reserves all
free HBM) use this variant: its split-K partials live in the library's static
device scratch instead of the cache's workspace.  It must give the same output
as kvq_attend_decode, call after call (the scratch keeps the previous call's
contents), and refuse shapes whose partials do not fit the scratch.

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
    return got.float().cpu().numpy(), ref.float().cpu().numpy()


def test_matches_existing_entry_point_on_consecutive_calls():
    # first call: a long cache that uses every split
    a = gpu_cache(FORMATS["affine4"], 2, 2, 16, 64, 1100, "bf16")
    k, v, _, _ = kv_pair(2, 2, 1000, 64, "bf16", seed=1)
    a.append(k, v)
    qa = torch.randn(2, 16, 1, 64, dtype=torch.bfloat16, device="cuda")
    got, ref = _decode_both(a, qa)
    assert np.abs(got - ref).max() <= 2e-2
    # second call right after: a short cache of another shape, so most splits
    # are empty and stale partials of the first call sit in the scratch
    b = gpu_cache(FORMATS["sym2"], 1, 4, 8, 128, 64, "bf16")
    k, v, _, _ = kv_pair(1, 4, 40, 128, "bf16", seed=2)
    b.append(k, v)
    qb = torch.randn(1, 8, 1, 128, dtype=torch.bfloat16, device="cuda")
    got, ref = _decode_both(b, qb)
    assert np.abs(got - ref).max() <= 2e-2
    # and the first cache again
    got, ref = _decode_both(a, qa)
    assert np.abs(got - ref).max() <= 2e-2


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
