import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


@pytest.fixture(autouse=True)
def _device_error_word_is_clear(request):
    """After every GPU test: the library's device-side error word must be zero.

    Every bounded wait in the kernels (TMA rings, tagged handoffs of the fused
    decode step, merges) that gives up sets this word and returns early, which
    would leave wrong output behind; a test that compares only part of the
    output could miss that, so each GPU test also reads and clears the word."""
    yield
    if request.node.get_closest_marker("gpu") is None:
        return
    import torch
    if not torch.cuda.is_available():
        return
    from paper_2609_04263_gb300 import kvq
    if kvq._lib is None:
        return
    word = kvq.kvq_device_status(torch.cuda.current_stream().cuda_stream)
    assert word == 0, f"device error word {word:#x}: a bounded wait in a kernel gave up"
