"""Fixtures for the GPU parity tests: build the library once and require a GPU."""
import pytest
import torch


def require_gpu():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    from paper_2609_04263_gb300 import build, kvq
    build.build()
    kvq.lib()
