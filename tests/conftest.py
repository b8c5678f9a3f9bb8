import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running statistical test")


def bits16(t):
    """Raw bits of a bf16 torch tensor as a uint16 numpy array (fp32 passes through)."""
    import torch
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def bf16_bits_from_float(x):
    """Round float32 values to bf16 (nearest even) and return the bits."""
    import torch
    return bits16(torch.as_tensor(np.asarray(x, np.float32)).to(torch.bfloat16))


@pytest.fixture(scope="session")
def oracle_lib():
    import oracle
    return oracle.load()
