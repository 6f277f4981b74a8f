import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103) and the built CUDA library")


def read_golden(name):
    """key -> list of floats, from a tests/golden/*.txt fixture ('#' lines are citations)."""
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            parts = line.split()
            if parts[0][0].isalpha():
                out[parts[0]] = [float(v) for v in parts[1:]]
            else:
                out.setdefault("_rows", []).append([float(v) for v in parts])
    return out


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle
    oracle.lib()
    return oracle


def bf16_bits(t):
    """torch bf16 tensor -> numpy uint16 bit patterns (on the host)."""
    import numpy as np
    import torch
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
