import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running case")


def micro_workload(**kw):
    """A very small LLaMA-shaped decoder with GQA for fast oracle tests."""
    import synth
    w = synth.Workload("micro", 2, 64, 4, 2, 16, 96, 64, 6, 12, 3, 0, skip=[1, 2])
    for k, v in kw.items():
        setattr(w, k, v)
    return w


@pytest.fixture(scope="session")
def tiny():
    import synth
    return synth.workloads()["tiny"]


@pytest.fixture(scope="session")
def tiny_weights(tiny):
    import synth
    return synth.host_weights(tiny, seed=1)
