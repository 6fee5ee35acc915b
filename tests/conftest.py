import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libsdsat")
    config.addinivalue_line("markers", "slow: full-size cases (minutes)")


@pytest.fixture(scope="session")
def tiny_shape():
    import synth
    return synth.SHAPES["tiny"]


@pytest.fixture(scope="session")
def tiny_model_cpu(tiny_shape):
    """bf16 weights of the tiny model on the CPU, norm gains != 1 so a dropped gain shows."""
    import synth
    return synth.make_model(tiny_shape, seed=0, device="cpu", gain_std=0.1)


@pytest.fixture(scope="session")
def tiny_model_cpu_unit_gain(tiny_shape):
    import synth
    return synth.make_model(tiny_shape, seed=0, device="cpu")
