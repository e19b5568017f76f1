import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

# The property tests of the oracle need hypothesis, which the CPU test
# environment has; where it is missing (the GPU hosts, which run only the
# gpu-marked tests) the module is left out of collection instead of being
# reported as a skip.
try:
    import hypothesis  # noqa: F401
except ImportError:
    collect_ignore = ["test_oracle_properties.py"]


def pytest_configure(config):
    config.addinivalue_line(
        "markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and libedp.so")


@pytest.fixture(scope="session")
def orc():
    import oracle
    oracle.lib()
    return oracle


@pytest.fixture(scope="session")
def edp_lib():
    """libedp built for sm_103a and loaded; the GPU tests run through it."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test collected on a machine without CUDA")
    from paper_2609_24456_gb300 import build, edp
    build.build()
    edp.lib()
    return edp
