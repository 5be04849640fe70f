import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and runs the CUDA library")


@pytest.fixture(scope="session")
def kv():
    """The CUDA binding, with the library built for sm_103a; GPU tests only."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test run without a CUDA device")
    from paper_2608_09225_gb300 import build as kbuild
    kbuild.build()
    from paper_2608_09225_gb300 import kvgov
    kvgov.lib()
    return kvgov
