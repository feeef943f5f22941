import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the compiled liblookme.so")
    config.addinivalue_line("markers", "slow: full-size workload (tens of GB on the device)")


@pytest.fixture(scope="session")
def oracle():
    import oracle as oracle_pkg

    return oracle_pkg.Oracle()


@pytest.fixture(scope="session")
def lookme_lib():
    """The CUDA library through its Python binding (GPU tests only)."""
    import torch

    if not torch.cuda.is_available():
        raise RuntimeError("GPU test collected on a machine without CUDA; run with -m 'not gpu'")
    from paper_2607_16305_gb300 import lookme

    return lookme.load()
