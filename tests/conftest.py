import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a); runs the CUDA library")
    config.addinivalue_line("markers", "slow: long CPU-side check")


@pytest.fixture(scope="session")
def oracle_lib():
    from oracle import build_oracle
    return build_oracle()


@pytest.fixture(scope="session")
def cuda_lib():
    """The CUDA library, built in-tree if missing (nvcc cross-compiles without a GPU).
    FADEMEM_CUDA_LIB names another build (the sanitizer tests use one built with ASan/UBSan)."""
    from paper_2606_10671_gb300 import build
    return os.environ.get("FADEMEM_CUDA_LIB") or build.build_library()
