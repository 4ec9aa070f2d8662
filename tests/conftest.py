import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running")


def pytest_collection_modifyitems(config, items):
    # a gpu test with no GPU present is an error, not a skip, when the marker is selected
    pass


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle
    oracle.build()
    return oracle


@pytest.fixture(scope="session")
def wl():
    from paper_2608_03579_gb300 import workloads
    workloads.build()
    return workloads


@pytest.fixture(scope="session")
def salt_lib():
    """Build libsalt.so in-tree (nvcc, sm_103a) and import the binding."""
    from paper_2608_03579_gb300 import _build
    _build.build()
    from paper_2608_03579_gb300 import salt
    return salt
