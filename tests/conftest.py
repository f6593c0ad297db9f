import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle
    oracle.build_oracle()
    return oracle


# Parity tests of entry points whose kernels have not yet run on a GPU.  They are collected
# (moved up into tests/) once a GPU run has passed them, so that an unverified kernel never
# runs first inside the suite.
collect_ignore = ["gpu_pending"]
