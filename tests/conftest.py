import ctypes
import os
import shutil
import subprocess
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


def load_gdn_emu(path):
    """ctypes handle of a host build of tests/host_emu/gdn_cuda_core_emu.cpp."""
    lib = ctypes.CDLL(path)
    lib.gdn_bwd_emu.argtypes = [ctypes.c_int] * 7 + [ctypes.c_float] + [ctypes.c_void_p] * 3
    lib.gdn_bwd_emu.restype = ctypes.c_int
    lib.gdn_spectral_emu.argtypes = [ctypes.c_int] * 7 + [ctypes.c_float, ctypes.c_int, ctypes.c_int,
                                                          ctypes.c_void_p, ctypes.c_void_p]
    lib.gdn_spectral_emu.restype = ctypes.c_int
    return lib


@pytest.fixture(scope="session")
def gdn_emu(tmp_path_factory):
    """The CUDA-core Gated DeltaNet kernels compiled for the host (CPU tests of their arithmetic)."""
    gxx = shutil.which("g++")
    inc = "/usr/local/cuda/include"
    if gxx is None or not os.path.isdir(inc):
        pytest.skip("g++ or the CUDA headers are not available")
    src = os.path.join(ROOT, "tests", "host_emu", "gdn_cuda_core_emu.cpp")
    out = str(tmp_path_factory.mktemp("gdn_emu") / "gdn_cuda_core_emu.so")
    r = subprocess.run([gxx, "-O2", "-std=c++17", "-fPIC", "-shared", "-I" + inc, src, "-o", out],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr[-4000:]
    return load_gdn_emu(out)
