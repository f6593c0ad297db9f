"""Failure detection without a GPU fault: a kernel whose bounded wait runs out
(a barrier nothing completes) must report CCQ_ERR_TIMEOUT through the device
status word, clear it once read, and leave the context usable."""
import ctypes

import pytest
import torch

from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import GLA, TOL, gpu_forward, oracle_forward, rel_err

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout_and_context_survives():
    lib = ccq.load_library()
    lib.ccq_diag_wait_timeout.argtypes = [ctypes.c_void_p]
    lib.ccq_diag_wait_timeout.restype = ctypes.c_int
    ccq.device_status()  # start from a clear status word
    assert lib.ccq_diag_wait_timeout(torch.cuda.current_stream().cuda_stream) == ccq.CCQ_OK
    with pytest.raises(ccq.CCQError) as e:
        ccq.device_status()
    assert e.value.status == ccq.CCQ_ERR_TIMEOUT
    ccq.device_status()  # read once: cleared
    # the same context still runs the hot path correctly
    P = gen.make_inputs(GLA, 1, 130, 2, 128, 128, dtype=torch.bfloat16, seed=41, lam="trained")
    o, _ = gpu_forward(GLA, P, algo="chunkwise")
    ccq.device_status()
    assert rel_err(o, oracle_forward(GLA, P)["o"]) <= TOL[torch.bfloat16]
