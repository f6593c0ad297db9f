"""ccq_gla_fwd_fixed_scratch: the CCQ-GLA forward for callers that cannot give
the library device memory (everything it needs beyond the caller's inputs and
outputs lives in a fixed array inside the library).  Checked through the C ABI
against ccq_gla_fwd with a caller workspace, on two calls in a row, with
sequences split into segments so the fixed scratch is really used."""
import ctypes

import pytest
import torch

from paper_2606_01294_gb300 import _build, ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import TOL, rel_err

pytestmark = pytest.mark.gpu

_VP, _I = ctypes.c_void_p, ctypes.c_int


@pytest.fixture(scope="module")
def lib():
    _build.build()
    lib = ccq.load_library()
    lib.ccq_gla_fwd_fixed_scratch.argtypes = ([_VP] * 5 + [_I, _I] + [_VP] * 9 + [_I] * 5
                                              + [ctypes.POINTER(ccq._Params), _VP])
    lib.ccq_gla_fwd_fixed_scratch.restype = _I
    return lib


def _ptr(x):
    return None if x is None else ctypes.c_void_p(x.data_ptr())


def _call(lib, fixed, D, B, T, H, p, ws=None):
    o = torch.empty(B, T, H, 128, dtype=torch.bfloat16, device="cuda")
    st = ccq.CCQState.empty(B, H, 128, 128, "cuda")
    stream = _VP(torch.cuda.current_stream().cuda_stream)
    head = [_ptr(D["q"]), _ptr(D["k"]), _ptr(D["v"]), _ptr(D["gate"]), _ptr(D["lam"]), 0, 0,
            None, None, None, None, _ptr(o), _ptr(st.S), _ptr(st.C), _ptr(st.m), _ptr(st.t),
            B, T, H, 128, 128]
    if fixed:
        rc = lib.ccq_gla_fwd_fixed_scratch(*head, ctypes.byref(p), stream)
    else:
        rc = lib.ccq_gla_fwd(*head, _ptr(ws), 0 if ws is None else ws.numel(), ctypes.byref(p), stream)
    assert rc == 0, lib.ccq_last_error()
    torch.cuda.synchronize()
    return o, st


def test_fixed_scratch_matches_workspace_entry_point_twice(lib):
    B, T, H = 1, 1200, 4  # 19 chunks per sequence
    p = ccq.params(seq_split=3)
    ws = ccq.gla_workspace(B, T, H, 128, 128, "cuda", seq_split=3)
    assert ws is not None and ws.numel() > 0  # the split really needs scratch
    for seed in (61, 62):  # two calls in a row, different data
        P = gen.make_inputs(gen.GLA, B, T, H, 128, 128, dtype=torch.bfloat16, seed=seed, lam="trained",
                            keys="structured")
        D = {n: (None if x is None else x.cuda()) for n, x in P.items()}
        o_ref, s_ref = _call(lib, False, D, B, T, H, p, ws)
        o_fix, s_fix = _call(lib, True, D, B, T, H, p)
        ccq.device_status()
        tol = TOL[torch.bfloat16]
        assert rel_err(o_fix, o_ref.double().cpu().numpy()) <= tol
        for n in ("S", "C", "m"):
            assert rel_err(getattr(s_fix, n), getattr(s_ref, n).double().cpu().numpy()) <= tol, n
        assert torch.equal(s_fix.t, s_ref.t)


def test_fixed_scratch_rejects_oversized_request(lib):
    # 64 sequences x 20 segments x 129 KiB is beyond the 24 MiB fixed scratch
    B, T, H = 4, 64 * 20, 16
    p = ccq.params(seq_split=20)
    fake = torch.empty(16, dtype=torch.bfloat16, device="cuda")
    head = [_ptr(fake)] * 5 + [0, 0] + [None] * 4 + [_ptr(fake)] + [None] * 4 + [B, T, H, 128, 128]
    rc = lib.ccq_gla_fwd_fixed_scratch(*head, ctypes.byref(p), None)
    assert rc == ccq.CCQ_ERR_INVALID_ARG
    assert b"fixed scratch" in lib.ccq_last_error()
