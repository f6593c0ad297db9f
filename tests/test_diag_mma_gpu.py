"""Every tensor-core operand form the CCQ kernels use, checked in isolation:
D = A B through the kernels' shared-memory tiles, descriptors and tcgen05.mma
sequence, against a plain fp64 matrix product of the same bf16 values."""
import ctypes

import pytest
import torch

from paper_2606_01294_gb300 import ccq

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("a_mn,b_mn,N,K", [(0, 0, 64, 128), (0, 0, 128, 128), (0, 1, 128, 64),
                                           (0, 1, 128, 128), (1, 1, 128, 64), (0, 1, 64, 64),
                                           (1, 0, 128, 128), (1, 0, 64, 64)])
def test_mma_layout(a_mn, b_mn, N, K):
    lib = ccq.load_library()
    lib.ccq_diag_mma.argtypes = [ctypes.c_void_p] * 3 + [ctypes.c_int] * 5 + [ctypes.c_void_p]
    lib.ccq_diag_mma.restype = ctypes.c_int
    g = torch.Generator().manual_seed(N * 7 + K + 3 * a_mn + b_mn)
    A = torch.randn(128, K, generator=g).to(torch.bfloat16).cuda()
    B = torch.randn(K, N, generator=g).to(torch.bfloat16).cuda()
    D = torch.full((128, N), float("nan"), device="cuda")
    st = lib.ccq_diag_mma(A.data_ptr(), B.data_ptr(), D.data_ptr(), 128, N, K, a_mn, b_mn,
                          torch.cuda.current_stream().cuda_stream)
    assert st == 0
    ccq.device_status()
    ref = A.double() @ B.double()
    err = (D.double() - ref).abs().max().item()
    assert err <= 1e-3 * ref.abs().max().item(), f"max abs err {err}"


@pytest.mark.parametrize("a_mn,b_mn,N,K", [(0, 0, 64, 128), (0, 0, 128, 128), (0, 1, 128, 64),
                                           (0, 1, 128, 128), (1, 1, 128, 64), (1, 0, 64, 64)])
def test_mma_m64_layout(a_mn, b_mn, N, K):
    """M = 64 products read back through the 16-lane split TMEM load."""
    lib = ccq.load_library()
    lib.ccq_diag_mma.argtypes = [ctypes.c_void_p] * 3 + [ctypes.c_int] * 5 + [ctypes.c_void_p]
    lib.ccq_diag_mma.restype = ctypes.c_int
    g = torch.Generator().manual_seed(N + K + b_mn + 5 * a_mn)
    A = torch.randn(64, K, generator=g).to(torch.bfloat16).cuda()
    B = torch.randn(K, N, generator=g).to(torch.bfloat16).cuda()
    D = torch.full((128, N), float("nan"), device="cuda")
    st = lib.ccq_diag_mma(A.data_ptr(), B.data_ptr(), D.data_ptr(), 64, N, K, a_mn, b_mn,
                          torch.cuda.current_stream().cuda_stream)
    assert st == 0
    ccq.device_status()
    ref = A.double() @ B.double()
    err = (D[:64].double() - ref).abs().max().item()
    assert err <= 1e-3 * ref.abs().max().item(), f"max abs err {err}"
