"""Host-side checks of the C ABI: the library loads without a GPU, exports
every function include/*.h declares, and rejects bad arguments before any
CUDA call is made."""
import ctypes

import pytest

from paper_2606_01294_gb300 import _build, ccq


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return ccq.load_library()


def test_library_exports_every_header_symbol(lib):
    names = ccq.header_symbols()
    assert {"ccq_gla_fwd", "ccq_gdn_fwd", "ccq_gdn_workspace_size", "ccq_decode_step", "ccq_device_status",
            "ccq_status_string", "ccq_last_error", "ccq_default_params"} <= set(names)
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/ but not exported"


def test_default_params(lib):
    p = ccq._Params()
    lib.ccq_default_params(ctypes.byref(p))
    assert (p.l2norm_qk, p.scale, p.centered, p.chunk, p.algo, p.seq_split) == (1, 0.0, 1, 64, 0, 0)


def test_status_strings(lib):
    for s in range(6):
        assert lib.ccq_status_string(s)
    assert b"unknown" in lib.ccq_status_string(99)


def _gla(lib, ptrs=None, sizes=(1, 4, 1, 128, 128), p=None, dtypes=(0, 0)):
    fake = ctypes.c_void_p(0x10000)  # aligned, never dereferenced on these paths
    args = ptrs if ptrs is not None else [fake] * 5
    return lib.ccq_gla_fwd(*args, *dtypes, *([None] * 4), fake, *([None] * 4),
                           *sizes, None, 0, ctypes.byref(p or ccq.params()), None)


def test_rejects_null_and_misaligned_pointers(lib):
    fake = ctypes.c_void_p(0x10000)
    assert _gla(lib, [None] + [fake] * 4) == ccq.CCQ_ERR_INVALID_ARG
    assert b"NULL" in lib.ccq_last_error()
    assert _gla(lib, [ctypes.c_void_p(0x10002)] + [fake] * 4) == ccq.CCQ_ERR_INVALID_ARG
    assert b"aligned" in lib.ccq_last_error()


def test_rejects_bad_sizes_and_params(lib):
    assert _gla(lib, sizes=(0, 4, 1, 128, 128)) == ccq.CCQ_ERR_INVALID_ARG
    assert _gla(lib, sizes=(1, -1, 1, 128, 128)) == ccq.CCQ_ERR_INVALID_ARG
    assert _gla(lib, sizes=(1, 4, 1, 96, 96)) == ccq.CCQ_ERR_UNSUPPORTED
    assert _gla(lib, sizes=(1, 4, 1, 128, 64)) == ccq.CCQ_ERR_UNSUPPORTED
    assert _gla(lib, p=ccq.params(chunk=32)) == ccq.CCQ_ERR_UNSUPPORTED
    assert _gla(lib, dtypes=(7, 0)) == ccq.CCQ_ERR_INVALID_ARG
    bad = ccq.params()
    bad.algo = 9
    assert _gla(lib, p=bad) == ccq.CCQ_ERR_INVALID_ARG
    # the chunkwise kernel needs bf16 and Dk = 128
    assert _gla(lib, sizes=(1, 4, 1, 64, 64), p=ccq.params(algo="chunkwise")) == ccq.CCQ_ERR_UNSUPPORTED
    assert _gla(lib, dtypes=(1, 1), p=ccq.params(algo="chunkwise")) == ccq.CCQ_ERR_UNSUPPORTED


def test_decode_rejects_bad_backbone_and_gate(lib):
    fake = ctypes.c_void_p(0x10000)
    p = ccq.params()
    st = lib.ccq_decode_step(5, *([fake] * 6), 0, 0, *([fake] * 5), 1, 1, 128, 128, ctypes.byref(p), None)
    assert st == ccq.CCQ_ERR_INVALID_ARG
    st = lib.ccq_decode_step(1, *([fake] * 6), 0, 0, *([fake] * 5), 1, 1, 128, 128, ctypes.byref(p), None)
    assert st == ccq.CCQ_ERR_INVALID_ARG  # GDN decay must be fp32
    st = lib.ccq_decode_step(1, fake, fake, fake, fake, None, fake, 0, 1, *([fake] * 5), 1, 1, 128, 128,
                             ctypes.byref(p), None)
    assert st == ccq.CCQ_ERR_INVALID_ARG  # GDN needs beta


def test_binding_refuses_cpu_tensors():
    import torch
    x = torch.zeros(1, 4, 1, 128, dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="CUDA"):
        ccq.gla_fwd(x, x, x, x, torch.zeros(1, 4, 1))


def test_gdn_workspace_size(lib):
    n = ctypes.c_size_t(7)
    assert lib.ccq_gdn_workspace_size(8, 4096, 16, 128, 128, 0, ctypes.byref(ccq.params()), ctypes.byref(n)) == 0
    assert n.value == 8 * 16 * 64 * 64 * 64 * 2  # Tb: 64 x 64 bf16 per chunk
    assert lib.ccq_gdn_workspace_size(1, 100, 2, 128, 128, 1, ctypes.byref(ccq.params()), ctypes.byref(n)) == 0
    assert n.value == 0  # fp32 inputs run the recurrent kernel
    assert lib.ccq_gdn_workspace_size(1, 100, 2, 128, 128, 0, ctypes.byref(ccq.params(algo="recurrent")),
                                      ctypes.byref(n)) == 0
    assert n.value == 0
    fake = ctypes.c_void_p(0x10000)
    st = lib.ccq_gdn_fwd(*([fake] * 6), 0, *([None] * 4), fake, *([None] * 4), 1, 64, 1, 128, 128,
                         None, 0, ctypes.byref(ccq.params()), None)
    assert st == ccq.CCQ_ERR_INVALID_ARG and b"workspace" in lib.ccq_last_error()


def test_gla_workspace_size_and_split(lib):
    n = ctypes.c_size_t(7)
    seg_bytes = (2 * 128 * 128 + 2 * 128) * 4
    # many sequences: never split
    assert lib.ccq_gla_workspace_size(8, 4096, 16, 128, 128, 0, ctypes.byref(ccq.params()), ctypes.byref(n)) == 0
    assert n.value == 0
    # forced split: 4 segments of a 300-token (5-chunk) sequence -> 3 segments of 2 chunks
    assert lib.ccq_gla_workspace_size(1, 300, 2, 128, 128, 0, ctypes.byref(ccq.params(seq_split=4)),
                                      ctypes.byref(n)) == 0
    assert n.value == 1 * 2 * 3 * seg_bytes
    # split never applies to the recurrent kernel
    assert lib.ccq_gla_workspace_size(1, 300, 2, 128, 128, 1, ctypes.byref(ccq.params(seq_split=4)),
                                      ctypes.byref(n)) == 0
    assert n.value == 0
    fake = ctypes.c_void_p(0x10000)
    st = lib.ccq_gla_fwd(*([fake] * 5), 0, 0, *([None] * 4), fake, *([None] * 4), 1, 300, 2, 128, 128,
                         None, 0, ctypes.byref(ccq.params(seq_split=4)), None)
    assert st == ccq.CCQ_ERR_INVALID_ARG and b"workspace" in lib.ccq_last_error()
    bad = ccq.params()
    bad.seq_split = -1
    assert _gla(lib, p=bad) == ccq.CCQ_ERR_INVALID_ARG


def test_gla_ckpt_and_bwd_workspace_sizes(lib):
    n = ctypes.c_size_t(7)
    assert lib.ccq_gla_ckpt_size(4, 4096, 16, 128, 128, ctypes.byref(n)) == 0
    assert n.value == 4 * 16 * (64 * (65536 + 512) + 65536)
    assert lib.ccq_gla_ckpt_size(1, 65, 1, 128, 128, ctypes.byref(n)) == 0
    assert n.value == 2 * (65536 + 512) + 65536  # ragged tail: two chunks
    assert lib.ccq_gla_ckpt_size(1, 64, 1, 64, 64, ctypes.byref(n)) == ccq.CCQ_ERR_UNSUPPORTED
    p = ctypes.byref(ccq.params(seq_split=1))
    x = 4 * 4 * 4096 * 16 * 128 * 2 + 4 * 16 * 64 * (3 * 512 + 65536 + 3 * 512)  # exchange + per chunk
    assert lib.ccq_gla_bwd_workspace_size(4, 4096, 16, 128, 128, 0, 1, p, ctypes.byref(n)) == 0
    assert n.value == x
    assert lib.ccq_gla_bwd_workspace_size(4, 4096, 16, 128, 128, 0, 0, p, ctypes.byref(n)) == 0
    assert n.value == x + 4 * 16 * (64 * (65536 + 512) + 65536)
    assert lib.ccq_gla_bwd_workspace_size(1, 64, 1, 128, 128, 1, 1, p, ctypes.byref(n)) == ccq.CCQ_ERR_UNSUPPORTED
    assert lib.ccq_gla_bwd_workspace_size(1, 0, 1, 128, 128, 0, 0, p, ctypes.byref(n)) == 0
    assert n.value == 0


def _bwd(lib, ptrs=None, sizes=(1, 64, 1, 128, 128), p=None, dtypes=(0, 0), ws=None, ws_bytes=0, ckpt=None):
    fake = ctypes.c_void_p(0x10000)
    req = ptrs if ptrs is not None else [fake] * 10  # q k v gk lambda dout dq dk dv dgk
    return lib.ccq_gla_bwd(*req[:5], *dtypes, *([None] * 4), req[5], None, None, None, ckpt,
                           *req[6:10], None, None, None, None, *sizes, ws, ws_bytes,
                           ctypes.byref(p or ccq.params(seq_split=1)), None)


def test_gla_bwd_rejects_bad_arguments(lib):
    fake = ctypes.c_void_p(0x10000)
    assert _bwd(lib, dtypes=(1, 1)) == ccq.CCQ_ERR_UNSUPPORTED  # fp32 inputs
    assert _bwd(lib, sizes=(1, 64, 1, 64, 64)) == ccq.CCQ_ERR_UNSUPPORTED
    assert _bwd(lib, p=ccq.params(algo="recurrent")) == ccq.CCQ_ERR_UNSUPPORTED
    assert _bwd(lib, ptrs=[fake] * 5 + [None] + [fake] * 4) == ccq.CCQ_ERR_INVALID_ARG  # no dout
    assert b"NULL" in lib.ccq_last_error()
    assert _bwd(lib) == ccq.CCQ_ERR_INVALID_ARG and b"workspace" in lib.ccq_last_error()
    assert _bwd(lib, ws=ctypes.c_void_p(0x10008), ws_bytes=1 << 30, ckpt=fake) == ccq.CCQ_ERR_INVALID_ARG
    assert b"aligned" in lib.ccq_last_error()
    # no tokens and no state gradients requested: nothing to do
    assert _bwd(lib, sizes=(1, 0, 1, 128, 128)) == ccq.CCQ_OK


def test_gla_fwd_save_rejects_bad_checkpoint_buffer(lib):
    fake = ctypes.c_void_p(0x10000)
    p = ctypes.byref(ccq.params(seq_split=1))
    st = lib.ccq_gla_fwd_save(*([fake] * 5), 0, 0, *([None] * 4), fake, *([None] * 4), 1, 64, 1, 128, 128,
                              None, 0, fake, 1024, p, None)
    assert st == ccq.CCQ_ERR_INVALID_ARG and b"checkpoint" in lib.ccq_last_error()
    st = lib.ccq_gla_fwd_save(*([fake] * 5), 1, 1, *([None] * 4), fake, *([None] * 4), 1, 64, 1, 128, 128,
                              None, 0, fake, 1 << 20, p, None)
    assert st == ccq.CCQ_ERR_UNSUPPORTED  # fp32 inputs have no checkpointing path


def _gdn_bwd(lib, ptrs=None, sizes=(1, 70, 2, 64, 64), ws=None, ws_bytes=0, dtype=1, opt=None):
    fake = ctypes.c_void_p(0x10000)
    req = ptrs if ptrs is not None else [fake] * 6
    o = opt or {}
    # q, k, v, g, beta, lambda, in_dtype, S0, C0, m0, t0, dout, dST, dCT, dmT, dq, dk, dv, dg, dbeta,
    # dlambda, dS0, dC0, dm0
    return lib.ccq_gdn_bwd(*req, dtype, o.get("S0"), None, None, None, fake, None, None, None,
                           fake, fake, fake, fake, fake, None, None, None, None,
                           *sizes, ws, ws_bytes, ctypes.byref(ccq.params()), None)


def test_gdn_bwd_workspace_size_and_rejections(lib):
    need = ctypes.c_size_t(0)
    p = ccq.params()
    chunks = 4 * 16 * 64
    arrays = chunks * (64 * 64 + 5 * 128 * 128 + 2 * 128 + 6 * 64 * 128 + 4 * 64) * 4
    # fp32 inputs: the backward's per-chunk arrays only
    assert lib.ccq_gdn_bwd_workspace_size(4, 4096, 16, 128, 128, 1, ctypes.byref(p), ctypes.byref(need)) == 0
    assert need.value == arrays
    # bf16 inputs with d = 128 also hold the tensor-core forward's workspace (from a 1 KB boundary),
    # which recomputes the forward's per-chunk quantities
    fwd = ctypes.c_size_t(0)
    pf = ccq.params(algo="chunkwise")
    assert lib.ccq_gdn_workspace_size(4, 4096, 16, 128, 128, 0, ctypes.byref(pf), ctypes.byref(fwd)) == 0
    assert lib.ccq_gdn_bwd_workspace_size(4, 4096, 16, 128, 128, 0, ctypes.byref(p), ctypes.byref(need)) == 0
    assert need.value == (arrays + 1023) // 1024 * 1024 + fwd.value
    assert lib.ccq_gdn_bwd_workspace_size(1, 0, 2, 64, 64, 1, ctypes.byref(p), ctypes.byref(need)) == 0
    assert need.value == 0
    assert lib.ccq_gdn_bwd_workspace_size(1, 64, 2, 96, 96, 1, ctypes.byref(p),
                                          ctypes.byref(need)) == ccq.CCQ_ERR_UNSUPPORTED
    fake = ctypes.c_void_p(0x10000)
    assert _gdn_bwd(lib, [None] + [fake] * 5) == ccq.CCQ_ERR_INVALID_ARG
    assert _gdn_bwd(lib, sizes=(1, 70, 0, 64, 64)) == ccq.CCQ_ERR_INVALID_ARG
    assert _gdn_bwd(lib, dtype=5) == ccq.CCQ_ERR_INVALID_ARG
    assert _gdn_bwd(lib, opt={"S0": ctypes.c_void_p(0x10004)}) == ccq.CCQ_ERR_INVALID_ARG
    # a workspace one byte short of the size is refused before any launch
    lib.ccq_gdn_bwd_workspace_size(1, 70, 2, 64, 64, 1, ctypes.byref(p), ctypes.byref(need))
    assert _gdn_bwd(lib, ws=fake, ws_bytes=need.value - 1) == ccq.CCQ_ERR_INVALID_ARG
    assert b"workspace" in lib.ccq_last_error()


def _gdn_dec(lib, ptrs=None, sizes=(1, 70, 2, 64, 64), ws=None, ws_bytes=0, dtype=1):
    fake = ctypes.c_void_p(0x10000)
    req = ptrs if ptrs is not None else [fake] * 6
    # q, k, v, g, beta, lambda, in_dtype, S0, C0, m0, n0, o, ST, CT, mT, nT
    return lib.ccq_gdn_fwd_decayed(*req, dtype, None, None, None, None, fake, None, None, None, None,
                                   *sizes, ws, ws_bytes, ctypes.byref(ccq.params()), None)


def test_gdn_decayed_workspace_size_and_rejections(lib):
    need = ctypes.c_size_t(0)
    p = ccq.params()
    assert lib.ccq_gdn_decayed_workspace_size(8, 4096, 16, 128, 128, 0, ctypes.byref(p),
                                              ctypes.byref(need)) == 0
    assert need.value == 8 * 16 * 64 * (64 * 64 + 3 * 128 * 128 + 2 * 128 + 4) * 4
    fake = ctypes.c_void_p(0x10000)
    assert _gdn_dec(lib, [fake] * 5 + [None]) == ccq.CCQ_ERR_INVALID_ARG
    assert _gdn_dec(lib, sizes=(1, 70, 2, 128, 64)) == ccq.CCQ_ERR_UNSUPPORTED
    assert _gdn_dec(lib, dtype=3) == ccq.CCQ_ERR_INVALID_ARG
    assert _gdn_dec(lib) == ccq.CCQ_ERR_INVALID_ARG  # no workspace
    assert b"workspace" in lib.ccq_last_error()


def test_gdn_spectral_rejects_unknown_contraction(lib):
    fake = ctypes.c_void_p(0x10000)

    def call(contraction, decayed):
        return lib.ccq_gdn_fwd_spectral(*([fake] * 6), 1, None, None, None, None, fake, None, None, None, None,
                                        1, 70, 2, 64, 64, contraction, decayed, None, 0,
                                        ctypes.byref(ccq.params()), None)
    assert call(3, 1) == ccq.CCQ_ERR_INVALID_ARG
    assert b"contraction" in lib.ccq_last_error()
    assert call(-1, 0) == ccq.CCQ_ERR_INVALID_ARG
    assert call(1, 2) == ccq.CCQ_ERR_INVALID_ARG
    assert call(2, 0) == ccq.CCQ_ERR_INVALID_ARG      # valid request, but no workspace
    assert b"workspace" in lib.ccq_last_error()
    # the fixed CG / Taylor counts are bounded only for unit-norm keys
    for contraction in (1, 2):
        st = lib.ccq_gdn_fwd_spectral(*([fake] * 6), 1, None, None, None, None, fake, None, None, None, None,
                                      1, 70, 2, 64, 64, contraction, 0, None, 0,
                                      ctypes.byref(ccq.params(l2norm=False)), None)
        assert st == ccq.CCQ_ERR_UNSUPPORTED
        assert b"l2norm_qk" in lib.ccq_last_error()


def test_varlen_rejects_bad_offsets(lib):
    fake = ctypes.c_void_p(0x10000)

    def call(cu, H=16, backbone=0, fp32=False):
        arr = (ctypes.c_int64 * len(cu))(*cu)
        dt, D = (1, 64) if fp32 else (0, 128)
        return lib.ccq_fwd_varlen(backbone, *([fake] * 6), dt, 1 if backbone else dt,
                                  ctypes.cast(arr, ctypes.c_void_p), len(cu) - 1,
                                  None, None, None, None, fake, None, None, None, None, H, D, D, None, 0,
                                  ctypes.byref(ccq.params()), None)
    assert call([1, 5]) == ccq.CCQ_ERR_INVALID_ARG          # must start at 0
    assert b"cu_seqlens[0]" in lib.ccq_last_error()
    assert call([0, 9, 5]) == ccq.CCQ_ERR_INVALID_ARG       # decreasing
    # the per-sequence path (fp32, d = 64) offsets fp32 [T][H] row pointers: 3 * 2 rows are not
    # 16-byte aligned; the single launch (bf16, d = 128) indexes rows itself and needs no alignment
    assert call([0, 3, 8], H=2, fp32=True) == ccq.CCQ_ERR_INVALID_ARG
    assert b"multiple of 4" in lib.ccq_last_error()
    assert call([0, 3, 8], H=2) == ccq.CCQ_ERR_INVALID_ARG  # single launch: no workspace given
    assert b"workspace" in lib.ccq_last_error()
    assert call([0, 3, 8], backbone=2) == ccq.CCQ_ERR_INVALID_ARG
    arr = (ctypes.c_int64 * 1)(0)
    assert lib.ccq_fwd_varlen(0, *([fake] * 6), 0, 0, ctypes.cast(arr, ctypes.c_void_p), 0, None, None, None, None,
                              fake, None, None, None, None, 16, 128, 128, None, 0, ctypes.byref(ccq.params()),
                              None) == ccq.CCQ_ERR_INVALID_ARG  # no sequences


def test_varlen_argument_checks_pass_for_a_pack(lib):
    """A pack of several sequences (empty ones included) with per-sequence position counters
    passes every argument check: without a GPU the call then fails at its first launch
    (CCQ_ERR_CUDA), not with CCQ_ERR_INVALID_ARG.  Row s of t0 / tT sits 8 bytes after row s-1."""
    fake = ctypes.c_void_p(0x10000)
    cu = [0, 4, 4, 12, 16]
    arr = (ctypes.c_int64 * len(cu))(*cu)

    def call(backbone, beta, algo="auto", fp32=True):
        p = ccq.params(algo=algo)
        dt = 1 if fp32 else 0
        D = 64 if fp32 else 128
        return lib.ccq_fwd_varlen(backbone, fake, fake, fake, fake, beta, fake, dt, 1,
                                  ctypes.cast(arr, ctypes.c_void_p), len(cu) - 1,
                                  fake, fake, fake, fake, fake, fake, fake, fake, fake, 4, D, D, None, 0,
                                  ctypes.byref(p), None)
    for backbone in (0, 1):
        st = call(backbone, fake)
        assert st == ccq.CCQ_ERR_CUDA, (backbone, st, lib.ccq_last_error())
    # every call is checked before the first launch: GDN without beta is rejected as an
    # argument error although sequence 0 alone would have been launched first
    assert call(1, None) == ccq.CCQ_ERR_INVALID_ARG
    assert b"NULL" in lib.ccq_last_error()
    # an empty sequence passes its state through even when the chunkwise path is forced
    # (fp32 inputs make the non-empty ones unsupported there, which is reported, not launched)
    assert call(0, fake, algo="chunkwise") == ccq.CCQ_ERR_UNSUPPORTED
    assert b"chunkwise" in lib.ccq_last_error()


def test_varlen_binding_checks_offsets_against_the_pack():
    import torch
    q = torch.zeros(10, 2, 64)
    for cu, msg in (([1, 10], "start at 0"), ([0, 6, 4, 10], "non-decreasing"), ([0, 4, 12], "packed length")):
        with pytest.raises(ValueError, match=msg):
            ccq.fwd_varlen(0, q, q, q, q, torch.zeros(10, 2), cu)
