"""Python binding of libccq.so (include/ccq.h): argument marshalling only.

Every step of the CCQ computation runs in the library's CUDA kernels; this
module checks tensor placement/dtype/layout, allocates outputs with torch on
the input's device, and passes raw device pointers plus the current CUDA
stream through ctypes.  There is no CPU path: if the library is missing, or a
tensor is not on a CUDA device, the call raises.
"""
from __future__ import annotations

import ctypes
import os
import re
from dataclasses import dataclass
from typing import Optional

import torch

from . import _build

CCQ_OK, CCQ_ERR_INVALID_ARG, CCQ_ERR_UNSUPPORTED, CCQ_ERR_CUDA, CCQ_ERR_TIMEOUT, CCQ_ERR_RANGE = range(6)
BF16, FP32 = 0, 1
ALGO = {"auto": 0, "recurrent": 1, "chunkwise": 2, "wide": 3}
GLA, GDN = 0, 1


class CCQError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"[ccq status {status}] {msg}")
        self.status = status


class _Params(ctypes.Structure):
    _fields_ = [("l2norm_qk", ctypes.c_int), ("scale", ctypes.c_float),
                ("centered", ctypes.c_int), ("chunk", ctypes.c_int),
                ("algo", ctypes.c_int), ("seq_split", ctypes.c_int)]


_lib = None
_VP = ctypes.c_void_p
_I = ctypes.c_int


def library_path() -> str:
    return _build.LIB_PATH


def load_library() -> ctypes.CDLL:
    """Open libccq.so (it must have been built); raises if it is absent."""
    global _lib
    if _lib is None:
        path = _build.LIB_PATH
        if not os.path.exists(path):
            raise RuntimeError(
                f"{path} is missing: build the CUDA library first "
                "(python -c 'import __graft_entry__ as g; g.build()')")
        lib = ctypes.CDLL(path)
        lib.ccq_default_params.argtypes = [ctypes.POINTER(_Params)]
        lib.ccq_default_params.restype = None
        lib.ccq_status_string.argtypes = [_I]
        lib.ccq_status_string.restype = ctypes.c_char_p
        lib.ccq_last_error.argtypes = []
        lib.ccq_last_error.restype = ctypes.c_char_p
        lib.ccq_device_status.argtypes = [_VP]
        lib.ccq_device_status.restype = _I
        lib.ccq_gla_fwd.argtypes = ([_VP] * 5 + [_I, _I] + [_VP] * 9 + [_I] * 5
                                    + [_VP, ctypes.c_size_t, ctypes.POINTER(_Params), _VP])
        lib.ccq_gla_fwd.restype = _I
        lib.ccq_gla_workspace_size.argtypes = ([_I] * 6 + [ctypes.POINTER(_Params),
                                                           ctypes.POINTER(ctypes.c_size_t)])
        lib.ccq_gla_workspace_size.restype = _I
        lib.ccq_gdn_fwd.argtypes = ([_VP] * 6 + [_I] + [_VP] * 9 + [_I] * 5
                                    + [_VP, ctypes.c_size_t, ctypes.POINTER(_Params), _VP])
        lib.ccq_gdn_workspace_size.argtypes = ([_I] * 6 + [ctypes.POINTER(_Params),
                                                           ctypes.POINTER(ctypes.c_size_t)])
        lib.ccq_gdn_workspace_size.restype = _I
        lib.ccq_gdn_fwd.restype = _I
        lib.ccq_decode_step.argtypes = ([_I] + [_VP] * 6 + [_I, _I] + [_VP] * 5
                                        + [_I] * 4 + [ctypes.POINTER(_Params), _VP])
        lib.ccq_decode_step.restype = _I
        lib.ccq_gla_ckpt_size.argtypes = [_I] * 5 + [ctypes.POINTER(ctypes.c_size_t)]
        lib.ccq_gla_ckpt_size.restype = _I
        lib.ccq_gla_fwd_save.argtypes = ([_VP] * 5 + [_I, _I] + [_VP] * 9 + [_I] * 5
                                         + [_VP, ctypes.c_size_t, _VP, ctypes.c_size_t,
                                            ctypes.POINTER(_Params), _VP])
        lib.ccq_gla_fwd_save.restype = _I
        lib.ccq_gla_bwd.argtypes = ([_VP] * 5 + [_I, _I] + [_VP] * 17 + [_I] * 5
                                    + [_VP, ctypes.c_size_t, ctypes.POINTER(_Params), _VP])
        lib.ccq_gla_bwd.restype = _I
        lib.ccq_gla_bwd_workspace_size.argtypes = ([_I] * 7 + [ctypes.POINTER(_Params),
                                                               ctypes.POINTER(ctypes.c_size_t)])
        lib.ccq_gla_bwd_workspace_size.restype = _I
        # q, k, v, g, beta, lambda | in_dtype | S0, C0, m0, t0, dout, dST, dCT, dmT, dq, dk, dv,
        # dg, dbeta, dlambda, dS0, dC0, dm0 | B, T, H, Dk, Dv | workspace, bytes, params, stream
        lib.ccq_gdn_bwd.argtypes = ([_VP] * 6 + [_I] + [_VP] * 17 + [_I] * 5
                                    + [_VP, ctypes.c_size_t, ctypes.POINTER(_Params), _VP])
        lib.ccq_gdn_bwd.restype = _I
        lib.ccq_gdn_bwd_workspace_size.argtypes = ([_I] * 6 + [ctypes.POINTER(_Params),
                                                               ctypes.POINTER(ctypes.c_size_t)])
        lib.ccq_gdn_bwd_workspace_size.restype = _I
        # q, k, v, g, beta, lambda | in_dtype | S0, C0, m0, n0, o, ST, CT, mT, nT | B, T, H, Dk, Dv
        # | workspace, bytes, params, stream
        lib.ccq_gdn_fwd_decayed.argtypes = ([_VP] * 6 + [_I] + [_VP] * 9 + [_I] * 5
                                            + [_VP, ctypes.c_size_t, ctypes.POINTER(_Params), _VP])
        lib.ccq_gdn_fwd_decayed.restype = _I
        lib.ccq_gdn_fwd_spectral.argtypes = ([_VP] * 6 + [_I] + [_VP] * 9 + [_I] * 7
                                             + [_VP, ctypes.c_size_t, ctypes.POINTER(_Params), _VP])
        lib.ccq_gdn_fwd_spectral.restype = _I
        # backbone | q, k, v, gate, beta, lambda | in_dtype, gate_dtype | cu_seqlens (host), num_seqs |
        # S0, C0, m0, t0, o, ST, CT, mT, tT | H, Dk, Dv | workspace, bytes, params, stream
        lib.ccq_fwd_varlen.argtypes = ([_I] + [_VP] * 6 + [_I, _I] + [_VP, _I] + [_VP] * 9 + [_I] * 3
                                       + [_VP, ctypes.c_size_t, ctypes.POINTER(_Params), _VP])
        lib.ccq_fwd_varlen.restype = _I
        lib.ccq_fwd_varlen_workspace_size.argtypes = ([_I, _VP] + [_I] * 5 + [ctypes.POINTER(_Params),
                                                                               ctypes.POINTER(ctypes.c_size_t)])
        lib.ccq_fwd_varlen_workspace_size.restype = _I
        lib.ccq_gdn_decayed_workspace_size.argtypes = ([_I] * 6 + [ctypes.POINTER(_Params),
                                                                   ctypes.POINTER(ctypes.c_size_t)])
        lib.ccq_gdn_decayed_workspace_size.restype = _I
        _lib = lib
    return _lib


def header_symbols() -> list:
    """Names of every function include/*.h declares with CCQ_API."""
    names = []
    for f in sorted(os.listdir(_build.INCLUDE)):
        if f.endswith(".h"):
            with open(os.path.join(_build.INCLUDE, f)) as fh:
                names += re.findall(r"CCQ_API\s+[\w\s\*]*?\b(ccq_\w+)\s*\(", fh.read())
    return names


def _check(status: int):
    if status != CCQ_OK:
        lib = load_library()
        raise CCQError(status, lib.ccq_last_error().decode())


def params(*, l2norm: bool = True, scale: Optional[float] = None, centered: bool = True,
           chunk: int = 64, algo: str = "auto", seq_split: int = 0) -> _Params:
    p = _Params()
    load_library().ccq_default_params(ctypes.byref(p))
    p.l2norm_qk = int(bool(l2norm))
    p.scale = 0.0 if scale is None else float(scale)
    p.centered = int(bool(centered))
    p.chunk = int(chunk)
    p.algo = ALGO[algo]
    p.seq_split = int(seq_split)
    return p


def _ptr(x: Optional[torch.Tensor]):
    return None if x is None else ctypes.c_void_p(x.data_ptr())


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return FP32
    raise TypeError(f"unsupported dtype {t.dtype}: bf16 or fp32")


def _req(t, name, device, dtype=None, shape=None):
    if t is None:
        raise ValueError(f"{name} is required")
    if not isinstance(t, torch.Tensor) or t.device.type != "cuda":
        raise ValueError(f"{name} must be a CUDA tensor (there is no CPU path)")
    if t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t


def _stream(device, stream):
    s = stream if stream is not None else torch.cuda.current_stream(device)
    return ctypes.c_void_p(s.cuda_stream)


@dataclass
class CCQState:
    """Recurrent cache (Algorithm 2's triple plus the position): S^T [B,H,Dk,Dv],
    key second-moment SUM C [B,H,Dk,Dk], key SUM m [B,H,Dk] (fp32), t [B] int64."""
    S: torch.Tensor
    C: torch.Tensor
    m: torch.Tensor
    t: torch.Tensor

    @staticmethod
    def zeros(B, H, Dk, Dv, device):
        return CCQState(torch.zeros(B, H, Dk, Dv, device=device),
                        torch.zeros(B, H, Dk, Dk, device=device),
                        torch.zeros(B, H, Dk, device=device),
                        torch.zeros(B, dtype=torch.int64, device=device))

    @staticmethod
    def empty(B, H, Dk, Dv, device):
        return CCQState(torch.empty(B, H, Dk, Dv, device=device),
                        torch.empty(B, H, Dk, Dk, device=device),
                        torch.empty(B, H, Dk, device=device),
                        torch.empty(B, dtype=torch.int64, device=device))


def _state_in(state, B, H, Dk, Dv, device):
    if state is None:
        return None, None, None, None
    return (_req(state.S, "S0", device, torch.float32, (B, H, Dk, Dv)),
            _req(state.C, "C0", device, torch.float32, (B, H, Dk, Dk)),
            _req(state.m, "m0", device, torch.float32, (B, H, Dk)),
            _req(state.t, "t0", device, torch.int64, (B,)))


def gla_fwd(q, k, v, gk, lam, state: Optional[CCQState] = None, *, out=None,
            final_state: Optional[CCQState] = None, return_state: bool = True,
            workspace: Optional[torch.Tensor] = None, stream=None, **kw):
    """CCQ-GLA forward: o [B,T,H,Dv] and (optionally) the final CCQState.

    q, k [B,T,H,Dk], v [B,T,H,Dv] bf16 or fp32 (same dtype); gk [B,T,H,Dk]
    log-forget gate (bf16 or fp32); lam [B,T,H] fp32.  ``state`` is the initial
    cache (None = zero).  ``workspace`` (CUDA bytes, ccq_gla_workspace_size)
    is allocated on the fly when needed and not given.  Keyword arguments go to
    :func:`params`.
    """
    dev = q.device
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    _req(q, "q", dev)
    _req(k, "k", dev, q.dtype, q.shape)
    _req(v, "v", dev, q.dtype, (B, T, H, Dv))
    _req(gk, "gk", dev, None, (B, T, H, Dk))
    _req(lam, "lam", dev, torch.float32, (B, T, H))
    S0, C0, m0, t0 = _state_in(state, B, H, Dk, Dv, dev)
    o = out if out is not None else torch.empty(B, T, H, Dv, dtype=q.dtype, device=dev)
    _req(o, "out", dev, q.dtype, (B, T, H, Dv))
    fs = final_state
    if fs is None and return_state:
        fs = CCQState.empty(B, H, Dk, Dv, dev)
    p = params(**kw)
    lib = load_library()
    if workspace is None:
        need = ctypes.c_size_t(0)
        _check(lib.ccq_gla_workspace_size(B, T, H, Dk, Dv, _dtype_code(q), ctypes.byref(p),
                                          ctypes.byref(need)))
        if need.value:
            workspace = torch.empty(need.value, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.ccq_gla_fwd(
        _ptr(q), _ptr(k), _ptr(v), _ptr(gk), _ptr(lam), _dtype_code(q), _dtype_code(gk),
        _ptr(S0), _ptr(C0), _ptr(m0), _ptr(t0), _ptr(o),
        _ptr(fs.S if fs else None), _ptr(fs.C if fs else None), _ptr(fs.m if fs else None),
        _ptr(fs.t if fs else None), B, T, H, Dk, Dv, _ptr(workspace), ws_bytes,
        ctypes.byref(p), _stream(dev, stream))
    _check(st)
    return (o, fs) if return_state else o


def gla_ckpt_size(B, T, H, Dk=128, Dv=128) -> int:
    """Bytes of the checkpoint buffer :func:`gla_fwd_save` writes."""
    need = ctypes.c_size_t(0)
    _check(load_library().ccq_gla_ckpt_size(B, T, H, Dk, Dv, ctypes.byref(need)))
    return need.value


def gla_fwd_save(q, k, v, gk, lam, state: Optional[CCQState] = None, *, ckpt=None, out=None,
                 final_state: Optional[CCQState] = None, return_state: bool = True,
                 workspace: Optional[torch.Tensor] = None, stream=None, **kw):
    """:func:`gla_fwd` that also writes the chunk-start states the backward
    needs into ``ckpt`` (a CUDA uint8 tensor of :func:`gla_ckpt_size` bytes,
    allocated when not given).  Returns (o, final_state, ckpt)."""
    dev = q.device
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    _req(q, "q", dev)
    _req(k, "k", dev, q.dtype, q.shape)
    _req(v, "v", dev, q.dtype, (B, T, H, Dv))
    _req(gk, "gk", dev, None, (B, T, H, Dk))
    _req(lam, "lam", dev, torch.float32, (B, T, H))
    S0, C0, m0, t0 = _state_in(state, B, H, Dk, Dv, dev)
    o = out if out is not None else torch.empty(B, T, H, Dv, dtype=q.dtype, device=dev)
    _req(o, "out", dev, q.dtype, (B, T, H, Dv))
    fs = final_state
    if fs is None and return_state:
        fs = CCQState.empty(B, H, Dk, Dv, dev)
    if ckpt is None:
        ckpt = torch.empty(gla_ckpt_size(B, T, H, Dk, Dv), dtype=torch.uint8, device=dev)
    _req(ckpt, "ckpt", dev, torch.uint8)
    p = params(**kw)
    lib = load_library()
    if workspace is None:
        need = ctypes.c_size_t(0)
        _check(lib.ccq_gla_workspace_size(B, T, H, Dk, Dv, _dtype_code(q), ctypes.byref(p),
                                          ctypes.byref(need)))
        if need.value:
            workspace = torch.empty(need.value, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.ccq_gla_fwd_save(
        _ptr(q), _ptr(k), _ptr(v), _ptr(gk), _ptr(lam), _dtype_code(q), _dtype_code(gk),
        _ptr(S0), _ptr(C0), _ptr(m0), _ptr(t0), _ptr(o),
        _ptr(fs.S if fs else None), _ptr(fs.C if fs else None), _ptr(fs.m if fs else None),
        _ptr(fs.t if fs else None), B, T, H, Dk, Dv, _ptr(workspace), ws_bytes,
        _ptr(ckpt), ckpt.numel(), ctypes.byref(p), _stream(dev, stream))
    _check(st)
    return o, fs, ckpt


def gla_bwd_workspace(B, T, H, Dk, Dv, device, *, with_ckpt: bool, dtype=torch.bfloat16, **kw):
    """Allocate the workspace ccq_gla_bwd needs (None if none)."""
    p = params(**kw)
    need = ctypes.c_size_t(0)
    code = BF16 if dtype == torch.bfloat16 else FP32
    _check(load_library().ccq_gla_bwd_workspace_size(B, T, H, Dk, Dv, code, int(bool(with_ckpt)),
                                                      ctypes.byref(p), ctypes.byref(need)))
    return torch.empty(need.value, dtype=torch.uint8, device=device) if need.value else None


def gla_bwd(q, k, v, gk, lam, dout, state: Optional[CCQState] = None, *, dST=None, dCT=None,
            dmT=None, ckpt=None, out: Optional[dict] = None, workspace=None, stream=None, **kw):
    """CCQ-GLA backward.  Returns a dict of gradients dq, dk, dv (q's dtype),
    dgk (gk's dtype), dlambda, dS0, dC0, dm0 (fp32).  ``dST``/``dCT``/``dmT`` are
    the gradients of the final states (None = 0); ``ckpt`` the checkpoints of
    :func:`gla_fwd_save` on the same inputs (None = recompute them).  ``out``
    may hold preallocated tensors under those names."""
    dev = q.device
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    _req(q, "q", dev)
    _req(k, "k", dev, q.dtype, q.shape)
    _req(v, "v", dev, q.dtype, (B, T, H, Dv))
    _req(gk, "gk", dev, None, (B, T, H, Dk))
    _req(lam, "lam", dev, torch.float32, (B, T, H))
    _req(dout, "dout", dev, q.dtype, (B, T, H, Dv))
    S0, C0, m0, t0 = _state_in(state, B, H, Dk, Dv, dev)
    if dST is not None:
        _req(dST, "dST", dev, torch.float32, (B, H, Dk, Dv))
    if dCT is not None:
        _req(dCT, "dCT", dev, torch.float32, (B, H, Dk, Dk))
    if dmT is not None:
        _req(dmT, "dmT", dev, torch.float32, (B, H, Dk))
    if ckpt is not None:
        _req(ckpt, "ckpt", dev, torch.uint8)
    g = dict(out or {})
    shapes = {"dq": ((B, T, H, Dk), q.dtype), "dk": ((B, T, H, Dk), q.dtype),
              "dv": ((B, T, H, Dv), q.dtype), "dgk": ((B, T, H, Dk), gk.dtype),
              "dlambda": ((B, T, H), torch.float32), "dS0": ((B, H, Dk, Dv), torch.float32),
              "dC0": ((B, H, Dk, Dk), torch.float32), "dm0": ((B, H, Dk), torch.float32)}
    for name, (shape, dt) in shapes.items():
        if g.get(name) is None:
            g[name] = torch.empty(shape, dtype=dt, device=dev)
        _req(g[name], name, dev, dt, shape)
    p = params(**kw)
    lib = load_library()
    if workspace is None:
        workspace = gla_bwd_workspace(B, T, H, Dk, Dv, dev, with_ckpt=ckpt is not None,
                                      dtype=q.dtype, **kw)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.ccq_gla_bwd(
        _ptr(q), _ptr(k), _ptr(v), _ptr(gk), _ptr(lam), _dtype_code(q), _dtype_code(gk),
        _ptr(S0), _ptr(C0), _ptr(m0), _ptr(t0), _ptr(dout), _ptr(dST), _ptr(dCT), _ptr(dmT),
        _ptr(ckpt), _ptr(g["dq"]), _ptr(g["dk"]), _ptr(g["dv"]), _ptr(g["dgk"]),
        _ptr(g["dlambda"]), _ptr(g["dS0"]), _ptr(g["dC0"]), _ptr(g["dm0"]),
        B, T, H, Dk, Dv, _ptr(workspace), ws_bytes, ctypes.byref(p), _stream(dev, stream))
    _check(st)
    return g


def gdn_fwd(q, k, v, g, beta, lam, state: Optional[CCQState] = None, *, out=None,
            final_state: Optional[CCQState] = None, return_state: bool = True,
            workspace: Optional[torch.Tensor] = None, stream=None, **kw):
    """CCQ-Gated-DeltaNet forward.  g (log decay) and beta are [B,T,H] fp32.
    ``workspace`` (a CUDA byte tensor of at least ccq_gdn_workspace_size bytes)
    is allocated on the fly when not given."""
    dev = q.device
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    _req(q, "q", dev)
    _req(k, "k", dev, q.dtype, q.shape)
    _req(v, "v", dev, q.dtype, (B, T, H, Dv))
    _req(g, "g", dev, torch.float32, (B, T, H))
    _req(beta, "beta", dev, torch.float32, (B, T, H))
    _req(lam, "lam", dev, torch.float32, (B, T, H))
    S0, C0, m0, t0 = _state_in(state, B, H, Dk, Dv, dev)
    o = out if out is not None else torch.empty(B, T, H, Dv, dtype=q.dtype, device=dev)
    _req(o, "out", dev, q.dtype, (B, T, H, Dv))
    fs = final_state
    if fs is None and return_state:
        fs = CCQState.empty(B, H, Dk, Dv, dev)
    p = params(**kw)
    lib = load_library()
    need = ctypes.c_size_t(0)
    _check(lib.ccq_gdn_workspace_size(B, T, H, Dk, Dv, _dtype_code(q), ctypes.byref(p),
                                      ctypes.byref(need)))
    if workspace is None and need.value:
        workspace = torch.empty(need.value, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.ccq_gdn_fwd(
        _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(beta), _ptr(lam), _dtype_code(q),
        _ptr(S0), _ptr(C0), _ptr(m0), _ptr(t0), _ptr(o),
        _ptr(fs.S if fs else None), _ptr(fs.C if fs else None), _ptr(fs.m if fs else None),
        _ptr(fs.t if fs else None), B, T, H, Dk, Dv, _ptr(workspace), ws_bytes,
        ctypes.byref(p), _stream(dev, stream))
    _check(st)
    return (o, fs) if return_state else o


def gdn_bwd(q, k, v, g, beta, lam, dout, state: Optional[CCQState] = None, *, dST=None, dCT=None,
            dmT=None, out: Optional[dict] = None, workspace=None, stream=None, **kw):
    """CCQ-Gated-DeltaNet backward.  Returns a dict of gradients dq, dk, dv (q's dtype),
    dg, dbeta, dlambda [B,T,H] and dS0, dC0, dm0 (fp32).  ``dST``/``dCT``/``dmT`` are the
    gradients of the final states (None = 0).  ``out`` may hold preallocated tensors under
    those names; ``workspace`` (a CUDA byte tensor of at least
    ccq_gdn_bwd_workspace_size bytes) is allocated on the fly when not given."""
    dev = q.device
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    _req(q, "q", dev)
    _req(k, "k", dev, q.dtype, q.shape)
    _req(v, "v", dev, q.dtype, (B, T, H, Dv))
    _req(g, "g", dev, torch.float32, (B, T, H))
    _req(beta, "beta", dev, torch.float32, (B, T, H))
    _req(lam, "lam", dev, torch.float32, (B, T, H))
    _req(dout, "dout", dev, q.dtype, (B, T, H, Dv))
    S0, C0, m0, t0 = _state_in(state, B, H, Dk, Dv, dev)
    if dST is not None:
        _req(dST, "dST", dev, torch.float32, (B, H, Dk, Dv))
    if dCT is not None:
        _req(dCT, "dCT", dev, torch.float32, (B, H, Dk, Dk))
    if dmT is not None:
        _req(dmT, "dmT", dev, torch.float32, (B, H, Dk))
    grads = dict(out or {})
    shapes = {"dq": ((B, T, H, Dk), q.dtype), "dk": ((B, T, H, Dk), q.dtype),
              "dv": ((B, T, H, Dv), q.dtype), "dg": ((B, T, H), torch.float32),
              "dbeta": ((B, T, H), torch.float32), "dlambda": ((B, T, H), torch.float32),
              "dS0": ((B, H, Dk, Dv), torch.float32), "dC0": ((B, H, Dk, Dk), torch.float32),
              "dm0": ((B, H, Dk), torch.float32)}
    for name, (shape, dt) in shapes.items():
        if grads.get(name) is None:
            grads[name] = torch.empty(shape, dtype=dt, device=dev)
        _req(grads[name], name, dev, dt, shape)
    p = params(**kw)
    lib = load_library()
    need = ctypes.c_size_t(0)
    _check(lib.ccq_gdn_bwd_workspace_size(B, T, H, Dk, Dv, _dtype_code(q), ctypes.byref(p),
                                          ctypes.byref(need)))
    if workspace is None and need.value:
        workspace = torch.empty(need.value, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.ccq_gdn_bwd(
        _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(beta), _ptr(lam), _dtype_code(q),
        _ptr(S0), _ptr(C0), _ptr(m0), _ptr(t0), _ptr(dout), _ptr(dST), _ptr(dCT), _ptr(dmT),
        _ptr(grads["dq"]), _ptr(grads["dk"]), _ptr(grads["dv"]), _ptr(grads["dg"]),
        _ptr(grads["dbeta"]), _ptr(grads["dlambda"]), _ptr(grads["dS0"]), _ptr(grads["dC0"]),
        _ptr(grads["dm0"]), B, T, H, Dk, Dv, _ptr(workspace), ws_bytes, ctypes.byref(p),
        _stream(dev, stream))
    _check(st)
    return grads


CONTRACTION = {"linear": 0, "resolvent": 1, "exponential": 2}


def gdn_fwd_decayed(q, k, v, g, beta, lam, *, S0=None, C0=None, m0=None, n0=None, out=None,
                    return_state: bool = True, workspace=None, stream=None, contraction="linear",
                    decayed: bool = True, **kw):
    """CCQ-Gated-DeltaNet forward on the CUDA-core kernels with the decay-aligned covariance
    (statistics decayed by the backbone's own decay, normalised by the decayed count n) or,
    with ``decayed=False``, the paper's undecayed statistics (n = the token count), and the
    query contracted by ``contraction``: "linear" (the paper's I - lambda Sigma),
    "resolvent" ((I + lambda Sigma)^{-1}) or "exponential" (exp(-lambda Sigma)).
    S0 [B,H,Dk,Dv], C0 [B,H,Dk,Dk], m0 [B,H,Dk], n0 [B,H] fp32 (None = zero).  Returns o, or
    (o, dict S, C, m, n of final states) when ``return_state``."""
    dev = q.device
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    _req(q, "q", dev)
    _req(k, "k", dev, q.dtype, q.shape)
    _req(v, "v", dev, q.dtype, (B, T, H, Dv))
    for x, name in ((g, "g"), (beta, "beta"), (lam, "lam")):
        _req(x, name, dev, torch.float32, (B, T, H))
    for x, name, shape in ((S0, "S0", (B, H, Dk, Dv)), (C0, "C0", (B, H, Dk, Dk)), (m0, "m0", (B, H, Dk)),
                           (n0, "n0", (B, H))):
        if x is not None:
            _req(x, name, dev, torch.float32, shape)
    o = out if out is not None else torch.empty(B, T, H, Dv, dtype=q.dtype, device=dev)
    _req(o, "out", dev, q.dtype, (B, T, H, Dv))
    fs = None
    if return_state:
        fs = {"S": torch.empty(B, H, Dk, Dv, dtype=torch.float32, device=dev),
              "C": torch.empty(B, H, Dk, Dk, dtype=torch.float32, device=dev),
              "m": torch.empty(B, H, Dk, dtype=torch.float32, device=dev),
              "n": torch.empty(B, H, dtype=torch.float32, device=dev)}
    p = params(**kw)
    lib = load_library()
    need = ctypes.c_size_t(0)
    _check(lib.ccq_gdn_decayed_workspace_size(B, T, H, Dk, Dv, _dtype_code(q), ctypes.byref(p),
                                              ctypes.byref(need)))
    if workspace is None and need.value:
        workspace = torch.empty(need.value, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.ccq_gdn_fwd_spectral(
        _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(beta), _ptr(lam), _dtype_code(q),
        _ptr(S0), _ptr(C0), _ptr(m0), _ptr(n0), _ptr(o),
        _ptr(fs["S"] if fs else None), _ptr(fs["C"] if fs else None), _ptr(fs["m"] if fs else None),
        _ptr(fs["n"] if fs else None), B, T, H, Dk, Dv, CONTRACTION[contraction], int(bool(decayed)),
        _ptr(workspace), ws_bytes, ctypes.byref(p), _stream(dev, stream))
    _check(st)
    return (o, fs) if return_state else o


def varlen_workspace_size(backbone, cu_seqlens, H, Dk, Dv, dtype=torch.bfloat16, **kw) -> int:
    """Bytes of device workspace ccq_fwd_varlen needs for this pack (ccq_fwd_varlen_workspace_size)."""
    cu = [int(x) for x in (cu_seqlens.tolist() if hasattr(cu_seqlens, "tolist") else cu_seqlens)]
    cu_arr = (ctypes.c_int64 * len(cu))(*cu)
    p = params(**kw)
    need = ctypes.c_size_t(0)
    code = BF16 if dtype == torch.bfloat16 else FP32
    _check(load_library().ccq_fwd_varlen_workspace_size(int(backbone), ctypes.cast(cu_arr, _VP), len(cu) - 1, H,
                                                        Dk, Dv, code, ctypes.byref(p), ctypes.byref(need)))
    return need.value


def fwd_varlen(backbone, q, k, v, gate, lam, cu_seqlens, *, beta=None, state: Optional[CCQState] = None,
               out=None, final_state: Optional[CCQState] = None, return_state: bool = True, workspace=None,
               stream=None, **kw):
    """Forward of packed variable-length sequences (ccq_fwd_varlen).  q, k [total,H,Dk]; v
    [total,H,Dv]; gate [total,H,Dk] (GLA) or [total,H] fp32 (GDN, with beta [total,H]); lam
    [total,H]; ``cu_seqlens`` the num_seqs + 1 offsets (a list or CPU integer tensor; it stays on
    the host).  ``state`` / the returned CCQState hold one row per sequence.  Returns o
    [total,H,Dv] and (optionally) the final CCQState."""
    dev = q.device
    total, H, Dk = q.shape
    Dv = v.shape[-1]
    cu = [int(x) for x in (cu_seqlens.tolist() if hasattr(cu_seqlens, "tolist") else cu_seqlens)]
    ns = len(cu) - 1
    # The C ABI cannot see the packed length: an offset past it would make the kernels read
    # and write beyond the tensors, so the pack is checked here.
    if ns < 1 or cu[0] != 0:
        raise ValueError("cu_seqlens must start at 0 and hold num_seqs + 1 >= 2 offsets")
    if any(b < a for a, b in zip(cu, cu[1:])):
        raise ValueError("cu_seqlens must be non-decreasing")
    if cu[-1] != total:
        raise ValueError(f"cu_seqlens[-1] = {cu[-1]} must equal the packed length {total}")
    _req(q, "q", dev)
    _req(k, "k", dev, q.dtype, q.shape)
    _req(v, "v", dev, q.dtype, (total, H, Dv))
    _req(gate, "gate", dev, None, (total, H, Dk) if backbone == 0 else (total, H))
    _req(lam, "lam", dev, torch.float32, (total, H))
    if beta is not None:
        _req(beta, "beta", dev, torch.float32, (total, H))
    S0, C0, m0, t0 = _state_in(state, ns, H, Dk, Dv, dev)
    o = out if out is not None else torch.empty(total, H, Dv, dtype=q.dtype, device=dev)
    _req(o, "out", dev, q.dtype, (total, H, Dv))
    fs = (final_state or CCQState.empty(ns, H, Dk, Dv, dev)) if return_state else None
    if fs is not None:
        _state_in(fs, ns, H, Dk, Dv, dev)
    cu_arr = (ctypes.c_int64 * len(cu))(*cu)
    p = params(**kw)
    lib = load_library()
    need = ctypes.c_size_t(0)
    _check(lib.ccq_fwd_varlen_workspace_size(int(backbone), ctypes.cast(cu_arr, _VP), ns, H, Dk, Dv,
                                             _dtype_code(q), ctypes.byref(p), ctypes.byref(need)))
    if workspace is None and need.value:
        workspace = torch.empty(need.value, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.ccq_fwd_varlen(
        int(backbone), _ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(beta), _ptr(lam), _dtype_code(q),
        _dtype_code(gate), ctypes.cast(cu_arr, _VP), ns, _ptr(S0), _ptr(C0), _ptr(m0), _ptr(t0), _ptr(o),
        _ptr(fs.S if fs else None), _ptr(fs.C if fs else None), _ptr(fs.m if fs else None),
        _ptr(fs.t if fs else None), H, Dk, Dv, _ptr(workspace), ws_bytes, ctypes.byref(p), _stream(dev, stream))
    _check(st)
    return (o, fs) if return_state else o


def gla_workspace(B, T, H, Dk, Dv, device, dtype=torch.bfloat16, **kw):
    """Allocate the workspace ccq_gla_fwd needs for these sizes (None if none)."""
    p = params(**kw)
    need = ctypes.c_size_t(0)
    code = BF16 if dtype == torch.bfloat16 else FP32
    _check(load_library().ccq_gla_workspace_size(B, T, H, Dk, Dv, code, ctypes.byref(p),
                                                  ctypes.byref(need)))
    return torch.empty(need.value, dtype=torch.uint8, device=device) if need.value else None


def gdn_workspace(B, T, H, Dk, Dv, device, dtype=torch.bfloat16, **kw):
    """Allocate the workspace ccq_gdn_fwd needs for these sizes (None if none)."""
    p = params(**kw)
    need = ctypes.c_size_t(0)
    code = BF16 if dtype == torch.bfloat16 else FP32
    _check(load_library().ccq_gdn_workspace_size(B, T, H, Dk, Dv, code, ctypes.byref(p),
                                                  ctypes.byref(need)))
    return torch.empty(need.value, dtype=torch.uint8, device=device) if need.value else None


def gdn_bwd_workspace(B, T, H, Dk, Dv, device, dtype=torch.bfloat16, **kw):
    """Allocate the workspace ccq_gdn_bwd needs for these sizes (None if none)."""
    p = params(**kw)
    need = ctypes.c_size_t(0)
    code = BF16 if dtype == torch.bfloat16 else FP32
    _check(load_library().ccq_gdn_bwd_workspace_size(B, T, H, Dk, Dv, code, ctypes.byref(p),
                                                      ctypes.byref(need)))
    return torch.empty(need.value, dtype=torch.uint8, device=device) if need.value else None


def decode_step(backbone: int, q, k, v, gate, lam, state: CCQState, beta=None, *,
                out=None, stream=None, **kw):
    """One recurrent token (Algorithm 2): q, k [B,H,Dk], v [B,H,Dv]; gate
    [B,H,Dk] (GLA, bf16/fp32) or [B,H] fp32 (GDN); lam (and beta) [B,H] fp32.
    Updates ``state`` in place and returns o [B,H,Dv]."""
    dev = q.device
    B, H, Dk = q.shape
    Dv = v.shape[-1]
    _req(q, "q", dev)
    _req(k, "k", dev, q.dtype, q.shape)
    _req(v, "v", dev, q.dtype, (B, H, Dv))
    _req(gate, "gate", dev, None, (B, H, Dk) if backbone == GLA else (B, H))
    _req(lam, "lam", dev, torch.float32, (B, H))
    if backbone == GDN:
        _req(beta, "beta", dev, torch.float32, (B, H))
    S, C, m, t = _state_in(state, B, H, Dk, Dv, dev)
    o = out if out is not None else torch.empty(B, H, Dv, dtype=q.dtype, device=dev)
    _req(o, "out", dev, q.dtype, (B, H, Dv))
    p = params(**kw)
    st = load_library().ccq_decode_step(
        int(backbone), _ptr(q), _ptr(k), _ptr(v), _ptr(gate), _ptr(beta), _ptr(lam),
        _dtype_code(q), _dtype_code(gate), _ptr(S), _ptr(C), _ptr(m), _ptr(t), _ptr(o),
        B, H, Dk, Dv, ctypes.byref(p), _stream(dev, stream))
    _check(st)
    return o


def device_status(stream=None, device=None):
    """Synchronise and read/clear the kernels' status word; raises on a timeout."""
    dev = device or torch.device("cuda", torch.cuda.current_device())
    _check(load_library().ccq_device_status(_stream(dev, stream)))
