"""ctypes marshalling for the fp64 C oracle (test infrastructure only).

Compiles ``ccq_oracle.c`` with gcc into ``_ccq_oracle.so`` beside it the first
time it is needed (or when the source is newer), then calls
``ccq_oracle_forward``.  All arrays are converted to contiguous float64 (or
int64 for positions); inputs that were rounded to bf16/fp32 are passed as
their exactly upcast values.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

GLA = 0
GDN = 1

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ccq_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_ccq_oracle.so")
_lib = None
_lock = threading.Lock()


def build_oracle(force: bool = False) -> str:
    """Compile the oracle shared library with gcc; return its path."""
    stale = (not os.path.exists(_LIB_PATH)) or (
        os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC))
    if force or stale:
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread", _SRC,
             "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def load_library(path: str):
    """Open a compiled oracle library at ``path`` and declare its signature."""
    lib = ctypes.CDLL(path)
    dp = ctypes.POINTER(ctypes.c_double)
    ip = ctypes.POINTER(ctypes.c_int64)
    lib.ccq_oracle_forward.argtypes = (
        [ctypes.c_int] * 6 + [dp] * 9 + [ip] + [dp] * 4 + [ip] + [dp]
        + [ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_int,
           ctypes.c_int])
    lib.ccq_oracle_forward.restype = ctypes.c_int
    lib.ccq_oracle_gla_backward.argtypes = (
        [ctypes.c_int] * 5 + [dp] * 8 + [ip] + [dp] * 4 + [dp] * 8
        + [ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_int])
    lib.ccq_oracle_gla_backward.restype = ctypes.c_int
    lib.ccq_oracle_gdn_backward.argtypes = (
        [ctypes.c_int] * 5 + [dp] * 9 + [ip] + [dp] * 4 + [dp] * 9
        + [ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_int])
    lib.ccq_oracle_gdn_backward.restype = ctypes.c_int
    lib.ccq_oracle_gdn_forward_decayed.argtypes = (
        [ctypes.c_int] * 5 + [dp] * 10 + [dp] * 6
        + [ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_int])
    lib.ccq_oracle_gdn_forward_decayed.restype = ctypes.c_int
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = load_library(build_oracle())
    return _lib


def _f64(x):
    if x is None:
        return None
    if hasattr(x, "detach"):  # torch tensor
        x = x.detach().to("cpu").double().numpy()
    return np.ascontiguousarray(x, dtype=np.float64)


def _i64(x):
    if x is None:
        return None
    if hasattr(x, "detach"):
        x = x.detach().to("cpu").numpy()
    return np.ascontiguousarray(x, dtype=np.int64)


def _ptr(a, kind=ctypes.c_double):
    if a is None:
        return None
    return a.ctypes.data_as(ctypes.POINTER(kind))


def forward(backbone, q, k, v, gate, lam, beta=None, S0=None, C0=None, m0=None,
            t0=None, *, l2norm=True, centered=True, scale=None, chunk=0,
            nthreads=None, want_qclean=False, lib=None):
    """Oracle CCQ forward.

    Shapes: q, k [B,T,H,Dk]; v [B,T,H,Dv]; gate [B,T,H,Dk] (GLA log-forget)
    or [B,T,H] (GDN log-decay); beta [B,T,H] (GDN); lam [B,T,H];
    S0 [B,H,Dk,Dv] (the transpose of the paper's d_v x d_k state);
    C0 [B,H,Dk,Dk]; m0 [B,H,Dk]; t0 [B].
    Returns dict with o [B,T,H,Dv], S [B,H,Dk,Dv], C [B,H,Dk,Dk], m [B,H,Dk],
    t [B] and (optionally) qclean [B,T,H,Dk]; all float64 / int64.
    """
    lib = lib or _load()
    q, k, v, gate, lam = map(_f64, (q, k, v, gate, lam))
    beta, S0, C0, m0 = map(_f64, (beta, S0, C0, m0))
    t0 = _i64(t0)
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    if scale is None:
        scale = Dk ** -0.5
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    o = np.zeros((B, T, H, Dv))
    S = np.zeros((B, H, Dk, Dv))
    C = np.zeros((B, H, Dk, Dk))
    m = np.zeros((B, H, Dk))
    t = np.zeros((B,), dtype=np.int64)
    qc = np.zeros((B, T, H, Dk)) if want_qclean else None
    rc = lib.ccq_oracle_forward(
        int(backbone), B, T, H, Dk, Dv, _ptr(q), _ptr(k), _ptr(v), _ptr(gate),
        _ptr(beta), _ptr(lam), _ptr(S0), _ptr(C0), _ptr(m0),
        _ptr(t0, ctypes.c_int64), _ptr(o), _ptr(S), _ptr(C), _ptr(m),
        _ptr(t, ctypes.c_int64), _ptr(qc), int(bool(l2norm)),
        int(bool(centered)), float(scale), int(chunk), int(nthreads))
    if rc != 0:
        raise ValueError("ccq_oracle_forward rejected its arguments")
    out = {"o": o, "S": S, "C": C, "m": m, "t": t}
    if want_qclean:
        out["qclean"] = qc
    return out


def decode_step(backbone, q, k, v, gate, lam, S, C, m, t, beta=None, *,
                l2norm=True, centered=True, scale=None, nthreads=None):
    """One recurrent token (Algorithm 2) for a batch of states.

    q, k [B,H,Dk]; v [B,H,Dv]; gate [B,H,Dk] (GLA) or [B,H] (GDN); lam, beta
    [B,H]; S [B,H,Dk,Dv]; C [B,H,Dk,Dk]; m [B,H,Dk]; t [B].
    Returns o [B,H,Dv] and the updated (S, C, m, t).
    """
    q, k, v, gate, lam, beta = map(_f64, (q, k, v, gate, lam, beta))
    add_t = lambda a: None if a is None else a[:, None]  # noqa: E731
    res = forward(backbone, add_t(q), add_t(k), add_t(v), add_t(gate),
                  add_t(lam), beta=add_t(beta), S0=S, C0=C, m0=m, t0=t,
                  l2norm=l2norm, centered=centered, scale=scale,
                  nthreads=nthreads)
    return {"o": res["o"][:, 0], "S": res["S"], "C": res["C"], "m": res["m"],
            "t": res["t"]}


def gla_backward(q, k, v, gk, lam, dout, S0=None, C0=None, m0=None, t0=None, dST=None,
                 dCT=None, dmT=None, *, l2norm=True, centered=True, scale=None,
                 nthreads=None, lib=None):
    """Reverse mode of the CCQ-GLA forward: gradients of sum(dout * o)
    + sum(dST * S_T) + sum(dCT * C_T) + sum(dmT * m_T) with respect to
    q, k, v, gk, lam, S0, C0, m0 (shapes as in :func:`forward`)."""
    lib = lib or _load()
    q, k, v, gk, lam, dout = map(_f64, (q, k, v, gk, lam, dout))
    S0, C0, m0, dST, dCT, dmT = map(_f64, (S0, C0, m0, dST, dCT, dmT))
    t0 = _i64(t0)
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    if scale is None:
        scale = Dk ** -0.5
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    g = {"dq": np.zeros_like(q), "dk": np.zeros_like(k), "dv": np.zeros_like(v),
         "dgk": np.zeros_like(gk), "dlam": np.zeros_like(lam),
         "dS0": np.zeros((B, H, Dk, Dv)), "dC0": np.zeros((B, H, Dk, Dk)),
         "dm0": np.zeros((B, H, Dk))}
    rc = lib.ccq_oracle_gla_backward(
        B, T, H, Dk, Dv, _ptr(q), _ptr(k), _ptr(v), _ptr(gk), _ptr(lam), _ptr(S0), _ptr(C0),
        _ptr(m0), _ptr(t0, ctypes.c_int64), _ptr(dout), _ptr(dST), _ptr(dCT), _ptr(dmT),
        _ptr(g["dq"]), _ptr(g["dk"]), _ptr(g["dv"]), _ptr(g["dgk"]), _ptr(g["dlam"]),
        _ptr(g["dS0"]), _ptr(g["dC0"]), _ptr(g["dm0"]), int(bool(l2norm)), int(bool(centered)),
        float(scale), int(nthreads))
    if rc != 0:
        raise ValueError("ccq_oracle_gla_backward rejected its arguments")
    return g


def gdn_backward(q, k, v, g, beta, lam, dout, S0=None, C0=None, m0=None, t0=None, dST=None,
                 dCT=None, dmT=None, *, l2norm=True, centered=True, scale=None,
                 nthreads=None, lib=None):
    """Reverse mode of the CCQ-Gated-DeltaNet forward: gradients of sum(dout * o)
    + sum(dST * S_T) + sum(dCT * C_T) + sum(dmT * m_T) with respect to
    q, k, v, g (the log decay), beta, lam, S0, C0, m0 (shapes as in :func:`forward`)."""
    lib = lib or _load()
    q, k, v, g, beta, lam, dout = map(_f64, (q, k, v, g, beta, lam, dout))
    S0, C0, m0, dST, dCT, dmT = map(_f64, (S0, C0, m0, dST, dCT, dmT))
    t0 = _i64(t0)
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    if scale is None:
        scale = Dk ** -0.5
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    r = {"dq": np.zeros_like(q), "dk": np.zeros_like(k), "dv": np.zeros_like(v),
         "dg": np.zeros_like(g), "dbeta": np.zeros_like(beta), "dlam": np.zeros_like(lam),
         "dS0": np.zeros((B, H, Dk, Dv)), "dC0": np.zeros((B, H, Dk, Dk)),
         "dm0": np.zeros((B, H, Dk))}
    rc = lib.ccq_oracle_gdn_backward(
        B, T, H, Dk, Dv, _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(beta), _ptr(lam), _ptr(S0),
        _ptr(C0), _ptr(m0), _ptr(t0, ctypes.c_int64), _ptr(dout), _ptr(dST), _ptr(dCT), _ptr(dmT),
        _ptr(r["dq"]), _ptr(r["dk"]), _ptr(r["dv"]), _ptr(r["dg"]), _ptr(r["dbeta"]), _ptr(r["dlam"]),
        _ptr(r["dS0"]), _ptr(r["dC0"]), _ptr(r["dm0"]), int(bool(l2norm)), int(bool(centered)),
        float(scale), int(nthreads))
    if rc != 0:
        raise ValueError("ccq_oracle_gdn_backward rejected its arguments")
    return r


def gdn_forward_decayed(q, k, v, g, beta, lam, S0=None, C0=None, m0=None, n0=None, *, l2norm=True,
                        centered=True, scale=None, want_qclean=False, nthreads=None, lib=None):
    """CCQ-Gated-DeltaNet forward with the decay-aligned covariance: the running statistics
    decay with the backbone's own scalar decay and are normalised by the decayed count n
    (the reading stated in ccq_oracle.c).  q, k [B,T,H,Dk]; v [B,T,H,Dv]; g, beta, lam
    [B,T,H]; S0 [B,H,Dk,Dv], C0 [B,H,Dk,Dk], m0 [B,H,Dk], n0 [B,H] (None = zero).
    Returns dict o, S, C, m, n (and qclean when asked)."""
    lib = lib or _load()
    q, k, v, g, beta, lam = map(_f64, (q, k, v, g, beta, lam))
    S0, C0, m0, n0 = map(_f64, (S0, C0, m0, n0))
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    if scale is None:
        scale = Dk ** -0.5
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    out = {"o": np.zeros((B, T, H, Dv)), "S": np.zeros((B, H, Dk, Dv)), "C": np.zeros((B, H, Dk, Dk)),
           "m": np.zeros((B, H, Dk)), "n": np.zeros((B, H))}
    qc = np.zeros((B, T, H, Dk)) if want_qclean else None
    rc = lib.ccq_oracle_gdn_forward_decayed(
        B, T, H, Dk, Dv, _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(beta), _ptr(lam), _ptr(S0),
        _ptr(C0), _ptr(m0), _ptr(n0), _ptr(out["o"]), _ptr(out["S"]), _ptr(out["C"]), _ptr(out["m"]),
        _ptr(out["n"]), _ptr(qc), int(bool(l2norm)), int(bool(centered)), float(scale), int(nthreads))
    if rc != 0:
        raise ValueError("ccq_oracle_gdn_forward_decayed rejected its arguments")
    if want_qclean:
        out["qclean"] = qc
    return out


# Spectral contractions of the CCQ read (Sec. 3.2, after Eq. clean): the paper's operator
# I - lambda Sigma is the first-order form of (I + lambda Sigma)^{-1} and exp(-lambda Sigma).
LINEAR, RESOLVENT, EXPONENTIAL = 0, 1, 2


def gdn_forward_spectral(q, k, v, g, beta, lam, *, contraction=LINEAR, decayed=False, S0=None, C0=None,
                         m0=None, n0=None, l2norm=True, centered=True, scale=None, want_qclean=False):
    """CCQ-Gated-DeltaNet forward with the query contracted by f(lambda_t Sigma_t), f one of
    the spectral contractions I - x (the paper's), (I + x)^{-1} or exp(-x) that the paper names
    as alternatives with the same first-order form.  Plain numpy, token by token, in fp64:

      statistics (Sec. 3.2): C += kbar kbar^T, m += kbar, n += 1 -- or, with ``decayed``, the
        decay-aligned reading (C, m, n first multiplied by the token's alpha);
      Sigma = C/n - c (m/n)(m/n)^T  (c = 1 centred, 0 uncentred);
      q_clean = qbar - lambda Sigma qbar | solve((I + lambda Sigma), qbar) | expm(-lambda Sigma) qbar;
      S = alpha S (I - beta kbar kbar^T) + beta v kbar^T (the Gated DeltaNet write, stored as
        H = S^T);  o = scale S q_clean.

    q, k [B,T,H,Dk]; v [B,T,H,Dv]; g, beta, lam [B,T,H]; S0 [B,H,Dk,Dv]; C0 [B,H,Dk,Dk];
    m0 [B,H,Dk]; n0 [B,H] (the count entering, t0 for the undecayed statistics).  Returns
    dict o, S, C, m, n (and qclean [B,T,H,Dk] when asked)."""
    import scipy.linalg

    q, k, v, g, beta, lam = map(_f64, (q, k, v, g, beta, lam))
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    scale = Dk ** -0.5 if scale is None else scale
    c = 1.0 if centered else 0.0
    out = {"o": np.zeros((B, T, H, Dv)), "S": np.zeros((B, H, Dk, Dv)), "C": np.zeros((B, H, Dk, Dk)),
           "m": np.zeros((B, H, Dk)), "n": np.zeros((B, H))}
    if want_qclean:
        out["qclean"] = np.zeros((B, T, H, Dk))

    def unit(x):
        nrm = np.linalg.norm(x)
        return x / nrm if (l2norm and nrm > 0) else (x.copy() if not l2norm else np.zeros_like(x))

    for b in range(B):
        for h in range(H):
            Hs = np.zeros((Dk, Dv)) if S0 is None else _f64(S0)[b, h].copy()
            C = np.zeros((Dk, Dk)) if C0 is None else _f64(C0)[b, h].copy()
            m = np.zeros(Dk) if m0 is None else _f64(m0)[b, h].copy()
            n = 0.0 if n0 is None else float(_f64(n0)[b, h])
            for t in range(T):
                qb, kb = unit(q[b, t, h]), unit(k[b, t, h])
                a = np.exp(g[b, t, h])
                if decayed:
                    C, m, n = a * C, a * m, a * n
                C = C + np.outer(kb, kb)
                m = m + kb
                n = n + 1.0
                Sig = C / n - c * np.outer(m / n, m / n)
                x = lam[b, t, h] * Sig
                if contraction == LINEAR:
                    qc = qb - x @ qb
                elif contraction == RESOLVENT:
                    qc = np.linalg.solve(np.eye(Dk) + x, qb)
                elif contraction == EXPONENTIAL:
                    qc = scipy.linalg.expm(-x) @ qb
                else:
                    raise ValueError("unknown contraction")
                if want_qclean:
                    out["qclean"][b, t, h] = qc
                u = beta[b, t, h] * (v[b, t, h] - a * (kb @ Hs))
                Hs = a * Hs + np.outer(kb, u)
                out["o"][b, t, h] = scale * (qc @ Hs)
            out["S"][b, h], out["C"][b, h], out["m"][b, h], out["n"][b, h] = Hs, C, m, n
    return out
