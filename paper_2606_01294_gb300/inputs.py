"""Seeded synthetic inputs shaped like the paper's CCQ workloads.

This module only draws random tensors; it holds none of the CCQ arithmetic.
Both the GPU tests / benchmark and the CPU oracle consume what it returns.

Recipe (all draws fp32 from a CPU ``torch.Generator`` seeded with ``seed``, in
the order q, k, v, gate, beta, lambda, then cast to the requested dtype):
  q, k, v        ~ N(0, 1), layout [B, T, H, D] with D contiguous;
                   k (and for Gated DeltaNet also q) l2-normalised per head row
                   before the cast, as the workload description specifies.
  GLA gate       log-forget per key dim: logsigmoid(N(0,1)) / 16, [B,T,H,Dk].
  GDN gate       log decay per token/head: -softplus(N(0,1)) (alpha =
                 exp(-softplus)), [B,T,H] fp32; beta = sigmoid(N(0,1)) fp32.
  lambda         [B,T,H] fp32 in (0, 1):
                   "init"     0.01 everywhere (W_lambda = 0, sigma(b) = 0.01, App. D);
                   "trained"  sigmoid(N(logit(0.29), 0.5)) (App. E gate statistics);
                   "high"     0.9 (App. A.3: stable as lambda approaches 1);
                   a float    that constant.
  keys           "iso" (above) or "structured": k = normalise(m0 + U z + 0.25 eps),
                 U a fixed random orthonormal d x 16 basis, z ~ N(0, I_16),
                 eps ~ N(0, I_d), m0 a fixed random vector of norm 0.5 -- a
                 low-rank key spread with a non-zero mean, so Sigma_t is large and
                 the mean term matters; or "lowrank": k = normalise(U z + 0.1 eps)
                 with a fixed orthonormal d x 2 basis U, so Sigma_t has two
                 eigenvalues near 1/2 and the CCQ correction is large; or "rank2": the
                 same with 0.01 eps, so that the keys lie almost in the subspace.
  queries        "iso" (above) or "lowrank": q = U z + 0.01 eps in the same d x 2
                 subspace as the low-rank keys (drawn after lambda, so the other
                 draws are unchanged); with "rank2" keys and lambda near 1 the CCQ
                 term is more than half of o.
  gates          "default" (above); "strong": GLA logsigmoid(N(0,1)) without the
                 1/16, GDN -8 softplus(N(0,1)) (about -6 per token, as strongly
                 forgetting trained heads); or a float c: every GLA log-gate entry,
                 or every GDN log decay, equal to c (c <= 0).  The normal draw of the
                 default gate is made in every case, so the other draws are unchanged.
"""
from __future__ import annotations

import math

import torch
import torch.nn.functional as F

GLA = 0
GDN = 1


def _normalise_rows(x: torch.Tensor) -> torch.Tensor:
    return x / x.norm(dim=-1, keepdim=True).clamp_min(1e-30)


def _structured_keys(gen, B, T, H, Dk, rank=16):
    basis_gen = torch.Generator().manual_seed(7919)
    U, _ = torch.linalg.qr(torch.randn(Dk, min(rank, Dk), generator=basis_gen))
    m0 = torch.randn(Dk, generator=basis_gen)
    m0 = 0.5 * m0 / m0.norm()
    z = torch.randn(B, T, H, U.shape[1], generator=gen)
    eps = torch.randn(B, T, H, Dk, generator=gen)
    return m0 + z @ U.T + 0.25 * eps


def _lowrank_keys(gen, B, T, H, Dk, rank=2, noise=0.1):
    basis_gen = torch.Generator().manual_seed(104729)
    U, _ = torch.linalg.qr(torch.randn(Dk, rank, generator=basis_gen))
    z = torch.randn(B, T, H, rank, generator=gen)
    eps = torch.randn(B, T, H, Dk, generator=gen)
    return z @ U.T + noise * eps


def _lambda(gen, B, T, H, lam):
    if isinstance(lam, (int, float)):
        return torch.full((B, T, H), float(lam))
    if lam == "init":
        return torch.full((B, T, H), 0.01)
    if lam == "trained":
        logit = math.log(0.29 / 0.71)
        return torch.sigmoid(logit + 0.5 * torch.randn(B, T, H, generator=gen))
    if lam == "high":
        return torch.full((B, T, H), 0.9)
    raise ValueError(f"unknown lambda regime {lam!r}")


def make_inputs(backbone: int, B: int, T: int, H: int, Dk: int, Dv: int, *,
                dtype=torch.bfloat16, gate_dtype=None, seed: int = 1234,
                lam="init", keys: str = "iso", queries: str = "iso", gates="default") -> dict:
    """Draw one CCQ forward problem on the CPU.

    Returns a dict of CPU tensors: q, k [B,T,H,Dk] and v [B,T,H,Dv] in
    ``dtype``; ``gate`` ([B,T,H,Dk] in ``gate_dtype`` (default ``dtype``) for
    GLA, [B,T,H] fp32 for GDN); ``beta`` ([B,T,H] fp32, GDN only, else None);
    ``lam`` [B,T,H] fp32.
    """
    gen = torch.Generator().manual_seed(seed)
    q = torch.randn(B, T, H, Dk, generator=gen)
    if keys == "iso":
        k = torch.randn(B, T, H, Dk, generator=gen)
    elif keys == "structured":
        k = _structured_keys(gen, B, T, H, Dk)
    elif keys == "lowrank":
        k = _lowrank_keys(gen, B, T, H, Dk)
    elif keys == "rank2":
        k = _lowrank_keys(gen, B, T, H, Dk, noise=0.01)
    else:
        raise ValueError(f"unknown key distribution {keys!r}")
    k = _normalise_rows(k)
    if backbone == GDN:
        q = _normalise_rows(q)
    v = torch.randn(B, T, H, Dv, generator=gen)
    if backbone == GLA:
        z = torch.randn(B, T, H, Dk, generator=gen)
        if gates == "default":
            gate = F.logsigmoid(z) / 16
        elif gates == "strong":
            gate = F.logsigmoid(z)
        elif isinstance(gates, (int, float)) and gates <= 0:
            gate = torch.full_like(z, float(gates))
        else:
            raise ValueError(f"unknown gate distribution {gates!r}")
        gate = gate.to(gate_dtype or dtype)
        beta = None
    else:
        z = torch.randn(B, T, H, generator=gen)
        if gates == "default":
            gate = -F.softplus(z)
        elif gates == "strong":
            gate = -8.0 * F.softplus(z)
        elif isinstance(gates, (int, float)) and gates <= 0:
            gate = torch.full_like(z, float(gates))
        else:
            raise ValueError(f"unknown gate distribution {gates!r}")
        beta = torch.sigmoid(torch.randn(B, T, H, generator=gen))
    lam_t = _lambda(gen, B, T, H, lam)
    if queries == "lowrank":
        basis_gen = torch.Generator().manual_seed(104729)
        U, _ = torch.linalg.qr(torch.randn(Dk, 2, generator=basis_gen))
        q = torch.randn(B, T, H, 2, generator=gen) @ U.T + 0.01 * torch.randn(B, T, H, Dk, generator=gen)
        if backbone == GDN:
            q = _normalise_rows(q)
    elif queries != "iso":
        raise ValueError(f"unknown query distribution {queries!r}")
    return {"q": q.to(dtype), "k": k.to(dtype), "v": v.to(dtype), "gate": gate,
            "beta": beta, "lam": lam_t.float()}


def make_decode_inputs(backbone: int, B: int, H: int, Dk: int, Dv: int, *,
                       dtype=torch.bfloat16, seed: int = 4321, lam="init",
                       prefix: int = 64) -> dict:
    """Draw a decode problem: a ``prefix``-token history (a [B,prefix,H,*]
    forward problem whose final states seed the decode state) plus one new
    token per (batch, head) with the same value distributions."""
    hist = make_inputs(backbone, B, prefix + 1, H, Dk, Dv, dtype=dtype,
                       seed=seed, lam=lam)
    pre = {n: (None if x is None else x[:, :prefix].contiguous())
           for n, x in hist.items()}
    tok = {n: (None if x is None else x[:, prefix].contiguous())
           for n, x in hist.items()}
    return {"prefix": pre, "token": tok}


def make_backward_inputs(B: int, T: int, H: int, Dk: int, Dv: int, *, dtype=torch.bfloat16,
                         seed: int = 5678, prefix: int = 0, state_grads: bool = True) -> dict:
    """Draw the extra inputs of a backward problem on the CPU: the output
    gradient ``dout`` [B,T,H,Dv] (N(0,1) in ``dtype``); final-state gradients
    ``dST`` [B,H,Dk,Dv], ``dCT`` [B,H,Dk,Dk], ``dmT`` [B,H,Dk] (fp32, N(0,1)
    scaled by 1/Dk so that each weighs about as much as the output's; None
    unless ``state_grads``); and, when ``prefix`` > 0, a consistent initial
    state from a ``prefix``-token history of unit keys (S0 ~ N(0,1)/sqrt(Dk),
    C0 = sum k k^T, m0 = sum k, t0 = prefix), else None."""
    gen = torch.Generator().manual_seed(seed)
    out = {"dout": torch.randn(B, T, H, Dv, generator=gen).to(dtype),
           "dST": None, "dCT": None, "dmT": None, "state": None}
    if state_grads:
        out["dST"] = torch.randn(B, H, Dk, Dv, generator=gen) / Dk
        out["dCT"] = torch.randn(B, H, Dk, Dk, generator=gen) / Dk
        out["dmT"] = torch.randn(B, H, Dk, generator=gen) / Dk
    if prefix > 0:
        kp = _normalise_rows(torch.randn(B, prefix, H, Dk, generator=gen)).double()
        out["state"] = {"S": torch.randn(B, H, Dk, Dv, generator=gen).double() / Dk ** 0.5,
                        "C": torch.einsum("bthd,bthe->bhde", kp, kp),
                        "m": kp.sum(dim=1),
                        "t": torch.full((B,), prefix, dtype=torch.int64)}
    return out


# The workload shapes (name -> keyword arguments), one per benchmark line
# or parity case.  "chunk" is the chunk length of the chunkwise kernels.
WORKLOADS = {
    "gla_fp32_small": dict(backbone=GLA, B=1, H=2, T=256, Dk=64, Dv=64,
                           dtype=torch.float32, seed=1235),
    "gla_bf16_4k": dict(backbone=GLA, B=8, H=16, T=4096, Dk=128, Dv=128,
                        dtype=torch.bfloat16, seed=1236),
    "gdn_bf16_4k": dict(backbone=GDN, B=8, H=16, T=4096, Dk=128, Dv=128,
                        dtype=torch.bfloat16, seed=1237),
    "gla_bf16_20k": dict(backbone=GLA, B=1, H=16, T=20480, Dk=128, Dv=128,
                         dtype=torch.bfloat16, seed=1238),
    "gdn_bf16_20k": dict(backbone=GDN, B=1, H=16, T=20480, Dk=128, Dv=128,
                         dtype=torch.bfloat16, seed=1238),
    "gla_bf16_4k_fwdbwd": dict(backbone=GLA, B=4, H=16, T=4096, Dk=128, Dv=128,
                               dtype=torch.bfloat16, seed=1239),
}
