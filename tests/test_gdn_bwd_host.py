"""CPU check of the CCQ-Gated-DeltaNet backward kernels' arithmetic and indexing.

The kernels (paper_2606_01294_gb300/csrc/ccq_gdn_bwd_kernels.cuh) are compiled for the host
by tests/host_emu/gdn_cuda_core_emu.cpp (the gdn_emu fixture), which runs every CTA with one
thread, phase by phase (the kernels are written so that this computes what the CTA
computes), each CTA with exactly its dynamic shared memory filled with NaN.  Their gradients are compared with the oracle's fp64
reverse mode on the same inputs: fp32 inputs to 1e-4 (the fp32 bar; observed about 2e-6),
bf16 inputs to 2e-2.  This checks the algebra of the chunked adjoint, the chunk and tail
indexing and the workspace layout without a GPU; the GPU parity test checks the same
entry point through the C ABI on the device."""
import ctypes

import numpy as np
import pytest

import oracle


def bf16_round(a):
    """Round fp32 values to bf16 (nearest even) and back, as the kernels' bf16 inputs hold them."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return u.astype(np.uint32).view(np.float32)


def problem(D, B, T, H, seed, *, bf16=False, lam=None, states=True, t0v=7):
    rng = np.random.default_rng(seed)
    f32 = lambda a: np.ascontiguousarray(a, dtype=np.float32)  # noqa: E731
    P = {n: f32(rng.standard_normal((B, T, H, D))) for n in ("q", "k", "v", "dout")}
    if bf16:
        P = {n: bf16_round(x) for n, x in P.items()}
    P["g"] = f32(-np.log1p(np.exp(rng.standard_normal((B, T, H)))))
    P["beta"] = f32(1 / (1 + np.exp(-rng.standard_normal((B, T, H)))))
    P["lam"] = f32(np.full((B, T, H), lam) if lam is not None else
                   1 / (1 + np.exp(-(np.log(0.29 / 0.71) + 0.5 * rng.standard_normal((B, T, H))))))
    if states:
        hist = rng.standard_normal((B, H, t0v, D))
        hist /= np.linalg.norm(hist, axis=-1, keepdims=True)
        P.update(S0=f32(rng.standard_normal((B, H, D, D)) / D), C0=f32(np.einsum("bhti,bhtj->bhij", hist, hist)),
                 m0=f32(hist.sum(2)), t0=np.full((B,), t0v, dtype=np.int64),
                 dST=f32(rng.standard_normal((B, H, D, D)) / D), dCT=f32(rng.standard_normal((B, H, D, D)) / D),
                 dmT=f32(rng.standard_normal((B, H, D)) / D))
    else:
        P.update(S0=None, C0=None, m0=None, t0=None, dST=None, dCT=None, dmT=None)
    return P


def run_case(lib, D, P, *, bf16=False, l2norm=True, centered=True):
    B, T, H, _ = P["q"].shape
    scale = D ** -0.5
    names_in = ("q", "k", "v", "dout", "g", "beta", "lam", "S0", "C0", "m0", "dST", "dCT", "dmT")
    shapes = {"dq": (B, T, H, D), "dk": (B, T, H, D), "dv": (B, T, H, D), "dg": (B, T, H),
              "dbeta": (B, T, H), "dlam": (B, T, H), "dS0": (B, H, D, D), "dC0": (B, H, D, D), "dm0": (B, H, D)}
    out = {n: np.zeros(s, dtype=np.float32) for n, s in shapes.items()}
    ptr = lambda x: None if x is None else x.ctypes.data  # noqa: E731
    ins = (ctypes.c_void_p * 13)(*[ptr(P[n]) for n in names_in])
    outs = (ctypes.c_void_p * 9)(*[ptr(out[n]) for n in shapes])
    rc = lib.gdn_bwd_emu(D, int(bf16), B, T, H, int(l2norm), int(centered), scale, ins,
                         ptr(P["t0"]), outs)
    assert rc == 0
    ref = oracle.gdn_backward(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], P["dout"], S0=P["S0"],
                              C0=P["C0"], m0=P["m0"], t0=P["t0"], dST=P["dST"], dCT=P["dCT"], dmT=P["dmT"],
                              l2norm=l2norm, centered=centered, scale=scale)
    errs = {}
    for n in shapes:
        x = out[n].astype(np.float64)
        errs[n] = float(np.abs(x - ref[n]).max() / max(np.abs(ref[n]).max(), 1e-30)) \
            if np.all(np.isfinite(x)) else float("inf")
    return errs


CASES = [
    dict(D=16, B=1, T=130, H=2, seed=1),
    dict(D=16, B=2, T=200, H=1, seed=2, lam=0.9),
    dict(D=16, B=1, T=64, H=2, seed=3, states=False),
    dict(D=16, B=1, T=1, H=2, seed=4),
    dict(D=16, B=1, T=65, H=1, seed=5, opts=dict(l2norm=False)),
    dict(D=16, B=1, T=100, H=2, seed=6, opts=dict(centered=False)),
    dict(D=16, B=1, T=130, H=2, seed=7, bf16=True),
    dict(D=64, B=1, T=70, H=1, seed=8),
    # bf16 with D = 64: the tensor-core instantiation of the per-chunk kernels, whose products the
    # host computes on bf16-rounded operands (the bf16 bar for every gradient)
    dict(D=64, B=1, T=130, H=1, seed=9, bf16=True),
    dict(D=64, B=1, T=65, H=1, seed=10, bf16=True, lam=0.9, states=False),
    dict(D=64, B=1, T=100, H=1, seed=11, bf16=True, opts=dict(centered=False)),
    dict(D=64, B=1, T=70, H=1, seed=12, bf16=True, opts=dict(l2norm=False)),
    # D = 128: the two-block chains and the M = 128 products
    dict(D=128, B=1, T=80, H=1, seed=13, bf16=True),
]


@pytest.mark.parametrize("case", CASES, ids=[str(i) for i in range(len(CASES))])
def test_gdn_bwd_kernels_on_host(gdn_emu, oracle_mod, case):
    case = dict(case)
    opts = case.pop("opts", {})
    D, B, T, H, seed = (case.pop(n) for n in ("D", "B", "T", "H", "seed"))
    bf16 = case.get("bf16", False)
    P = problem(D, B, T, H, seed, **case)
    errs = run_case(gdn_emu, D, P, bf16=bf16, **opts)
    # bf16 inputs: dq, dk, dv are rounded to bf16 on output; with D >= 64 every product also takes
    # bf16 operands (the tensor-core path)
    tc = bf16 and D >= 64
    tol = {n: (2e-2 if tc or (bf16 and n in ("dq", "dk", "dv")) else 1e-4) for n in errs}
    bad = {n: e for n, e in errs.items() if not e <= tol[n]}
    assert not bad, f"{case}: {errs}"
