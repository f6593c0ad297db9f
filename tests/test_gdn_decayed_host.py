"""CPU check of the decay-aligned-covariance CCQ-Gated-DeltaNet forward kernels
(paper_2606_01294_gb300/csrc/ccq_gdn_decayed_kernels.cuh) against the oracle's
gdn_forward_decayed, itself pinned by brute-force weighted covariances
(tests/test_oracle_decayed.py).

The kernels are compiled for the host by tests/host_emu/gdn_cuda_core_emu.cpp (the gdn_emu
fixture) and run one thread per CTA, phase by phase, each CTA with exactly its dynamic shared
memory filled with NaN.  o, S_T, C_T, m_T and n_T are compared element by element: fp32
inputs to 1e-4, the fp32 bar; with bf16 inputs the output o is rounded to bf16 (2e-2)."""
import ctypes

import numpy as np
import pytest

import oracle
from tests.test_gdn_bwd_host import bf16_round


def problem(D, B, T, H, seed, *, bf16=False, lam=None, states=True, g_scale=1.0):
    rng = np.random.default_rng(seed)
    f32 = lambda a: np.ascontiguousarray(a, dtype=np.float32)  # noqa: E731
    P = {n: f32(rng.standard_normal((B, T, H, D))) for n in ("q", "k", "v")}
    if bf16:
        P = {n: bf16_round(x) for n, x in P.items()}
    P["g"] = f32(-np.log1p(np.exp(rng.standard_normal((B, T, H)))) * g_scale)
    P["beta"] = f32(1 / (1 + np.exp(-rng.standard_normal((B, T, H)))))
    P["lam"] = f32(np.full((B, T, H), lam) if lam is not None else
                   1 / (1 + np.exp(-(np.log(0.29 / 0.71) + 0.5 * rng.standard_normal((B, T, H))))))
    if states:
        # a consistent decayed history: C0 = sum_j w_j k_j k_j^T, m0 = sum_j w_j k_j, n0 = sum_j w_j
        hist = rng.standard_normal((B, H, 9, D))
        hist /= np.linalg.norm(hist, axis=-1, keepdims=True)
        w = np.exp(-0.3 * np.arange(9)[::-1])
        P.update(S0=f32(rng.standard_normal((B, H, D, D)) / D),
                 C0=f32(np.einsum("t,bhti,bhtj->bhij", w, hist, hist)),
                 m0=f32(np.einsum("t,bhti->bhi", w, hist)), n0=f32(np.full((B, H), w.sum())))
    else:
        P.update(S0=None, C0=None, m0=None, n0=None)
    return P


def run_case(lib, D, P, *, bf16=False, l2norm=True, centered=True, contraction=0, decayed=True):
    B, T, H, _ = P["q"].shape
    scale = D ** -0.5
    names_in = ("q", "k", "v", "g", "beta", "lam", "S0", "C0", "m0", "n0")
    shapes = {"o": (B, T, H, D), "S": (B, H, D, D), "C": (B, H, D, D), "m": (B, H, D), "n": (B, H)}
    out = {n: np.zeros(s, dtype=np.float32) for n, s in shapes.items()}
    ptr = lambda x: None if x is None else x.ctypes.data  # noqa: E731
    ins = (ctypes.c_void_p * 10)(*[ptr(P[n]) for n in names_in])
    outs = (ctypes.c_void_p * 5)(*[ptr(out[n]) for n in shapes])
    assert lib.gdn_spectral_emu(D, int(bf16), B, T, H, int(l2norm), int(centered), scale, contraction,
                                int(decayed), ins, outs) == 0
    if contraction == 0 and decayed:
        ref = oracle.gdn_forward_decayed(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], S0=P["S0"],
                                         C0=P["C0"], m0=P["m0"], n0=P["n0"], l2norm=l2norm, centered=centered,
                                         scale=scale)
    else:
        ref = oracle.gdn_forward_spectral(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"],
                                          contraction=contraction, decayed=decayed, S0=P["S0"], C0=P["C0"],
                                          m0=P["m0"], n0=P["n0"], l2norm=l2norm, centered=centered, scale=scale)
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
    dict(D=16, B=1, T=150, H=1, seed=7, g_scale=0.01),
    dict(D=16, B=1, T=130, H=2, seed=8, bf16=True),
    dict(D=64, B=1, T=70, H=1, seed=9),
]


@pytest.mark.parametrize("case", CASES, ids=[str(i) for i in range(len(CASES))])
def test_gdn_decayed_kernels_on_host(gdn_emu, oracle_mod, case):
    case = dict(case)
    opts = case.pop("opts", {})
    D, B, T, H, seed = (case.pop(n) for n in ("D", "B", "T", "H", "seed"))
    bf16 = case.get("bf16", False)
    errs = run_case(gdn_emu, D, problem(D, B, T, H, seed, **case), bf16=bf16, **opts)
    tol = {n: (2e-2 if bf16 and n == "o" else 1e-4) for n in errs}
    bad = {n: e for n, e in errs.items() if not e <= tol[n]}
    assert not bad, f"{case}: {errs}"


SPECTRAL = [
    dict(D=16, B=1, T=130, H=2, seed=11, opts=dict(contraction=1)),
    dict(D=16, B=1, T=130, H=2, seed=12, opts=dict(contraction=2)),
    dict(D=16, B=1, T=100, H=1, seed=13, lam=0.9, opts=dict(contraction=1, decayed=False)),
    dict(D=16, B=1, T=100, H=1, seed=14, lam=0.9, opts=dict(contraction=2, decayed=False)),
    dict(D=16, B=1, T=70, H=2, seed=15, opts=dict(contraction=0, decayed=False)),
    dict(D=16, B=1, T=65, H=1, seed=16, opts=dict(contraction=1, centered=False)),
    dict(D=16, B=1, T=1, H=1, seed=17, opts=dict(contraction=2)),
]


@pytest.mark.parametrize("case", SPECTRAL, ids=[str(i) for i in range(len(SPECTRAL))])
def test_gdn_spectral_kernels_on_host(gdn_emu, oracle_mod, case):
    """The resolvent and exponential contractions, with decayed and undecayed statistics,
    against oracle.gdn_forward_spectral; the undecayed linear case is the paper's CCQ-GDN."""
    case = dict(case)
    opts = case.pop("opts", {})
    D, B, T, H, seed = (case.pop(n) for n in ("D", "B", "T", "H", "seed"))
    P = problem(D, B, T, H, seed, **case)
    if not opts.get("decayed", True):
        P["n0"] = np.full((B, H), 9.0, dtype=np.float32)  # the entering count of the 9-key history
    errs = run_case(gdn_emu, D, P, **opts)
    assert max(errs.values()) <= 1e-4, f"{case} {opts}: {errs}"
