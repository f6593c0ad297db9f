"""Pins for the oracle's reverse mode of CCQ-Gated-DeltaNet: every gradient is checked
against central finite differences of the fp64 forward (h = 1e-6) for the loss
L = sum(R_o * o) + sum(R_S * S_T) + sum(R_C * C_T) + sum(R_m * m_T)
with random weights R, so a wrong or missing adjoint term of the delta-rule write
(the beta, decay, key and value paths) or of the cleaned query fails here."""
import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle
from oracle import ccq_oracle

GDN = 1
NAMES = ("q", "k", "v", "g", "beta", "lam", "S0", "C0", "m0")


def unit(x):
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def problem(rng, T, Dk, Dv, B=1, H=1):
    P = {
        "q": rng.standard_normal((B, T, H, Dk)),
        "k": rng.standard_normal((B, T, H, Dk)),
        "v": rng.standard_normal((B, T, H, Dv)),
        # scalar log decay -softplus(x) and beta = sigmoid(x), the workload's distributions
        "g": -np.log1p(np.exp(rng.standard_normal((B, T, H)))),
        "beta": 1 / (1 + np.exp(-rng.standard_normal((B, T, H)))),
        "lam": rng.uniform(0.1, 0.9, (B, T, H)),
        "S0": rng.standard_normal((B, H, Dk, Dv)),
    }
    prev = unit(rng.standard_normal((B, 7, H, Dk)))
    P["C0"] = np.einsum("bthd,bthe->bhde", prev, prev)
    P["m0"] = prev.sum(axis=1)
    R = {"o": rng.standard_normal((B, T, H, Dv)), "S": rng.standard_normal((B, H, Dk, Dv)),
         "C": rng.standard_normal((B, H, Dk, Dk)), "m": rng.standard_normal((B, H, Dk))}
    return P, R, np.full(B, 7, dtype=np.int64)


def loss(P, R, t0, **kw):
    r = oracle.forward(GDN, P["q"], P["k"], P["v"], P["g"], P["lam"], beta=P["beta"], S0=P["S0"],
                       C0=P["C0"], m0=P["m0"], t0=t0, scale=0.8, nthreads=1, **kw)
    return (np.sum(R["o"] * r["o"]) + np.sum(R["S"] * r["S"]) + np.sum(R["C"] * r["C"])
            + np.sum(R["m"] * r["m"]))


def grads(P, R, t0, **kw):
    return oracle.gdn_backward(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], R["o"], S0=P["S0"],
                               C0=P["C0"], m0=P["m0"], t0=t0, dST=R["S"], dCT=R["C"], dmT=R["m"],
                               scale=0.8, nthreads=1, **kw)


def fd_check(P, R, t0, sample=None, seed=0, **kw):
    g = grads(P, R, t0, **kw)
    rng = np.random.default_rng(seed)
    h = 1e-6
    for name in NAMES:
        x = P[name]
        flat = x.reshape(-1)
        idx = np.arange(flat.size) if sample is None else rng.choice(flat.size, min(sample, flat.size),
                                                                       replace=False)
        fd = np.empty(len(idx))
        for n, i in enumerate(idx):
            old = flat[i]
            flat[i] = old + h
            lp = loss(P, R, t0, **kw)
            flat[i] = old - h
            lm = loss(P, R, t0, **kw)
            flat[i] = old
            fd[n] = (lp - lm) / (2 * h)
        an = g["d" + name].reshape(-1)[idx]
        scale = max(np.abs(an).max(), 1e-12)
        err = np.abs(an - fd).max() / scale
        assert err < 1e-6, f"d{name}: max relative deviation from finite differences {err:.2e}"


@pytest.mark.parametrize("centered", [True, False])
def test_gdn_backward_matches_finite_differences_all_elements(centered):
    P, R, t0 = problem(np.random.default_rng(11), T=12, Dk=5, Dv=4)
    fd_check(P, R, t0, centered=centered)


def test_gdn_backward_unnormalised_keys():
    P, R, t0 = problem(np.random.default_rng(12), T=9, Dk=4, Dv=3)
    P["k"] *= 0.3  # the delta rule is then far from a projection
    fd_check(P, R, t0, l2norm=False)


def test_gdn_backward_across_checkpoint_blocks():
    """T = 130 spans three 64-token checkpoint blocks (sampled elements), two heads."""
    P, R, t0 = problem(np.random.default_rng(13), T=130, Dk=4, Dv=3, H=2)
    fd_check(P, R, t0, sample=12, seed=3)


def test_gdn_backward_reduces_to_plain_gated_deltanet_at_lambda_zero():
    """With lambda = 0 the query is not contracted: no gradient reaches lambda's
    partners C0 and m0, and dlam is -z . dq_clean, not zero."""
    P, R, t0 = problem(np.random.default_rng(14), T=10, Dk=4, Dv=3)
    P["lam"][:] = 0.0
    R["C"][:] = 0.0
    R["m"][:] = 0.0
    g = grads(P, R, t0)
    assert np.abs(g["dC0"]).max() == 0.0 and np.abs(g["dm0"]).max() == 0.0
    assert np.abs(g["dlam"]).max() > 0.0
    fd_check(P, R, t0)


# ---- the pins notice plausible mistakes in the delta-rule adjoints (each planted in a
# private copy of the oracle's C source, compiled on the CPU)
MUTANTS = {
    "u path dropped from dkbar": ("hs += Sp[(size_t)i * Dv + e] * du[e];", "hs += 0.0;"),
    "dbeta without the erase term": ("dbe += kb[i] * G * (vr[e] - a * u[e]);", "dbe += kb[i] * G * vr[e];"),
    "previous-state adjoint misses kbar du^T": (
        "dS[(size_t)i * Dv + e] = a * dS[(size_t)i * Dv + e] + kb[i] * du[e];",
        "dS[(size_t)i * Dv + e] = a * dS[(size_t)i * Dv + e];"),
    "dg not scaled by the decay": ("J->dgk[r] = a * da;", "J->dgk[r] = da;"),
    "dv without beta": ("J->dv[r * Dv + e] = be * acc;", "J->dv[r * Dv + e] = acc;"),
    "du sign flipped": ("du[e] = -a * be * acc;", "du[e] = a * be * acc;"),
}


def _battery(lib):
    rng = np.random.default_rng(5)
    P, R, t0 = problem(rng, T=6, Dk=3, Dv=2)
    g = oracle.gdn_backward(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], R["o"], S0=P["S0"],
                            C0=P["C0"], m0=P["m0"], t0=t0, dST=R["S"], dCT=R["C"], dmT=R["m"],
                            scale=0.8, nthreads=1, lib=lib)

    def L():
        r = oracle.forward(GDN, P["q"], P["k"], P["v"], P["g"], P["lam"], beta=P["beta"], S0=P["S0"],
                           C0=P["C0"], m0=P["m0"], t0=t0, scale=0.8, nthreads=1, lib=lib)
        return (np.sum(R["o"] * r["o"]) + np.sum(R["S"] * r["S"]) + np.sum(R["C"] * r["C"])
                + np.sum(R["m"] * r["m"]))

    h = 1e-6
    for name in NAMES:
        flat = P[name].reshape(-1)
        an = g["d" + name].reshape(-1)
        for i in range(flat.size):
            old = flat[i]
            flat[i] = old + h
            lp = L()
            flat[i] = old - h
            lm = L()
            flat[i] = old
            if abs(an[i] - (lp - lm) / (2 * h)) > 1e-6 * max(np.abs(an).max(), 1e-12):
                return False
    return True


def test_gdn_backward_battery_accepts_the_oracle():
    assert _battery(ccq_oracle._load())


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_gdn_backward_battery_rejects_mutant(tmp_path, name):
    with open(ccq_oracle._SRC) as f:
        src = f.read()
    old, new = MUTANTS[name]
    assert src.count(old) == 1, f"mutation site for {name!r} is not unique"
    c, so = os.path.join(tmp_path, "m.c"), os.path.join(tmp_path, "m.so")
    with open(c, "w") as f:
        f.write(src.replace(old, new))
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-pthread", c, "-o", so, "-lm"])
    assert not _battery(ccq_oracle.load_library(so)), f"pins did not notice: {name}"
    shutil.rmtree(tmp_path, ignore_errors=True)
