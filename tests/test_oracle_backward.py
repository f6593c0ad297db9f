"""Pins for the oracle's reverse mode (CCQ-GLA): every gradient is checked
against central finite differences of the fp64 forward (h = 1e-6) for the loss
L = sum(R_o * o) + sum(R_S * S_T) + sum(R_C * C_T) + sum(R_m * m_T)
with random weights R, so a wrong or missing adjoint term fails here."""
import numpy as np
import pytest

import oracle

GLA = 0
NAMES = ("q", "k", "v", "gk", "lam", "S0", "C0", "m0")


def problem(rng, T, Dk, Dv, B=1, H=1):
    P = {
        "q": rng.standard_normal((B, T, H, Dk)),
        "k": rng.standard_normal((B, T, H, Dk)),
        "v": rng.standard_normal((B, T, H, Dv)),
        "gk": np.log(1 / (1 + np.exp(-rng.standard_normal((B, T, H, Dk))))) / 4,
        "lam": rng.uniform(0.1, 0.9, (B, T, H)),
        "S0": rng.standard_normal((B, H, Dk, Dv)),
        "C0": None, "m0": None,
    }
    prev = unit(rng.standard_normal((B, 7, H, Dk)))
    P["C0"] = np.einsum("bthd,bthe->bhde", prev, prev)
    P["m0"] = prev.sum(axis=1)
    R = {"o": rng.standard_normal((B, T, H, Dv)), "S": rng.standard_normal((B, H, Dk, Dv)),
         "C": rng.standard_normal((B, H, Dk, Dk)), "m": rng.standard_normal((B, H, Dk))}
    return P, R, np.full(B, 7, dtype=np.int64)


def unit(x):
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def loss(P, R, t0, **kw):
    r = oracle.forward(GLA, P["q"], P["k"], P["v"], P["gk"], P["lam"], S0=P["S0"], C0=P["C0"],
                       m0=P["m0"], t0=t0, scale=0.8, nthreads=1, **kw)
    return (np.sum(R["o"] * r["o"]) + np.sum(R["S"] * r["S"]) + np.sum(R["C"] * r["C"])
            + np.sum(R["m"] * r["m"]))


def grads(P, R, t0, **kw):
    return oracle.gla_backward(P["q"], P["k"], P["v"], P["gk"], P["lam"], R["o"], S0=P["S0"],
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
def test_backward_matches_finite_differences_all_elements(centered):
    P, R, t0 = problem(np.random.default_rng(1), T=12, Dk=5, Dv=4)
    fd_check(P, R, t0, centered=centered)


def test_backward_across_checkpoint_blocks():
    """T = 130 spans three 64-token checkpoint blocks (sampled elements)."""
    P, R, t0 = problem(np.random.default_rng(2), T=130, Dk=6, Dv=5)
    fd_check(P, R, t0, sample=25, seed=3)


def test_backward_larger_dims_sampled():
    """T = 64, d = 16 (sampled elements)."""
    P, R, t0 = problem(np.random.default_rng(4), T=64, Dk=16, Dv=16)
    fd_check(P, R, t0, sample=20, seed=5)


def test_backward_zero_state_defaults_and_multi_head():
    rng = np.random.default_rng(6)
    B, T, H, Dk, Dv = 2, 9, 2, 4, 3
    q, k = rng.standard_normal((B, T, H, Dk)), rng.standard_normal((B, T, H, Dk))
    v = rng.standard_normal((B, T, H, Dv))
    gk = -np.abs(rng.standard_normal((B, T, H, Dk))) / 5
    lam = rng.uniform(0.1, 0.9, (B, T, H))
    do = rng.standard_normal((B, T, H, Dv))
    g = oracle.gla_backward(q, k, v, gk, lam, do, scale=0.5, nthreads=3)

    def L(qq):
        return np.sum(do * oracle.forward(GLA, qq, k, v, gk, lam, scale=0.5)["o"])
    h = 1e-6
    for (b, t, hh, d) in [(0, 0, 0, 0), (1, 8, 1, 3), (0, 4, 1, 2)]:
        qp, qm = q.copy(), q.copy()
        qp[b, t, hh, d] += h
        qm[b, t, hh, d] -= h
        fd = (L(qp) - L(qm)) / (2 * h)
        assert abs(fd - g["dq"][b, t, hh, d]) < 1e-7 * max(1.0, abs(fd))
