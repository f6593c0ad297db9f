"""Pins for the oracle's decay-aligned covariance (CCQ-Gated-DeltaNet).

The paper names a covariance from gamma-weighted running statistics as the variant suited to
decayed backbones, without fixing gamma or the normaliser. The oracle's reading: gamma_{j,t} is
the product of the Gated DeltaNet decays alpha_s over j < s <= t, and the normaliser is the
decayed count sum_j gamma_{j,t}. So Sigma^gamma_t is the gamma-weighted sample covariance of
the keys seen so far. These pins check the running-sum recursion against that definition,
written out independently:
  - brute force: the two-pass weighted covariance of an explicit key history (a prefix turned
    into the initial state plus the call's own tokens), hence the cleaned queries;
  - every alpha = 1 gives the undecayed oracle exactly (n takes the place of t);
  - the backbone write does not depend on the covariance: S_T equals the undecayed oracle's,
    and o_t = scale S_t^T q_clean_t against a plain numpy delta-rule recurrence;
  - a weighted covariance of unit keys has spectrum in [0, 1], so
    (1 - lambda)|qbar| <= |q_clean| <= |qbar|;
  - a very strong decay forgets every key but the current one;
  - two calls carrying (S, C, m, n) equal one call.
Three planted mistakes in the recursion (an undecayed count, an undecayed second moment, the
mean term over n instead of n^2) each fail the battery."""
import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle
from oracle import ccq_oracle

GDN = 1


def unit(x):
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def problem(rng, T, Dk=6, Dv=5, prefix=4, g_scale=1.0):
    q = rng.standard_normal((1, T, 1, Dk))
    k = rng.standard_normal((1, T, 1, Dk))
    v = rng.standard_normal((1, T, 1, Dv))
    g = -g_scale * np.log1p(np.exp(rng.standard_normal((1, T, 1))))
    beta = 1 / (1 + np.exp(-rng.standard_normal((1, T, 1))))
    lam = rng.uniform(0.1, 0.9, (1, T, 1))
    # an explicit history: prefix keys and their decays, folded into the initial statistics
    kp = unit(rng.standard_normal((prefix, Dk)))
    gp = -np.log1p(np.exp(rng.standard_normal(prefix)))
    return dict(q=q, k=k, v=v, g=g, beta=beta, lam=lam, kp=kp, gp=gp,
                S0=rng.standard_normal((1, 1, Dk, Dv)))


def prefix_state(kp, gp):
    """Decayed statistics of the prefix alone: key j weighted by the decays after it."""
    P = len(kp)
    w = np.array([np.exp(gp[j + 1:].sum()) for j in range(P)])
    C0 = np.einsum("j,jd,je->de", w, kp, kp)
    return C0[None, None], (w @ kp)[None, None], np.array([[w.sum()]])


def brute_qclean(P, centered=True):
    """q_clean_t from the weighted two-pass covariance of the explicit history."""
    q, k, lam = P["q"][0, :, 0], unit(P["k"][0, :, 0]), P["lam"][0, :, 0]
    g = P["g"][0, :, 0]
    keys = np.concatenate([P["kp"], k])
    decays = np.concatenate([P["gp"], g])
    Pn = len(P["kp"])
    out = []
    for t in range(len(q)):
        last = Pn + t
        w = np.array([np.exp(decays[j + 1:last + 1].sum()) for j in range(last + 1)])
        W = w.sum()
        mu = (w @ keys[:last + 1]) / W
        if centered:
            X = keys[:last + 1] - mu
            Sig = np.einsum("j,jd,je->de", w / W, X, X)
        else:
            Sig = np.einsum("j,jd,je->de", w / W, keys[:last + 1], keys[:last + 1])
        qb = unit(q[t])
        out.append(qb - lam[t] * Sig @ qb)
    return np.array(out)


def brute_output(P, qc, scale):
    """o_t = scale S_t^T q_clean_t with a plain delta-rule recurrence for S (rows = key dims)."""
    k, v = unit(P["k"][0, :, 0]), P["v"][0, :, 0]
    g, beta = P["g"][0, :, 0], P["beta"][0, :, 0]
    Hs = P["S0"][0, 0].copy()
    out = []
    for t in range(len(k)):
        a = np.exp(g[t])
        Hs = a * (Hs - beta[t] * np.outer(k[t], k[t] @ Hs)) + beta[t] * np.outer(k[t], v[t])
        out.append(scale * Hs.T @ qc[t])
    return np.array(out), Hs


def run(P, lib=None, **kw):
    C0, m0, n0 = prefix_state(P["kp"], P["gp"])
    return oracle.gdn_forward_decayed(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], S0=P["S0"],
                                      C0=C0, m0=m0, n0=n0, want_qclean=True, scale=0.7, nthreads=1,
                                      lib=lib, **kw)


@pytest.mark.parametrize("centered", [True, False])
def test_qclean_is_the_weighted_history_covariance(centered):
    P = problem(np.random.default_rng(1), T=11)
    r = run(P, centered=centered)
    np.testing.assert_allclose(r["qclean"][0, :, 0], brute_qclean(P, centered), atol=1e-12)


def test_output_and_state_follow_the_delta_rule():
    P = problem(np.random.default_rng(2), T=9)
    r = run(P)
    o, S_T = brute_output(P, r["qclean"][0, :, 0], 0.7)
    np.testing.assert_allclose(r["o"][0, :, 0], o, atol=1e-12)
    np.testing.assert_allclose(r["S"][0, 0], S_T, atol=1e-12)


def test_no_decay_is_the_undecayed_oracle():
    rng = np.random.default_rng(3)
    P = problem(rng, T=20)
    P["g"][:] = 0.0
    C0 = np.einsum("jd,je->de", P["kp"], P["kp"])[None, None]
    m0 = P["kp"].sum(0)[None, None]
    n = len(P["kp"])
    d = oracle.gdn_forward_decayed(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], S0=P["S0"], C0=C0,
                                   m0=m0, n0=np.array([[float(n)]]), scale=0.7, nthreads=1)
    u = oracle.forward(GDN, P["q"], P["k"], P["v"], P["g"], P["lam"], beta=P["beta"], S0=P["S0"], C0=C0,
                       m0=m0, t0=np.array([n]), scale=0.7, nthreads=1)
    for name in ("o", "S", "C", "m"):
        np.testing.assert_allclose(d[name], u[name], atol=1e-12, err_msg=name)
    assert d["n"][0, 0] == n + 20


@pytest.mark.parametrize("lam", [0.3, 0.9])
def test_cleaning_spectrum_bound(lam):
    P = problem(np.random.default_rng(4), T=40, g_scale=0.3)
    P["lam"][:] = lam
    r = run(P)
    qb = unit(P["q"][0, :, 0])
    nq = np.linalg.norm(r["qclean"][0, :, 0], axis=-1)
    assert np.all(nq <= 1 + 1e-12) and np.all(nq >= (1 - lam) - 1e-12)
    assert np.allclose(np.linalg.norm(qb, axis=-1), 1.0)


def test_strong_decay_keeps_only_the_current_key():
    P = problem(np.random.default_rng(5), T=7)
    P["g"][:] = -60.0
    for centered in (True, False):
        r = run(P, centered=centered)
        qb = unit(P["q"][0, :, 0])
        kb = unit(P["k"][0, :, 0])
        want = qb if centered else qb - P["lam"][0, :, 0, None] * kb * np.sum(kb * qb, -1, keepdims=True)
        np.testing.assert_allclose(r["qclean"][0, :, 0], want, atol=1e-12)


def test_two_calls_equal_one():
    P = problem(np.random.default_rng(6), T=30)
    whole = run(P)
    C0, m0, n0 = prefix_state(P["kp"], P["gp"])
    cut = 13
    part = lambda x, s: x[:, s]  # noqa: E731
    a = oracle.gdn_forward_decayed(*(part(P[n], slice(0, cut)) for n in ("q", "k", "v", "g", "beta", "lam")),
                                   S0=P["S0"], C0=C0, m0=m0, n0=n0, scale=0.7, nthreads=1)
    b = oracle.gdn_forward_decayed(*(part(P[n], slice(cut, None)) for n in ("q", "k", "v", "g", "beta", "lam")),
                                   S0=a["S"], C0=a["C"], m0=a["m"], n0=a["n"], scale=0.7, nthreads=1)
    np.testing.assert_allclose(np.concatenate([a["o"], b["o"]], axis=1), whole["o"], atol=1e-12)
    for name in ("S", "C", "m", "n"):
        np.testing.assert_allclose(b[name], whole[name], atol=1e-12, err_msg=name)


MUTANTS = {
    "count not decayed": ("n = a * n + 1.0;", "n = n + 1.0;"),
    "second moment not decayed": ("Cg[(size_t)i * Dk + j] = a * Cg[(size_t)i * Dk + j] + kb[i] * kb[j];",
                                  "Cg[(size_t)i * Dk + j] = Cg[(size_t)i * Dk + j] + kb[i] * kb[j];"),
    "mean term over n": ("mg[i] * mq / (n * n)", "mg[i] * mq / n"),
}


def _battery(lib):
    P = problem(np.random.default_rng(7), T=8)
    r = run(P, lib=lib)
    return bool(np.allclose(r["qclean"][0, :, 0], brute_qclean(P), atol=1e-12))


def test_decayed_battery_accepts_the_oracle():
    assert _battery(ccq_oracle._load())


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_decayed_battery_rejects_mutant(tmp_path, name):
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
