"""The oracle's pins are strong enough to notice plausible mistakes.

Each case plants one mistake in a private copy of the oracle's C source (on
the CPU, in a temporary directory), compiles it, and checks that the pin
battery below rejects the mutant while accepting the real oracle.
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle
from oracle import ccq_oracle
from tests.test_oracle_pins import (GDN, GLA, brute_gdn, brute_gla, brute_qclean,
                                    rand_problem)

MUTANTS = {
    "mean term dropped": ("if (centered) out[i] -= ms[i] * mq / (t * t);", ""),
    "mean term over t instead of t^2": ("ms[i] * mq / (t * t)", "ms[i] * mq / t"),
    "correction sign flipped": ("qc[i] = qb[i] - lam * sq[i];", "qc[i] = qb[i] + lam * sq[i];"),
    "normaliser off by one": ("out[i] = acc / t;", "out[i] = acc / (t + 1.0);"),
    "Sigma applied to the raw query": ("sigma_times(Cs, ms, qb, Dk", "sigma_times(Cs, ms, qr, Dk"),
    "GLA decays the new write": ("a * Hs[(size_t)i * Dv + j] + kb[i] * vr[j]",
                                 "a * (Hs[(size_t)i * Dv + j] + kb[i] * vr[j])"),
    "GLA writes the raw key": ("+ kb[i] * vr[j];\n", "+ kr[i] * vr[j];\n"),
    "GDN erase term not decayed": ("a * (Hs[(size_t)i * Dv + j] - be * kb[i] * kS[j])",
                                   "(a * Hs[(size_t)i * Dv + j] - be * kb[i] * kS[j])"),
    "GDN erase without beta": ("- be * kb[i] * kS[j])", "- kb[i] * kS[j])"),
    "chunkwise intra mask drops the diagonal": (
        "for (int j = 0; j <= i; ++j) {\n                const double *kj = Kb + (size_t)j * Dk;\n"
        "                double s = 0.0;\n                for (int e = 0; e < Dk; ++e) s += qi[e] * kj[e];",
        "for (int j = 0; j < i; ++j) {\n                const double *kj = Kb + (size_t)j * Dk;\n"
        "                double s = 0.0;\n                for (int e = 0; e < Dk; ++e) s += qi[e] * kj[e];"),
    "chunkwise GLA state decay uses the first gate": (
        "double acc = exp(Gn[a]) * Hs[(size_t)a * Dv + e];", "double acc = exp(G[a]) * Hs[(size_t)a * Dv + e];"),
    "chunkwise GDN triangular term sign": ("ui[e] -= Aij * U[(size_t)j * Dv + e];",
                                           "ui[e] += Aij * U[(size_t)j * Dv + e];"),
}


def battery(lib) -> bool:
    """True when every pin in the battery holds for ``lib``."""
    rng = np.random.default_rng(99)
    ok = True
    P = rand_problem(rng, 1, 13, 1, 5, 4, GLA)
    S0 = rng.standard_normal((1, 1, 5, 4))
    r = oracle.forward(GLA, P["q"], P["k"], P["v"], P["gate"], P["lam"], S0=S0, scale=0.8,
                       want_qclean=True, lib=lib)
    ok &= np.allclose(r["qclean"][0, :, 0], brute_qclean(P["q"][0, :, 0], P["k"][0, :, 0],
                                                         P["lam"][0, :, 0]), atol=1e-11)
    ok &= np.allclose(r["o"][0, :, 0], brute_gla(P["q"][0, :, 0], P["k"][0, :, 0], P["v"][0, :, 0],
                                                 P["gate"][0, :, 0], P["lam"][0, :, 0], S0[0, 0], 0.8),
                      atol=1e-11)
    G = rand_problem(rng, 1, 11, 1, 5, 4, GDN)
    S0 = rng.standard_normal((1, 1, 5, 4))
    r = oracle.forward(GDN, G["q"], G["k"], G["v"], G["gate"], G["lam"], beta=G["beta"], S0=S0,
                       scale=0.8, lib=lib)
    ok &= np.allclose(r["o"][0, :, 0], brute_gdn(G["q"][0, :, 0], G["k"][0, :, 0], G["v"][0, :, 0],
                                                 G["gate"][0, :, 0], G["beta"][0, :, 0],
                                                 G["lam"][0, :, 0], S0[0, 0], 0.8), atol=1e-11)
    for bb, PP in ((GLA, P), (GDN, G)):
        kw = dict(beta=PP["beta"], lib=lib)
        rec = oracle.forward(bb, PP["q"], PP["k"], PP["v"], PP["gate"], PP["lam"], **kw)
        chk = oracle.forward(bb, PP["q"], PP["k"], PP["v"], PP["gate"], PP["lam"], chunk=4, **kw)
        ok &= np.allclose(chk["o"], rec["o"], atol=1e-11) and np.allclose(chk["S"], rec["S"], atol=1e-11)
    return bool(ok)


def _compile(src_text, out_dir, name):
    c = os.path.join(out_dir, name + ".c")
    so = os.path.join(out_dir, name + ".so")
    with open(c, "w") as f:
        f.write(src_text)
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-pthread", c, "-o", so, "-lm"])
    return ccq_oracle.load_library(so)


@pytest.fixture(scope="module")
def source():
    with open(ccq_oracle._SRC) as f:
        return f.read()


def test_battery_accepts_the_oracle(oracle_mod):
    assert battery(ccq_oracle._load())


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_battery_rejects_mutant(source, tmp_path, name):
    old, new = MUTANTS[name]
    assert source.count(old) == 1, f"mutation site for {name!r} is not unique"
    lib = _compile(source.replace(old, new), str(tmp_path), "mutant")
    assert not battery(lib), f"pins did not notice: {name}"
    shutil.rmtree(tmp_path, ignore_errors=True)
