"""Pins for the oracle's spectral contractions of the CCQ read.

The paper's cleaning operator I - lambda Sigma is the first-order form of the alternatives it
names, (I + lambda Sigma)^{-1} and exp(-lambda Sigma) (Sec. 3.2, after Eq. clean).
oracle.gdn_forward_spectral evaluates all three token by token; these tests fix it to things
other than itself:
  - the linear contraction reproduces the C oracle: the paper's CCQ-Gated-DeltaNet (undecayed
    statistics, n = t) and the decay-aligned reading (gdn_forward_decayed);
  - the cleaned query equals U f(lambda sigma) U^T qbar from an eigendecomposition of the
    two-pass covariance of the explicit key history;
  - each alternative differs from the linear one by O(lambda^2) (halving lambda quarters it);
  - unit keys give Sigma a spectrum in [0, 1], so |q_clean| lies in [|qbar|/(1+lambda), |qbar|]
    (resolvent) and [e^{-lambda}|qbar|, |qbar|] (exponential), and since
    1 - x <= e^{-x} <= 1/(1+x) on [0, 1], |q_lin| <= |q_exp| <= |q_res|."""
import numpy as np
import pytest

import oracle
from oracle import ccq_oracle

GDN = oracle.GDN


def _problem(rng, T, Dk=6, Dv=5, H=1, lam=None):
    P = dict(q=rng.standard_normal((1, T, H, Dk)), k=rng.standard_normal((1, T, H, Dk)),
             v=rng.standard_normal((1, T, H, Dv)), g=-np.log1p(np.exp(rng.standard_normal((1, T, H)))),
             beta=1 / (1 + np.exp(-rng.standard_normal((1, T, H)))),
             lam=np.full((1, T, H), lam) if lam is not None else rng.uniform(0.1, 0.9, (1, T, H)))
    return P


def _state(rng, Dk=6, Dv=5, H=1, t0=5):
    hist = rng.standard_normal((1, H, t0, Dk))
    hist /= np.linalg.norm(hist, axis=-1, keepdims=True)
    return dict(S0=rng.standard_normal((1, H, Dk, Dv)) / Dk, C0=np.einsum("bhti,bhtj->bhij", hist, hist),
                m0=hist.sum(2), hist=hist)


@pytest.mark.parametrize("centered", [True, False])
def test_linear_is_the_c_oracle(oracle_mod, centered):
    rng = np.random.default_rng(1)
    P, st = _problem(rng, 40), _state(rng)
    ref = oracle.forward(GDN, P["q"], P["k"], P["v"], P["g"], P["lam"], beta=P["beta"], S0=st["S0"], C0=st["C0"],
                         m0=st["m0"], t0=np.array([5]), centered=centered)
    r = oracle.gdn_forward_spectral(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], S0=st["S0"], C0=st["C0"],
                                    m0=st["m0"], n0=np.array([[5.0]]), centered=centered)
    for n in ("o", "S", "C", "m"):
        np.testing.assert_allclose(r[n], ref[n], rtol=1e-11, atol=1e-12)
    assert r["n"][0, 0] == 45.0
    dec = oracle.gdn_forward_decayed(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], S0=st["S0"],
                                     C0=st["C0"], m0=st["m0"], n0=np.array([[5.0]]), centered=centered)
    r = oracle.gdn_forward_spectral(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], decayed=True,
                                    S0=st["S0"], C0=st["C0"], m0=st["m0"], n0=np.array([[5.0]]), centered=centered)
    for n in ("o", "S", "C", "m", "n"):
        np.testing.assert_allclose(r[n], dec[n], rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("contraction,f", [(ccq_oracle.RESOLVENT, lambda x: 1 / (1 + x)),
                                           (ccq_oracle.EXPONENTIAL, lambda x: np.exp(-x)),
                                           (ccq_oracle.LINEAR, lambda x: 1 - x)])
def test_qclean_from_the_eigendecomposition(contraction, f):
    rng = np.random.default_rng(2)
    T = 12
    P, st = _problem(rng, T), _state(rng)
    r = oracle.gdn_forward_spectral(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], contraction=contraction,
                                    C0=st["C0"], m0=st["m0"], n0=np.array([[5.0]]), want_qclean=True)
    keys = list(st["hist"][0, 0])
    for t in range(T):
        kb = P["k"][0, t, 0] / np.linalg.norm(P["k"][0, t, 0])
        keys.append(kb)
        K = np.array(keys)
        mu = K.mean(0)
        Sig = (K - mu).T @ (K - mu) / len(K)          # two-pass covariance of the history
        sig, U = np.linalg.eigh(Sig)
        qb = P["q"][0, t, 0] / np.linalg.norm(P["q"][0, t, 0])
        want = U @ (f(P["lam"][0, t, 0] * sig) * (U.T @ qb))
        np.testing.assert_allclose(r["qclean"][0, t, 0], want, rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("contraction", [ccq_oracle.RESOLVENT, ccq_oracle.EXPONENTIAL])
def test_first_order_agreement(contraction):
    rng = np.random.default_rng(3)
    P = _problem(rng, 20)
    diffs = []
    for lam in (2e-3, 1e-3):
        P["lam"] = np.full_like(P["lam"], lam)
        a = oracle.gdn_forward_spectral(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"],
                                        contraction=contraction, want_qclean=True)["qclean"]
        b = oracle.gdn_forward_spectral(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"],
                                        want_qclean=True)["qclean"]
        diffs.append(np.abs(a - b).max())
    assert diffs[1] > 0
    assert 3.6 < diffs[0] / diffs[1] < 4.4   # O(lambda^2)


@pytest.mark.parametrize("lam", [0.3, 0.9])
def test_spectrum_bounds_and_ordering(lam):
    rng = np.random.default_rng(4)
    P = _problem(rng, 30, lam=lam)
    qc = {c: oracle.gdn_forward_spectral(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], contraction=c,
                                         want_qclean=True)["qclean"][0, :, 0]
          for c in (ccq_oracle.LINEAR, ccq_oracle.RESOLVENT, ccq_oracle.EXPONENTIAL)}
    nrm = {c: np.linalg.norm(x, axis=-1) for c, x in qc.items()}
    one = np.ones_like(nrm[ccq_oracle.LINEAR])   # |qbar| = 1
    eps = 1e-12
    assert np.all(nrm[ccq_oracle.RESOLVENT] >= one / (1 + lam) - eps) and np.all(nrm[ccq_oracle.RESOLVENT] <= one + eps)
    assert np.all(nrm[ccq_oracle.EXPONENTIAL] >= np.exp(-lam) * one - eps)
    assert np.all(nrm[ccq_oracle.EXPONENTIAL] <= one + eps)
    assert np.all(nrm[ccq_oracle.LINEAR] <= nrm[ccq_oracle.EXPONENTIAL] + eps)
    assert np.all(nrm[ccq_oracle.EXPONENTIAL] <= nrm[ccq_oracle.RESOLVENT] + eps)
