"""A second pin for the oracle's CCQ-Gated-DeltaNet reverse mode: the chunkwise adjoint.

The oracle differentiates the gated delta rule token by token. This file derives the same
gradients a different way, from the chunk form of the write (Gated DeltaNet's WY/UT
representation, as the forward of App. B / Algorithm 1 carries the backbone chunk by chunk):
per chunk of C tokens with in-chunk log-decay prefix gc and entering state H (rows = key dims),

    A  = strict_lower(diag(beta) (Kbar Kbar^T) * Gamma),  Gamma_ij = exp(gc_i - gc_j)
    Tb = (I + A)^{-1} diag(beta),   R = V - diag(exp(gc)) Kbar H,   U = Tb R
    O  = scale (diag(exp(gc)) Qc H + (Qc Kbar^T * Gamma * causal) U)
    H' = exp(gc_C) H + Kd^T U,      Kd = diag(exp(gc_C - gc)) Kbar

and runs the reverse mode of that chunk map with three carried adjoints (dH, and the key
statistics' dC, dm), chunks last to first. The two routes are algebraically identical, so
they must agree to rounding (about 1e-15 here), for any chunk size, ragged tails included.
That is far tighter than the finite-difference pins, and an adjoint term the token-by-token
oracle dropped or mis-signed would have to be dropped the same way in the (differently
shaped) chunk adjoint to pass. It also fixes the chunk decomposition a blocked backward
follows: a reverse state pass that needs only dH per chunk, then chunk-local gradients."""
import numpy as np
import pytest

import oracle


def _normalise(x, enabled):
    if not enabled:
        return x.copy(), np.ones(x.shape[0])
    n = np.linalg.norm(x, axis=-1)
    safe = np.where(n > 0, n, 1.0)
    return np.where(n[:, None] > 0, x / safe[:, None], 0.0), n


def _normalise_back(xb, n, dxb, enabled):
    if not enabled:
        return dxb
    safe = np.where(n > 0, n, 1.0)
    dx = (dxb - xb * np.sum(xb * dxb, 1, keepdims=True)) / safe[:, None]
    return np.where(n[:, None] > 0, dx, 0.0)


def _chunk(Q, K, V, g, be, lam, H, SK, M, t_start, c, scale):
    """The chunk map (forward) with every intermediate the adjoint needs."""
    n = Q.shape[0]
    t = t_start + 1.0 + np.arange(n)
    gc = np.cumsum(g)
    E = np.exp(gc)
    Gam = np.exp(gc[:, None] - gc[None, :])
    causal = np.tril(np.ones((n, n)))
    KK = K @ K.T
    # key statistics including token i: Sigma_i qbar_i (App. A.2)
    CumK = M[None, :] + np.cumsum(K, 0)
    z = (Q @ SK + ((Q @ K.T) * causal) @ K) / t[:, None] \
        - c * CumK * np.sum(CumK * Q, 1)[:, None] / t[:, None] ** 2
    qc = Q - lam[:, None] * z
    A = np.tril(be[:, None] * Gam * KK, -1)
    Tt = np.linalg.inv(np.eye(n) + A)
    Tb = Tt * be[None, :]
    R = V - E[:, None] * (K @ H)
    U = Tb @ R
    S = qc @ K.T
    P = S * Gam * causal
    Kd = np.exp(gc[-1] - gc)[:, None] * K
    return dict(t=t, gc=gc, E=E, Gam=Gam, causal=causal, KK=KK, CumK=CumK, z=z, qc=qc, A=A,
                Tt=Tt, Tb=Tb, R=R, U=U, S=S, P=P, Kd=Kd,
                Hn=np.exp(gc[-1]) * H + Kd.T @ U)


def chunkwise_backward(q, k, v, g, beta, lam, dout, S0, C0, m0, t0, dST, dCT, dmT, *,
                       chunk, centered=True, l2norm=True, scale=None):
    """Chunkwise reverse mode for one sequence and head (q, k [T,Dk]; v [T,Dv]; g, beta,
    lam [T]); returns the same gradients as ``oracle.gdn_backward``."""
    T, Dk = q.shape
    scale = Dk ** -0.5 if scale is None else scale
    c = 1.0 if centered else 0.0
    qb, qn = _normalise(q, l2norm)
    kb, kn = _normalise(k, l2norm)
    spans = [slice(s, min(T, s + chunk)) for s in range(0, T, chunk)]
    # forward: the state entering every chunk
    H, SK, M, tt = S0.copy(), C0.copy(), m0.copy(), int(t0)
    enter = []
    for s in spans:
        enter.append((H, SK, M, tt))
        H = _chunk(qb[s], kb[s], v[s], g[s], beta[s], lam[s], H, SK, M, tt, c, scale)["Hn"]
        SK = SK + kb[s].T @ kb[s]
        M = M + kb[s].sum(0)
        tt += s.stop - s.start
    dH, DC, Dm = dST.copy(), dCT.copy(), dmT.copy()
    out = {n: np.zeros_like(x) for n, x in
           (("dq", q), ("dk", k), ("dv", v), ("dg", g), ("dbeta", beta), ("dlam", lam))}
    dqb, dkb = np.zeros_like(q), np.zeros_like(k)
    for s, (H, SK, M, tt) in reversed(list(zip(spans, enter))):
        Q, K, be, lm = qb[s], kb[s], beta[s], lam[s]
        f = _chunk(Q, K, v[s], g[s], be, lm, H, SK, M, tt, c, scale)
        E, Gam, gc, U, Tt, Tb = f["E"], f["Gam"], f["gc"], f["U"], f["Tt"], f["Tb"]
        D = scale * dout[s]
        # backbone: dU = P^T D + Kd dH' and dR = Tb^T dU; v enters only through R
        dU = f["P"].T @ D + f["Kd"] @ dH
        dR = Tb.T @ dU
        out["dv"][s] = dR
        dP = (D @ U.T) * Gam * f["causal"]
        dqc = E[:, None] * (D @ H.T) + dP @ K
        dK = dP.T @ f["qc"] + np.exp(gc[-1] - gc)[:, None] * (U @ dH.T) - E[:, None] * (dR @ H.T)
        # through Tb = (I + A)^{-1} diag(beta): dA = -(I+A)^{-T} dTt (I+A)^{-T}
        dTb = dU @ f["R"].T
        dbe = np.sum(dTb * Tt, 0)
        dA = np.tril(-Tt.T @ (dTb * be[None, :]) @ Tt.T, -1)
        dbe += np.sum(dA * Gam * f["KK"], 1)
        dKK = dA * be[:, None] * Gam
        dK += dKK @ K + dKK.T @ K
        # log-decay prefix: every exp(gc_i - gc_j) factor, the read and the write
        AA = dA * f["A"]
        PP = dP * f["S"]
        dgc = AA.sum(1) - AA.sum(0) + PP.sum(1) - PP.sum(0)
        dgc += E * np.sum((f["qc"] @ H) * D, 1)
        kd = np.sum(f["Kd"] * (U @ dH.T), 1)
        dgc -= kd
        dgc[-1] += np.exp(gc[-1]) * np.sum(dH * H) + kd.sum()
        dgc -= E * np.sum((K @ H) * dR, 1)
        out["dg"][s] = np.cumsum(dgc[::-1])[::-1]
        out["dbeta"][s] = dbe
        dH_enter = np.exp(gc[-1]) * dH + (E[:, None] * f["qc"]).T @ D - (E[:, None] * K).T @ dR
        # CCQ read: q_clean = qbar - lam z, z = Sigma qbar (Eq. clean)
        t, CumK, z = f["t"], f["CumK"], f["z"]
        out["dlam"][s] = -np.sum(z * dqc, 1)
        dz = -lm[:, None] * dqc
        W = dz / t[:, None]
        cq, cz = np.sum(CumK * Q, 1), np.sum(CumK * dz, 1)
        causal = f["causal"]
        dqb[s] = dqc + W @ SK + ((W @ K.T) * causal) @ K - c * CumK * cz[:, None] / t[:, None] ** 2
        dCum = -c * (dz * cq[:, None] + Q * cz[:, None]) / t[:, None] ** 2
        dK += ((Q @ K.T) * causal).T @ W + ((W @ K.T) * causal).T @ Q
        dK += K @ (DC + DC.T) + Dm[None, :] + np.cumsum(dCum[::-1], 0)[::-1]
        dkb[s] = dK
        DC = DC + W.T @ Q
        Dm = Dm + dCum.sum(0)
        dH = dH_enter
    out["dq"] = _normalise_back(qb, qn, dqb, l2norm)
    out["dk"] = _normalise_back(kb, kn, dkb, l2norm)
    out.update(dS0=dH, dC0=DC, dm0=Dm)
    return out


def _problem(rng, B, T, H, Dk, Dv, t0=7):
    q = rng.standard_normal((B, T, H, Dk))
    k = rng.standard_normal((B, T, H, Dk))
    prev = rng.standard_normal((B, t0, H, Dk))
    prev /= np.linalg.norm(prev, axis=-1, keepdims=True)
    P = dict(
        q=q, k=k, v=rng.standard_normal((B, T, H, Dv)),
        g=-np.log1p(np.exp(rng.standard_normal((B, T, H)))),
        beta=1 / (1 + np.exp(-rng.standard_normal((B, T, H)))),
        lam=rng.uniform(0.1, 0.9, (B, T, H)),
        dout=rng.standard_normal((B, T, H, Dv)),
        S0=rng.standard_normal((B, H, Dk, Dv)),
        C0=np.einsum("bthd,bthe->bhde", prev, prev), m0=prev.sum(1),
        t0=np.full(B, t0, dtype=np.int64),
        dST=rng.standard_normal((B, H, Dk, Dv)), dCT=rng.standard_normal((B, H, Dk, Dk)),
        dmT=rng.standard_normal((B, H, Dk)))
    return P


def _check(P, chunk, centered=True, l2norm=True, tol=1e-11):
    ref = oracle.gdn_backward(P["q"], P["k"], P["v"], P["g"], P["beta"], P["lam"], P["dout"],
                              P["S0"], P["C0"], P["m0"], P["t0"], P["dST"], P["dCT"], P["dmT"],
                              centered=centered, l2norm=l2norm)
    B, T, H, _ = P["q"].shape
    for b in range(B):
        for h in range(H):
            tok = {n: P[n][b, :, h] for n in ("q", "k", "v", "g", "beta", "lam", "dout")}
            st = {n: P[n][b, h] for n in ("S0", "C0", "m0", "dST", "dCT", "dmT")}
            got = chunkwise_backward(**tok, **st, t0=P["t0"][b], chunk=chunk,
                                     centered=centered, l2norm=l2norm)
            for name, val in got.items():
                want = ref[name][b, h] if name in ("dS0", "dC0", "dm0") else ref[name][b, :, h]
                err = np.max(np.abs(val - want)) / max(np.max(np.abs(want)), 1e-300)
                assert err < tol, f"{name} (b={b}, h={h}): relative error {err:.3e}"


@pytest.mark.parametrize("T,chunk", [(12, 4), (150, 64), (128, 64), (1, 64), (37, 16)])
def test_chunkwise_adjoint_matches_token_adjoint(T, chunk):
    _check(_problem(np.random.default_rng(1000 + T), 1, T, 1, 16, 12), chunk)


def test_chunkwise_adjoint_uncentred_and_several_heads():
    _check(_problem(np.random.default_rng(7), 2, 70, 2, 8, 8), 32, centered=False)


def test_chunkwise_adjoint_without_normalisation():
    P = _problem(np.random.default_rng(8), 1, 40, 1, 8, 8)
    # keys of norm <= 1 keep the un-normalised delta rule contractive
    P["k"] = P["k"] / (1.5 * np.linalg.norm(P["k"], axis=-1, keepdims=True))
    _check(P, 16, l2norm=False)


def test_chunkwise_adjoint_with_zero_rows():
    P = _problem(np.random.default_rng(9), 1, 50, 1, 8, 8)
    P["q"][0, 3, 0] = 0.0
    P["k"][0, 17, 0] = 0.0
    P["k"][0, 32, 0] = 0.0
    _check(P, 16)
