"""Pins for the fp64 oracle: each test checks it against something other than
itself -- a brute-force formula written independently in numpy, a closed form,
an invariant the paper proves, or a finite-difference derivative.

Paper references are to arxiv 2606.01294 (sections, equations, algorithms).
"""
import numpy as np
import pytest

GLA, GDN = 0, 1


def unit(x):
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def rand_problem(rng, B, T, H, Dk, Dv, backbone=GLA, lam=None):
    q = rng.standard_normal((B, T, H, Dk))
    k = rng.standard_normal((B, T, H, Dk))
    v = rng.standard_normal((B, T, H, Dv))
    if backbone == GLA:
        gate = np.log(1 / (1 + np.exp(-rng.standard_normal((B, T, H, Dk))))) / 4
        beta = None
    else:
        gate = -np.log1p(np.exp(rng.standard_normal((B, T, H))))
        beta = 1 / (1 + np.exp(-rng.standard_normal((B, T, H))))
    if lam is None:
        lam = rng.uniform(0.05, 0.95, (B, T, H))
    else:
        lam = np.full((B, T, H), float(lam))
    return dict(q=q, k=k, v=v, gate=gate, beta=beta, lam=lam)


def brute_sigma(kb_hist, centered=True):
    """Sample covariance of the key history by the two-pass formula
    (divide by t, App. A.2): mean first, then the centred outer products."""
    t = kb_hist.shape[0]
    if not centered:
        return kb_hist.T @ kb_hist / t
    mu = kb_hist.mean(axis=0)
    d = kb_hist - mu
    return d.T @ d / t


def brute_qclean(q, k, lam, centered=True, Ckeys0=None):
    """Eq. clean from the explicit key history at every position, one (b,h)."""
    T = q.shape[0]
    qb, kb = unit(q), unit(k)
    out = np.zeros_like(qb)
    for t in range(T):
        Sig = brute_sigma(kb[: t + 1], centered)
        out[t] = qb[t] - lam[t] * Sig @ qb[t]
    return out


# ---------------------------------------------------------------- Sigma_t, Eq. clean

@pytest.mark.parametrize("centered", [True, False])
def test_qclean_matches_explicit_history_covariance(oracle_mod, centered):
    rng = np.random.default_rng(0)
    P = rand_problem(rng, 2, 23, 2, 7, 5)
    res = oracle_mod.forward(GLA, P["q"], P["k"], P["v"], P["gate"], P["lam"],
                             centered=centered, want_qclean=True)
    for b in range(2):
        for h in range(2):
            ref = brute_qclean(P["q"][b, :, h], P["k"][b, :, h], P["lam"][b, :, h], centered)
            np.testing.assert_allclose(res["qclean"][b, :, h], ref, rtol=0, atol=1e-12)


def test_hessian_of_log_partition_is_sigma(oracle_mod):
    """Eq. hess / App. A.2: the Hessian of A_t(q) = log sum_m exp(k_m^T q) at
    q = 0 equals Sigma_t.  Sigma_t e_i is read back from the oracle as
    (e_i - q_clean)/lambda with the query e_i at the last position."""
    rng = np.random.default_rng(1)
    d, t = 8, 10
    keys = unit(rng.standard_normal((t, d)))
    B = d
    q = rng.standard_normal((B, t, 1, d))
    for i in range(d):
        q[i, -1, 0] = np.eye(d)[i]
    k = np.broadcast_to(keys[None, :, None, :], (B, t, 1, d)).copy()
    v = rng.standard_normal((B, t, 1, 3))
    gate = np.zeros((B, t, 1, d))
    lam = np.full((B, t, 1), 0.5)
    res = oracle_mod.forward(GLA, q, k, v, gate, lam, want_qclean=True)
    Sig = np.stack([(np.eye(d)[i] - res["qclean"][i, -1, 0]) / 0.5 for i in range(d)], axis=1)

    def A(x):
        s = keys @ x
        m = s.max()
        return m + np.log(np.exp(s - m).sum())

    h = 1e-3
    Hfd = np.zeros((d, d))
    E = np.eye(d) * h
    for i in range(d):
        for j in range(d):
            Hfd[i, j] = (A(E[i] + E[j]) - A(E[i] - E[j]) - A(-E[i] + E[j]) + A(-E[i] - E[j])) / (4 * h * h)
    np.testing.assert_allclose(Sig, Hfd, atol=1e-6)
    np.testing.assert_allclose(Sig, Sig.T, atol=1e-13)


def test_alternating_pm_u_closed_form(oracle_mod):
    """Keys alternate +u, -u: at even t mu = 0 and Sigma = u u^T, so
    q_clean = qbar - lambda (u.qbar) u; at odd t mu = u/t and
    Sigma = (1 - 1/t^2) u u^T."""
    rng = np.random.default_rng(2)
    d, T = 6, 12
    u = unit(rng.standard_normal(d))
    k = np.stack([u if t % 2 == 0 else -u for t in range(T)])[None, :, None, :]
    q = rng.standard_normal((1, T, 1, d))
    lam = rng.uniform(0.1, 0.9, (1, T, 1))
    res = oracle_mod.forward(GLA, q, k, rng.standard_normal((1, T, 1, 2)),
                             np.zeros((1, T, 1, d)), lam, want_qclean=True)
    for t in range(1, T + 1):
        qb = unit(q[0, t - 1, 0])
        rho = 1.0 if t % 2 == 0 else 1.0 - 1.0 / t ** 2
        ref = qb - lam[0, t - 1, 0] * rho * (u @ qb) * u
        np.testing.assert_allclose(res["qclean"][0, t - 1, 0], ref, atol=1e-14)


def test_cycled_orthonormal_basis_closed_form(oracle_mod):
    """Keys cycle through an orthonormal basis {b_i}: at t = m d,
    Cbar = I/d and mu = (1/d) sum_i b_i, so Sigma = I/d - mu mu^T."""
    rng = np.random.default_rng(3)
    d, m = 5, 3
    Qb, _ = np.linalg.qr(rng.standard_normal((d, d)))
    basis = Qb.T
    T = m * d
    k = np.stack([basis[t % d] for t in range(T)])[None, :, None, :]
    q = rng.standard_normal((1, T, 1, d))
    lam = np.full((1, T, 1), 0.7)
    res = oracle_mod.forward(GLA, q, k, rng.standard_normal((1, T, 1, 2)),
                             np.zeros((1, T, 1, d)), lam, want_qclean=True)
    mu = basis.sum(axis=0) / d
    Sig = np.eye(d) / d - np.outer(mu, mu)
    for mm in range(1, m + 1):
        t = mm * d
        qb = unit(q[0, t - 1, 0])
        np.testing.assert_allclose(res["qclean"][0, t - 1, 0], qb - 0.7 * Sig @ qb, atol=1e-14)


def test_first_token_is_identity(oracle_mod):
    """t = 1: Sigma_1 = 0, so q_clean = qbar exactly (any lambda)."""
    rng = np.random.default_rng(4)
    P = rand_problem(rng, 3, 1, 2, 9, 4, lam=0.99)
    res = oracle_mod.forward(GLA, P["q"], P["k"], P["v"], P["gate"], P["lam"], want_qclean=True)
    np.testing.assert_allclose(res["qclean"], unit(P["q"]), atol=1e-15)


def test_spectrum_bound_and_eigen_shrink(oracle_mod):
    """App. A.3 / App. G: unit keys give ||Sigma|| <= ||Cbar|| <= 1, so
    I - lambda Sigma has spectrum in [1 - lambda, 1]; each eigendirection of
    Sigma is shrunk by exactly 1 - lambda sigma_i."""
    rng = np.random.default_rng(5)
    T, d = 40, 6
    P = rand_problem(rng, 1, T, 1, d, 3)
    # a dominant direction so that some sigma_i are large
    P["k"][0, :, 0] += 3 * rng.standard_normal((T, 1)) * unit(rng.standard_normal(d))
    res = oracle_mod.forward(GLA, P["q"], P["k"], P["v"], P["gate"], P["lam"], want_qclean=True)
    kb = unit(P["k"][0, :, 0])
    for t in range(T):
        qb = unit(P["q"][0, t, 0])
        qc = res["qclean"][0, t, 0]
        lam = P["lam"][0, t, 0]
        assert np.linalg.norm(qc) <= np.linalg.norm(qb) + 1e-12
        assert np.linalg.norm(qc) >= (1 - lam) * np.linalg.norm(qb) - 1e-12
        Sig = brute_sigma(kb[: t + 1])
        w, V = np.linalg.eigh(Sig)
        assert w.min() > -1e-12 and w.max() <= 1 + 1e-12
        np.testing.assert_allclose(V.T @ qc, (1 - lam * w) * (V.T @ qb), atol=1e-12)


def test_score_space_form(oracle_mod):
    """App. A.4: k_j^T q_clean = k_j^T q - (lambda/t) sum_i (k_j.k_i)(k_i.q)
    + lambda (k_j.mu)(mu.q), for every stored key j <= t."""
    rng = np.random.default_rng(6)
    T, d = 17, 8
    P = rand_problem(rng, 1, T, 1, d, 3)
    res = oracle_mod.forward(GLA, P["q"], P["k"], P["v"], P["gate"], P["lam"], want_qclean=True)
    kb = unit(P["k"][0, :, 0])
    for t in range(T):
        qb = unit(P["q"][0, t, 0])
        lam = P["lam"][0, t, 0]
        K = kb[: t + 1]
        mu = K.mean(axis=0)
        for j in range(t + 1):
            three = (K[j] @ qb - lam / (t + 1) * np.sum((K @ K[j]) * (K @ qb))
                     + lam * (K[j] @ mu) * (mu @ qb))
            assert abs(K[j] @ res["qclean"][0, t, 0] - three) < 1e-12


def test_retrieval_margin_shift(oracle_mod):
    """App. H, Eq. margin_shift: with Sigma = rho u u^T exactly (keys +u, -u,
    rho = 1 at even t), the CCQ margin between a target (alignment alpha) and a
    distractor (alignment beta) grows by lambda rho (beta - alpha)(u^T q)."""
    rng = np.random.default_rng(7)
    d, T = 8, 10
    u = unit(rng.standard_normal(d))
    k = np.stack([u if t % 2 == 0 else -u for t in range(T)])[None, :, None, :]
    q = rng.standard_normal((1, T, 1, d))
    lam = 0.6
    res = oracle_mod.forward(GLA, q, k, np.zeros((1, T, 1, 2)), np.zeros((1, T, 1, d)),
                             np.full((1, T, 1), lam), want_qclean=True)
    qb = unit(q[0, -1, 0])
    qc = res["qclean"][0, -1, 0]
    k_star = unit(rng.standard_normal(d))
    k_d = unit(u + 0.3 * rng.standard_normal(d))
    a, b = k_star @ u, k_d @ u
    shift = (k_star @ qc - k_d @ qc) - (k_star @ qb - k_d @ qb)
    assert abs(shift - lam * 1.0 * (b - a) * (u @ qb)) < 1e-13


# ---------------------------------------------------------------- backbones

def brute_gla(q, k, v, gate, lam, S0=None, scale=1.0, centered=True):
    """GLA read from the explicit history: o_t = scale * sum_j v_j (kbar_j *
    prod_{j<s<=t} alpha_s)^T q_clean_t, plus the decayed initial state."""
    T, Dk = q.shape
    qc = brute_qclean(q, k, lam, centered)
    kb = unit(k)
    o = np.zeros((T, v.shape[1]))
    for t in range(T):
        for j in range(t + 1):
            dec = np.exp(gate[j + 1: t + 1].sum(axis=0))
            o[t] += (kb[j] * dec) @ qc[t] * v[j]
        if S0 is not None:
            o[t] += (qc[t] * np.exp(gate[: t + 1].sum(axis=0))) @ S0
    return scale * o


def brute_gdn(q, k, v, g, beta, lam, S0=None, scale=1.0):
    """Gated DeltaNet from explicit transition-matrix products: with
    A_s = alpha_s (I - beta_s k_s k_s^T) acting on S^T, the state after t
    tokens is sum_j (A_t ... A_{j+1}) beta_j k_j v_j^T + (A_t ... A_1) S0."""
    T, Dk = q.shape
    qc = brute_qclean(q, k, lam)
    kb = unit(k)
    A = [np.exp(g[s]) * (np.eye(Dk) - beta[s] * np.outer(kb[s], kb[s])) for s in range(T)]
    o = np.zeros((T, v.shape[1]))
    for t in range(T):
        H = np.zeros((Dk, v.shape[1]))
        for j in range(t + 1):
            P = np.eye(Dk)
            for s in range(j + 1, t + 1):
                P = A[s] @ P
            H += P @ np.outer(beta[j] * kb[j], v[j])
        if S0 is not None:
            P = np.eye(Dk)
            for s in range(t + 1):
                P = A[s] @ P
            H += P @ S0
        o[t] = scale * H.T @ qc[t]
    return o


@pytest.mark.parametrize("with_state", [False, True])
def test_gla_matches_explicit_history(oracle_mod, with_state):
    rng = np.random.default_rng(8)
    B, T, H, Dk, Dv = 1, 19, 2, 6, 5
    P = rand_problem(rng, B, T, H, Dk, Dv, GLA)
    S0 = rng.standard_normal((B, H, Dk, Dv)) if with_state else None
    res = oracle_mod.forward(GLA, P["q"], P["k"], P["v"], P["gate"], P["lam"], S0=S0, scale=0.7)
    for h in range(H):
        ref = brute_gla(P["q"][0, :, h], P["k"][0, :, h], P["v"][0, :, h], P["gate"][0, :, h],
                        P["lam"][0, :, h], None if S0 is None else S0[0, h], 0.7)
        np.testing.assert_allclose(res["o"][0, :, h], ref, atol=1e-12)


def test_vanilla_linear_attention_reduction(oracle_mod):
    """All forget gates 1 (log 0) and lambda = 0: o_t = sum_{j<=t} v_j (kbar_j.qbar_t)
    (Sec. 2.2, Eq. prelim_linattn)."""
    rng = np.random.default_rng(9)
    T, d = 15, 4
    P = rand_problem(rng, 1, T, 1, d, 3, lam=0.0)
    res = oracle_mod.forward(GLA, P["q"], P["k"], P["v"], np.zeros_like(P["gate"]), P["lam"], scale=1.0)
    qb, kb, v = unit(P["q"][0, :, 0]), unit(P["k"][0, :, 0]), P["v"][0, :, 0]
    scores = np.tril(qb @ kb.T)
    np.testing.assert_allclose(res["o"][0, :, 0], scores @ v, atol=1e-13)


@pytest.mark.parametrize("with_state", [False, True])
def test_gdn_matches_transition_products(oracle_mod, with_state):
    rng = np.random.default_rng(10)
    B, T, H, Dk, Dv = 1, 14, 2, 5, 4
    P = rand_problem(rng, B, T, H, Dk, Dv, GDN)
    S0 = rng.standard_normal((B, H, Dk, Dv)) if with_state else None
    res = oracle_mod.forward(GDN, P["q"], P["k"], P["v"], P["gate"], P["lam"], beta=P["beta"],
                             S0=S0, scale=0.9)
    for h in range(H):
        ref = brute_gdn(P["q"][0, :, h], P["k"][0, :, h], P["v"][0, :, h], P["gate"][0, :, h],
                        P["beta"][0, :, h], P["lam"][0, :, h], None if S0 is None else S0[0, h], 0.9)
        np.testing.assert_allclose(res["o"][0, :, h], ref, atol=1e-12)


def test_delta_rule_overwrites_value(oracle_mod):
    """Delta rule semantics: with alpha = 1 and beta = 1, writing (k, v1) and
    then (k, v2) leaves S k = v2 exactly; with lambda = 0 the read at the
    second token returns v2 (for q = k)."""
    rng = np.random.default_rng(11)
    d = 6
    kvec = unit(rng.standard_normal(d))
    q = np.stack([kvec, kvec])[None, :, None, :]
    k = q.copy()
    v = rng.standard_normal((1, 2, 1, 3))
    res = oracle_mod.forward(GDN, q, k, v, np.zeros((1, 2, 1)), np.zeros((1, 2, 1)),
                             beta=np.ones((1, 2, 1)), scale=1.0)
    np.testing.assert_allclose(res["o"][0, 1, 0], v[0, 1, 0], atol=1e-14)
    np.testing.assert_allclose(res["S"][0, 0].T @ kvec, v[0, 1, 0], atol=1e-14)


def test_lambda_zero_is_plain_backbone_and_correction_is_linear(oracle_mod):
    """Eq. read: o = S q - lambda S Sigma q, so o(lambda) - o(0) is linear in lambda."""
    rng = np.random.default_rng(12)
    P = rand_problem(rng, 1, 11, 1, 5, 4, GDN)
    outs = []
    for lam in (0.0, 0.3, 0.6):
        outs.append(oracle_mod.forward(GDN, P["q"], P["k"], P["v"], P["gate"],
                                       np.full_like(P["lam"], lam), beta=P["beta"])["o"])
    np.testing.assert_allclose(outs[2] - outs[0], 2 * (outs[1] - outs[0]), atol=1e-13)
    ref0 = brute_gdn(P["q"][0, :, 0], P["k"][0, :, 0], P["v"][0, :, 0], P["gate"][0, :, 0],
                     P["beta"][0, :, 0], np.zeros(11), None, 5 ** -0.5)
    np.testing.assert_allclose(outs[0][0, :, 0], ref0, atol=1e-12)


# ---------------------------------------------------------------- forms of the same computation

@pytest.mark.parametrize("backbone", [GLA, GDN])
@pytest.mark.parametrize("chunk", [1, 16, 64])
def test_chunkwise_equals_recurrent(oracle_mod, backbone, chunk):
    """Algorithm 1 (chunkwise, App. B) equals the token recurrence, including a
    ragged tail (T = 65) and a resumed state (t0 > 0, non-zero S, C, m)."""
    rng = np.random.default_rng(13)
    B, T, H, Dk, Dv = 2, 65, 2, 8, 6
    P = rand_problem(rng, B, T, H, Dk, Dv, backbone)
    prev = rand_problem(rng, B, 30, H, Dk, Dv, backbone)
    st = oracle_mod.forward(backbone, prev["q"], prev["k"], prev["v"], prev["gate"], prev["lam"],
                            beta=prev["beta"])
    kw = dict(beta=P["beta"], S0=st["S"], C0=st["C"], m0=st["m"], t0=st["t"])
    rec = oracle_mod.forward(backbone, P["q"], P["k"], P["v"], P["gate"], P["lam"], **kw)
    chk = oracle_mod.forward(backbone, P["q"], P["k"], P["v"], P["gate"], P["lam"], chunk=chunk, **kw)
    for name in ("o", "S", "C", "m"):
        np.testing.assert_allclose(chk[name], rec[name], rtol=1e-10,
                                   atol=1e-10 * np.abs(rec[name]).max())
    np.testing.assert_array_equal(chk["t"], rec["t"])


def test_algorithm2_running_mean_form(oracle_mod):
    """Algorithm 2 keeps the running means Cbar_t = Cbar_{t-1} + (kk^T - Cbar_{t-1})/t
    and mu_t likewise; the oracle keeps sums.  Both give the same Sigma_t and the
    same q_clean, and the final sums equal t * (Cbar, mu)."""
    rng = np.random.default_rng(14)
    T, d = 25, 6
    P = rand_problem(rng, 1, T, 1, d, 3)
    res = oracle_mod.forward(GLA, P["q"], P["k"], P["v"], P["gate"], P["lam"], want_qclean=True)
    Cbar = np.zeros((d, d))
    mu = np.zeros(d)
    for t in range(1, T + 1):
        kb = unit(P["k"][0, t - 1, 0])
        qb = unit(P["q"][0, t - 1, 0])
        Cbar = Cbar + (np.outer(kb, kb) - Cbar) / t
        mu = mu + (kb - mu) / t
        Sig = Cbar - np.outer(mu, mu)
        np.testing.assert_allclose(res["qclean"][0, t - 1, 0], qb - P["lam"][0, t - 1, 0] * Sig @ qb,
                                   atol=1e-13)
    np.testing.assert_allclose(res["C"][0, 0], T * Cbar, atol=1e-12)
    np.testing.assert_allclose(res["m"][0, 0], T * mu, atol=1e-12)
    assert res["t"][0] == T


@pytest.mark.parametrize("backbone", [GLA, GDN])
def test_split_call_resumes_exactly(oracle_mod, backbone):
    """Passing the final (S, C, m, t) of a first call as the initial state of a
    second call equals one call over the whole sequence."""
    rng = np.random.default_rng(15)
    P = rand_problem(rng, 2, 40, 2, 6, 5, backbone)
    full = oracle_mod.forward(backbone, P["q"], P["k"], P["v"], P["gate"], P["lam"], beta=P["beta"])
    cut = 17
    sl = lambda x, a, b: None if x is None else x[:, a:b]  # noqa: E731
    a = oracle_mod.forward(backbone, *(sl(P[n], 0, cut) for n in ("q", "k", "v", "gate", "lam")),
                           beta=sl(P["beta"], 0, cut))
    b = oracle_mod.forward(backbone, *(sl(P[n], cut, 40) for n in ("q", "k", "v", "gate", "lam")),
                           beta=sl(P["beta"], cut, 40), S0=a["S"], C0=a["C"], m0=a["m"], t0=a["t"])
    np.testing.assert_allclose(np.concatenate([a["o"], b["o"]], axis=1), full["o"], atol=1e-12)
    for n in ("S", "C", "m"):
        np.testing.assert_allclose(b[n], full[n], atol=1e-12)
    np.testing.assert_array_equal(b["t"], full["t"])


@pytest.mark.parametrize("backbone", [GLA, GDN])
def test_decode_step_is_one_token_forward(oracle_mod, backbone):
    rng = np.random.default_rng(16)
    P = rand_problem(rng, 3, 9, 2, 6, 5, backbone)
    full = oracle_mod.forward(backbone, P["q"], P["k"], P["v"], P["gate"], P["lam"], beta=P["beta"])
    sl = lambda x, a, b: None if x is None else x[:, a:b]  # noqa: E731
    pre = oracle_mod.forward(backbone, *(sl(P[n], 0, 8) for n in ("q", "k", "v", "gate", "lam")),
                             beta=sl(P["beta"], 0, 8))
    tok = {n: (None if P[n] is None else P[n][:, 8]) for n in P}
    d = oracle_mod.decode_step(backbone, tok["q"], tok["k"], tok["v"], tok["gate"], tok["lam"],
                               pre["S"], pre["C"], pre["m"], pre["t"], beta=tok["beta"])
    np.testing.assert_allclose(d["o"], full["o"][:, 8], atol=1e-13)
    np.testing.assert_allclose(d["S"], full["S"], atol=1e-13)
    np.testing.assert_array_equal(d["t"], full["t"])


def test_thread_count_does_not_change_results(oracle_mod):
    rng = np.random.default_rng(17)
    P = rand_problem(rng, 3, 20, 3, 5, 4)
    a = oracle_mod.forward(GLA, P["q"], P["k"], P["v"], P["gate"], P["lam"], nthreads=1)
    b = oracle_mod.forward(GLA, P["q"], P["k"], P["v"], P["gate"], P["lam"], nthreads=5)
    np.testing.assert_array_equal(a["o"], b["o"])


def test_zero_length_passes_states_through(oracle_mod):
    rng = np.random.default_rng(18)
    S0 = rng.standard_normal((2, 1, 4, 3))
    C0 = rng.standard_normal((2, 1, 4, 4))
    m0 = rng.standard_normal((2, 1, 4))
    z = np.zeros((2, 0, 1, 4))
    res = oracle_mod.forward(GLA, z, z, np.zeros((2, 0, 1, 3)), z, np.zeros((2, 0, 1)),
                             S0=S0, C0=C0, m0=m0, t0=np.array([5, 7]))
    np.testing.assert_array_equal(res["S"], S0)
    np.testing.assert_array_equal(res["C"], C0)
    np.testing.assert_array_equal(res["t"], [5, 7])


def test_zero_norm_rows_stay_finite(oracle_mod):
    """The paper gives no epsilon for the l2 norm; the oracle maps a zero row to zero."""
    q = np.zeros((1, 3, 1, 4))
    k = np.zeros((1, 3, 1, 4))
    k[0, 1, 0, 0] = 1.0
    v = np.ones((1, 3, 1, 2))
    res = oracle_mod.forward(GLA, q, k, v, np.zeros((1, 3, 1, 4)), np.full((1, 3, 1), 0.5))
    assert np.isfinite(res["o"]).all() and np.isfinite(res["S"]).all()
    np.testing.assert_array_equal(res["o"], 0.0)
