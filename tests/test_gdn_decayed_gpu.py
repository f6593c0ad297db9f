"""GPU parity of ccq_gdn_fwd_decayed (CCQ-Gated-DeltaNet with the decay-aligned covariance)
and ccq_gdn_fwd_spectral (the resolvent and exponential contractions) against the oracle's
gdn_forward_decayed and gdn_forward_spectral, element by element: o, S_T, C_T, m_T, n_T.
fp32 inputs to 1e-4, bf16 inputs to 2e-2."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import GDN, TOL, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _status():
    yield
    ccq.device_status()


def _state(B, H, D, seed):
    g = torch.Generator().manual_seed(seed)
    hist = torch.randn(B, H, 9, D, generator=g)
    hist = hist / hist.norm(dim=-1, keepdim=True)
    w = torch.exp(-0.3 * torch.arange(9, dtype=torch.float32).flip(0))
    return {"S": torch.randn(B, H, D, D, generator=g) / D,
            "C": torch.einsum("t,bhti,bhtj->bhij", w, hist, hist),
            "m": torch.einsum("t,bhti->bhi", w, hist), "n": torch.full((B, H), float(w.sum()))}


def _run(P, st, **kw):
    d = lambda x: None if x is None else x.cuda().contiguous()  # noqa: E731
    st = st or {}
    o, fs = ccq.gdn_fwd_decayed(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["beta"]), d(P["lam"]),
                                S0=d(st.get("S")), C0=d(st.get("C")), m0=d(st.get("m")), n0=d(st.get("n")),
                                **kw)
    torch.cuda.synchronize()
    ref = oracle.gdn_forward_decayed(P["q"], P["k"], P["v"], P["gate"], P["beta"], P["lam"], S0=st.get("S"),
                                     C0=st.get("C"), m0=st.get("m"), n0=st.get("n"),
                                     l2norm=kw.get("l2norm", True), centered=kw.get("centered", True))
    return {"o": rel_err(o, ref["o"]), "S": rel_err(fs["S"], ref["S"]), "C": rel_err(fs["C"], ref["C"]),
            "m": rel_err(fs["m"], ref["m"]), "n": rel_err(fs["n"], ref["n"])}


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("lam", ["trained", "high"])
def test_decayed_fp32_ragged_resumed(D, lam):
    P = gen.make_inputs(GDN, 2, 200, 3, D, D, dtype=torch.float32, seed=51, lam=lam, keys="structured")
    errs = _run(P, _state(2, 3, D, 52))
    assert max(errs.values()) <= TOL[torch.float32], errs


@pytest.mark.parametrize("opts", [dict(centered=False), dict(l2norm=False)])
def test_decayed_variants(opts):
    P = gen.make_inputs(GDN, 1, 130, 2, 64, 64, dtype=torch.float32, seed=53, lam="trained")
    errs = _run(P, None, **opts)
    assert max(errs.values()) <= TOL[torch.float32], errs


def test_decayed_bf16_4k():
    """bf16, B=1, H=4, T=4096, d=128 (64 chunks): every output element against the oracle."""
    P = gen.make_inputs(GDN, 1, 4096, 4, 128, 128, dtype=torch.bfloat16, seed=54, lam="trained",
                        keys="structured")
    errs = _run(P, None)
    assert max(errs.values()) <= TOL[torch.bfloat16], errs


def test_decayed_zero_length():
    P = gen.make_inputs(GDN, 1, 0, 2, 64, 64, dtype=torch.float32, seed=55)
    st = _state(1, 2, 64, 56)
    d = lambda x: x.cuda().contiguous()  # noqa: E731
    o, fs = ccq.gdn_fwd_decayed(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["beta"]), d(P["lam"]),
                                S0=d(st["S"]), C0=d(st["C"]), m0=d(st["m"]), n0=d(st["n"]))
    for n in ("S", "C", "m", "n"):
        assert torch.equal(fs[n].cpu(), st[n]), n


@pytest.mark.parametrize("contraction", ["resolvent", "exponential", "linear"])
@pytest.mark.parametrize("decayed", [True, False])
def test_spectral_contractions(contraction, decayed):
    """ccq_gdn_fwd_spectral against oracle.gdn_forward_spectral (numpy solve / expm per token);
    undecayed linear is the paper's CCQ-Gated-DeltaNet."""
    P = gen.make_inputs(GDN, 1, 150, 2, 64, 64, dtype=torch.float32, seed=57, lam="high", keys="structured")
    d = lambda x: x.cuda().contiguous()  # noqa: E731
    o, fs = ccq.gdn_fwd_decayed(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["beta"]), d(P["lam"]),
                                contraction=contraction, decayed=decayed)
    torch.cuda.synchronize()
    ref = oracle.gdn_forward_spectral(P["q"], P["k"], P["v"], P["gate"], P["beta"], P["lam"],
                                      contraction={"linear": oracle.LINEAR, "resolvent": oracle.RESOLVENT,
                                                   "exponential": oracle.EXPONENTIAL}[contraction],
                                      decayed=decayed)
    errs = {n: rel_err(x, ref[n]) for n, x in (("o", o), ("S", fs["S"]), ("C", fs["C"]), ("m", fs["m"]),
                                               ("n", fs["n"]))}
    assert max(errs.values()) <= TOL[torch.float32], errs
