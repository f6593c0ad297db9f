"""GPU parity of ccq_gdn_bwd against the oracle's fp64 reverse mode of CCQ-Gated-DeltaNet
(itself pinned by finite differences and by an independent chunkwise adjoint), element by
element.

With fp32 inputs every product runs in fp32 on the CUDA cores, held to the fp32 bar
(max|g - ref| / max|ref| <= 1e-4); with bf16 inputs the per-chunk products run on the tensor
cores with bf16 operands (the forward's precision), held to the bf16 bar (2e-2, the outputs dq,
dk, dv being rounded to bf16).  Every gradient is compared: dq, dk, dv, dg, dbeta, dlambda,
dS0, dC0, dm0."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import GDN, TOL, rel_err, slice_bh, state_to_dev

pytestmark = pytest.mark.gpu
NAMES = ("dq", "dk", "dv", "dg", "dbeta", "dlambda", "dS0", "dC0", "dm0")


@pytest.fixture(autouse=True)
def _status():
    yield
    ccq.device_status()


def _problem(B, T, H, D, *, dtype, seed, lam="trained", keys="structured", prefix=40, state_grads=True):
    P = gen.make_inputs(GDN, B, T, H, D, D, dtype=dtype, seed=seed, lam=lam, keys=keys)
    G = gen.make_backward_inputs(B, T, H, D, D, dtype=dtype, seed=seed + 1, prefix=prefix,
                                 state_grads=state_grads)
    return P, G


def _gpu(P, G, **kw):
    d = lambda x: None if x is None else x.cuda().contiguous()
    st = state_to_dev(G["state"])
    g = ccq.gdn_bwd(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["beta"]), d(P["lam"]),
                    d(G["dout"]), st, dST=d(G["dST"]), dCT=d(G["dCT"]), dmT=d(G["dmT"]), **kw)
    torch.cuda.synchronize()
    return g


def _ref(P, G, **kw):
    st = G["state"] or {}
    f32 = lambda x: None if x is None else x.float()  # the library's states are fp32
    return oracle.gdn_backward(P["q"], P["k"], P["v"], P["gate"], P["beta"], P["lam"], G["dout"],
                               S0=f32(st.get("S")), C0=f32(st.get("C")), m0=f32(st.get("m")),
                               t0=st.get("t"), dST=G["dST"], dCT=G["dCT"], dmT=G["dmT"], **kw)


def _compare(g, ref, tol, what):
    errs = {n: rel_err(g[n], ref["dlam" if n == "dlambda" else n]) for n in NAMES}
    bad = {k: v for k, v in errs.items() if not v <= tol}
    assert not bad, f"{what}: relative errors above {tol}: {errs}"
    return errs


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("lam", ["init", "trained", "high"])
def test_bwd_fp32_ragged_resumed(D, lam):
    """fp32 inputs, T = 200 (three chunks and an 8-token tail), resumed from a 40-token state,
    with final-state gradients."""
    P, G = _problem(2, 200, 3, D, dtype=torch.float32, seed=31, lam=lam)
    _compare(_gpu(P, G), _ref(P, G), TOL[torch.float32], f"D={D} {lam}")


@pytest.mark.parametrize("keys", ["iso", "structured", "lowrank"])
def test_bwd_bf16(keys):
    """bf16 inputs, D = 128, T = 130, from the zero state."""
    P, G = _problem(2, 130, 2, 128, dtype=torch.bfloat16, seed=32, keys=keys, prefix=0)
    _compare(_gpu(P, G), _ref(P, G), TOL[torch.bfloat16], keys)


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("lam", ["init", "high"])
def test_bwd_bf16_ragged_resumed(D, lam):
    """bf16 inputs (tensor-core products), T = 200 (three chunks and an 8-token tail), resumed
    from a 40-token state, with final-state gradients."""
    P, G = _problem(2, 200, 3, D, dtype=torch.bfloat16, seed=51, lam=lam)
    _compare(_gpu(P, G), _ref(P, G), TOL[torch.bfloat16], f"bf16 D={D} {lam}")


@pytest.mark.parametrize("T", [1, 63, 65])
def test_bwd_bf16_lengths(T):
    """bf16 inputs: a single token, one short chunk, and a chunk plus one token."""
    P, G = _problem(1, T, 2, 128, dtype=torch.bfloat16, seed=52 + T, prefix=40 if T == 1 else 0)
    _compare(_gpu(P, G), _ref(P, G), TOL[torch.bfloat16], f"bf16 T={T}")


@pytest.mark.parametrize("opts", [dict(centered=False), dict(l2norm=False)])
def test_bwd_bf16_variants(opts):
    """bf16 inputs with the uncentred covariance (App. D) and with un-normalised q, k."""
    P, G = _problem(1, 150, 2, 128, dtype=torch.bfloat16, seed=56)
    _compare(_gpu(P, G, **opts), _ref(P, G, **opts), TOL[torch.bfloat16], f"bf16 {opts}")


@pytest.mark.parametrize("T", [1, 63, 64, 65])
def test_bwd_lengths(T):
    P, G = _problem(1, T, 2, 64, dtype=torch.float32, seed=33 + T, prefix=40 if T == 1 else 0,
                    state_grads=T != 64)
    _compare(_gpu(P, G), _ref(P, G), TOL[torch.float32], f"T={T}")


@pytest.mark.parametrize("opts", [dict(centered=False), dict(l2norm=False)])
def test_bwd_variants(opts):
    """The uncentred covariance (App. D) and un-normalised q, k."""
    P, G = _problem(1, 150, 2, 64, dtype=torch.float32, seed=41)
    _compare(_gpu(P, G, **opts), _ref(P, G, **opts), TOL[torch.float32], str(opts))


def test_bwd_zero_length():
    """T = 0: the initial-state gradients are the final-state ones."""
    P, G = _problem(1, 0, 2, 64, dtype=torch.float32, seed=42, prefix=0)
    g = _gpu(P, G)
    for n, r in (("dS0", "dST"), ("dC0", "dCT"), ("dm0", "dmT")):
        assert torch.equal(g[n].cpu(), G[r]), n


def test_bwd_full_size_sampled():
    """B=4, H=16, T=4096, bf16 (the training step's shape): every (batch, head) pair is
    computed on the GPU; two of them are compared with the oracle run on that pair alone."""
    P, G = _problem(4, 4096, 16, 128, dtype=torch.bfloat16, seed=43, prefix=0, state_grads=False)
    g = _gpu(P, G)
    for b, h in ((0, 0), (3, 15)):
        Ps, Gs = slice_bh(P, b, h), {**G, "dout": G["dout"][b:b + 1, :, h:h + 1].contiguous()}
        ref = _ref(Ps, Gs)
        part = {n: (x[b:b + 1, h:h + 1] if n in ("dS0", "dC0", "dm0") else x[b:b + 1, :, h:h + 1])
                for n, x in g.items()}
        _compare(part, ref, TOL[torch.bfloat16], f"b={b} h={h}")
