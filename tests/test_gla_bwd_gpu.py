"""GPU parity of ccq_gla_bwd against the oracle's fp64 reverse mode (itself
pinned by finite differences), element by element.

Every gradient (dq, dk, dv, dgk, dlambda, dS0, dC0, dm0) is held to
max|g - ref| / max|ref| <= 2e-2, the bf16 bound of the forward: the backward
computes in bf16 operands with fp32 accumulation like the forward, and its
inputs (dout) are bf16."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import GLA, TOL, rel_err, slice_bh, state_to_dev

pytestmark = pytest.mark.gpu
TOLB = TOL[torch.bfloat16]
NAMES = ("dq", "dk", "dv", "dgk", "dlambda", "dS0", "dC0", "dm0")


@pytest.fixture(autouse=True)
def _status():
    yield
    ccq.device_status()


def _problem(B, T, H, *, seed, lam="trained", keys="structured", prefix=40, state_grads=True,
             gate_dtype=None):
    P = gen.make_inputs(GLA, B, T, H, 128, 128, dtype=torch.bfloat16, seed=seed, lam=lam, keys=keys,
                        gate_dtype=gate_dtype)
    G = gen.make_backward_inputs(B, T, H, 128, 128, seed=seed + 1, prefix=prefix,
                                 state_grads=state_grads)
    return P, G


def _gpu(P, G, ckpt=None, **kw):
    d = lambda x: None if x is None else x.cuda().contiguous()
    st = state_to_dev(G["state"])
    g = ccq.gla_bwd(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["lam"]), d(G["dout"]), st,
                    dST=d(G["dST"]), dCT=d(G["dCT"]), dmT=d(G["dmT"]), ckpt=ckpt, **kw)
    torch.cuda.synchronize()
    return g


def _ref(P, G, **kw):
    st = G["state"] or {}
    f32 = lambda x: None if x is None else x.float()  # the library's states are fp32
    return oracle.gla_backward(P["q"], P["k"], P["v"], P["gate"], P["lam"], G["dout"],
                               S0=f32(st.get("S")), C0=f32(st.get("C")), m0=f32(st.get("m")),
                               t0=st.get("t"), dST=G["dST"], dCT=G["dCT"], dmT=G["dmT"], **kw)


def _compare(g, ref, what, tol=TOLB):
    errs = {}
    for n in NAMES:
        r = ref["dlam" if n == "dlambda" else n]
        errs[n] = rel_err(g[n], r)
    bad = {k: v for k, v in errs.items() if not v <= tol}
    assert not bad, f"{what}: relative errors above {tol}: {errs}"
    return errs


@pytest.mark.parametrize("lam", ["init", "trained", "high"])
@pytest.mark.parametrize("keys", ["iso", "structured"])
def test_bwd_ragged_resumed(lam, keys):
    """T = 200 (three chunks and an 8-token tail), resumed from a 40-token
    state, with final-state gradients."""
    P, G = _problem(2, 200, 3, seed=21, lam=lam, keys=keys)
    _compare(_gpu(P, G, seq_split=1), _ref(P, G), f"{lam} {keys}")


@pytest.mark.parametrize("T", [1, 37, 64, 65, 130])
def test_bwd_lengths(T):
    """Short and boundary lengths without state gradients, from the zero state
    (T = 1 resumes from a 40-token state: from the zero state its dgk and
    dlambda vanish exactly, since S_0 = 0 and Sigma_1 = 0)."""
    P, G = _problem(1, T, 2, seed=22 + T, prefix=40 if T == 1 else 0, state_grads=False)
    _compare(_gpu(P, G, seq_split=1), _ref(P, G), f"T={T}")


def test_bwd_uncentred_and_unnormalised():
    P, G = _problem(1, 150, 2, seed=23, lam="high")
    _compare(_gpu(P, G, centered=False, seq_split=1), _ref(P, G, centered=False), "uncentred")
    # without the in-kernel l2 norm the inputs must already be reasonable: unit rows
    P2 = dict(P, q=torch.nn.functional.normalize(P["q"].float(), dim=-1).to(torch.bfloat16))
    _compare(_gpu(P2, G, l2norm=False, seq_split=1), _ref(P2, G, l2norm=False), "no l2norm")


def test_bwd_fp32_gates():
    P, G = _problem(1, 130, 2, seed=24, gate_dtype=torch.float32)
    g = _gpu(P, G, seq_split=1)
    assert g["dgk"].dtype == torch.float32
    _compare(g, _ref(P, G), "fp32 gates")


def test_bwd_correction_isolated():
    """The CCQ part of dq alone: dq(lambda) - dq(0) against the oracle's
    difference (lambda = 0.9, low-rank keys so that the term is large).  The
    lambda-dependent part of dk is a few percent of dk here, below what two
    bf16 gradients can resolve when subtracted; the full dk comparisons cover it."""
    P, G = _problem(1, 192, 2, seed=25, lam="high", keys="lowrank")
    P0 = dict(P, lam=torch.zeros_like(P["lam"]))
    g1, g0 = _gpu(P, G, seq_split=1), _gpu(P0, G, seq_split=1)
    r1, r0 = _ref(P, G), _ref(P0, G)
    d = g1["dq"].double().cpu().numpy() - g0["dq"].double().cpu().numpy()
    dr = r1["dq"] - r0["dq"]
    assert np.abs(dr).max() > 0.05 * np.abs(r1["dq"]).max()
    # bf16 outputs carry half an ulp each (2^-9 of their magnitude)
    bound = TOLB + 2 * 2.0 ** -9 * np.abs(r1["dq"]).max() / np.abs(dr).max()
    assert rel_err(d, dr) <= bound


def test_bwd_saved_checkpoints_match_recompute():
    """ccq_gla_fwd_save's checkpoints give the same gradients, bit for bit, as
    the recompute inside ccq_gla_bwd; the saving forward's o is the plain one."""
    P, G = _problem(2, 250, 2, seed=26)
    d = lambda x: x.cuda().contiguous()
    st = state_to_dev(G["state"])
    o1, _ = ccq.gla_fwd(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["lam"]), st, seq_split=1)
    o2, _, ck = ccq.gla_fwd_save(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["lam"]), st,
                                 seq_split=1)
    assert torch.equal(o1, o2)
    ga = _gpu(P, G, ckpt=ck, seq_split=1)
    gb = _gpu(P, G, seq_split=1)
    for n in NAMES:
        assert torch.equal(ga[n], gb[n]), n


@pytest.mark.parametrize("split", [2, 3])
def test_bwd_from_segmented_forward(split):
    """Checkpoints written by the segment-parallel forward."""
    P, G = _problem(1, 640, 2, seed=27)
    _compare(_gpu(P, G, seq_split=split), _ref(P, G), f"split {split}")


def test_bwd_no_tokens_passes_state_gradients():
    G = gen.make_backward_inputs(2, 0, 3, 128, 128, seed=28)
    z = torch.zeros(2, 0, 3, 128, dtype=torch.bfloat16, device="cuda")
    lam = torch.zeros(2, 0, 3, device="cuda")
    g = ccq.gla_bwd(z, z, z, z, lam, z, dST=G["dST"].cuda(), dCT=G["dCT"].cuda(), dmT=G["dmT"].cuda())
    torch.cuda.synchronize()
    assert torch.equal(g["dS0"].cpu(), G["dST"]) and torch.equal(g["dC0"].cpu(), G["dCT"])
    assert torch.equal(g["dm0"].cpu(), G["dmT"])


def test_bwd_full_size_sampled():
    """The fwd+bwd workload (B=4, H=16, T=4096, bf16) in the benchmark's launch
    configuration (checkpoints from ccq_gla_fwd_save with the default split);
    the oracle computes a sample of (sequence, head) pairs, each independent."""
    w = gen.WORKLOADS["gla_bf16_4k_fwdbwd"]
    B, T, H = w["B"], w["T"], w["H"]
    P = gen.make_inputs(GLA, B, T, H, 128, 128, dtype=torch.bfloat16, seed=w["seed"], lam="trained")
    G = gen.make_backward_inputs(B, T, H, 128, 128, seed=w["seed"] + 1, state_grads=False)
    d = lambda x: x.cuda().contiguous()
    _, _, ck = ccq.gla_fwd_save(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["lam"]))
    g = _gpu(P, G, ckpt=ck)
    for (b, h) in [(0, 0), (1, 7), (3, 15)]:
        Ps = slice_bh(P, b, h)
        Gs = dict(G, dout=G["dout"][b:b + 1, :, h:h + 1].contiguous())
        ref = _ref(Ps, Gs)
        gs = {n: (g[n][b:b + 1, :, h:h + 1] if g[n].dim() in (3, 4) and g[n].shape[1] == T
                  else g[n][b:b + 1, h:h + 1]) for n in NAMES}
        _compare(gs, ref, f"b={b} h={h}")


@pytest.mark.parametrize("split", [1, 2])
def test_bwd_from_wide_forward_checkpoints(split):
    """Checkpoints written by the two-reference forward (algo "wide") carry the same tile
    images as the default kernel's, so the backward reads either."""
    P, G = _problem(1, 300, 2, seed=29)
    d = lambda x: x.cuda().contiguous()  # noqa: E731
    st = state_to_dev(G["state"])
    o1, _ = ccq.gla_fwd(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["lam"]), st, seq_split=split)
    o2, _, ck = ccq.gla_fwd_save(d(P["q"]), d(P["k"]), d(P["v"]), d(P["gate"]), d(P["lam"]), st,
                                 seq_split=split, algo="wide")
    assert rel_err(o2, o1.double().cpu().numpy()) <= TOLB
    _compare(_gpu(P, G, ckpt=ck, seq_split=split), _ref(P, G), f"wide checkpoints, split {split}")
