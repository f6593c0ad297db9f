"""GPU parity of ccq_decode_step (Algorithm 2, one token, cache updated in
place) and of ccq_gdn_fwd against the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import (GDN, GLA, TOL, compare, gpu_forward, oracle_forward, rel_err, slice_bh,
                           state_f32, state_to_dev)

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _status():
    yield
    ccq.device_status()


def _decode_case(backbone, B, H, d, dtype, seed, lam="trained"):
    D = gen.make_decode_inputs(backbone, B, H, d, d, dtype=dtype, seed=seed, lam=lam)
    pre = oracle_forward(backbone, D["prefix"])
    return D["token"], state_f32(pre)


@pytest.mark.parametrize("backbone", [GLA, GDN])
@pytest.mark.parametrize("dtype,d", [(torch.bfloat16, 128), (torch.float32, 64), (torch.float32, 128)])
def test_decode_step_matches_oracle(backbone, dtype, d):
    tok, st = _decode_case(backbone, 4, 3, d, dtype, seed=21)
    ref = oracle.decode_step(backbone, tok["q"], tok["k"], tok["v"], tok["gate"], tok["lam"],
                             st["S"], st["C"], st["m"], st["t"], beta=tok["beta"])
    S = state_to_dev(st)
    T = {n: (None if x is None else x.cuda()) for n, x in tok.items()}
    o = ccq.decode_step(backbone, T["q"], T["k"], T["v"], T["gate"], T["lam"], S, beta=T["beta"])
    torch.cuda.synchronize()
    tol = TOL[dtype]
    assert rel_err(o, ref["o"]) <= tol
    for n in ("S", "C", "m"):
        assert rel_err(getattr(S, n), ref[n]) <= tol, n
    np.testing.assert_array_equal(S.t.cpu().numpy(), ref["t"])


@pytest.mark.parametrize("backbone", [GLA, GDN])
def test_prefill_then_decode_equals_longer_prefill(backbone):
    """A forward over T tokens followed by one decode step equals a forward
    over T + 1 tokens (GPU only: the two entry points agree)."""
    P = gen.make_inputs(backbone, 2, 97, 2, 128, 128, dtype=torch.bfloat16, seed=22, lam="trained")
    head = {n: (None if x is None else x[:, :96].contiguous()) for n, x in P.items()}
    tok = {n: (None if x is None else x[:, 96].contiguous().cuda()) for n, x in P.items()}
    _, st = gpu_forward(backbone, head)
    o = ccq.decode_step(backbone, tok["q"], tok["k"], tok["v"], tok["gate"], tok["lam"], st,
                        beta=tok["beta"])
    full = oracle_forward(backbone, P)
    assert rel_err(o, full["o"][:, 96]) <= TOL[torch.bfloat16]
    assert rel_err(st.S, full["S"]) <= TOL[torch.bfloat16]
    assert int(st.t[0]) == 97


def test_decode_full_size_sampled():
    """B=256, H=16, Dk=Dv=128 (the decode benchmark's launch), sampled pairs."""
    B, H, d = 256, 16, 128
    tok, st = _decode_case(GLA, B, H, d, torch.bfloat16, seed=23)
    S = state_to_dev(st)
    T = {n: (None if x is None else x.cuda()) for n, x in tok.items()}
    o = ccq.decode_step(GLA, T["q"], T["k"], T["v"], T["gate"], T["lam"], S)
    torch.cuda.synchronize()
    for b, h in [(0, 0), (17, 5), (255, 15)]:
        sub = {n: (None if x is None else x[b:b + 1, h:h + 1]) for n, x in tok.items()}
        ref = oracle.decode_step(GLA, sub["q"], sub["k"], sub["v"], sub["gate"], sub["lam"],
                                 st["S"][b:b + 1, h:h + 1], st["C"][b:b + 1, h:h + 1],
                                 st["m"][b:b + 1, h:h + 1], st["t"][b:b + 1])
        assert rel_err(o[b:b + 1, h:h + 1], ref["o"]) <= TOL[torch.bfloat16]
        assert rel_err(S.S[b:b + 1, h:h + 1], ref["S"]) <= TOL[torch.bfloat16]
        assert rel_err(S.C[b:b + 1, h:h + 1], ref["C"]) <= TOL[torch.bfloat16]


@pytest.mark.parametrize("lam", ["init", "high"])
@pytest.mark.parametrize("dtype,d", [(torch.float32, 64), (torch.bfloat16, 128)])
def test_gdn_forward_matches_oracle(lam, dtype, d):
    P = gen.make_inputs(GDN, 2, 150, 2, d, d, dtype=dtype, seed=24, lam=lam, keys="structured")
    o, fs = gpu_forward(GDN, P)
    compare(o, fs, oracle_forward(GDN, P), TOL[dtype], f"gdn {lam}")


def test_gdn_full_size_sampled():
    w = dict(gen.WORKLOADS["gdn_bf16_4k"])
    backbone = w.pop("backbone")
    w["B"] = 2  # the recurrent GDN kernel is a CUDA-core path; keep the runtime short
    P = gen.make_inputs(backbone, **w)
    o, fs = gpu_forward(GDN, P)
    for b, h in [(0, 0), (1, 11)]:
        ref = oracle_forward(GDN, slice_bh(P, b, h))
        assert rel_err(o[b:b + 1, :, h:h + 1], ref["o"]) <= TOL[torch.bfloat16]
        assert rel_err(fs.S[b:b + 1, h:h + 1], ref["S"]) <= TOL[torch.bfloat16]
