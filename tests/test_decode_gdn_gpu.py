"""GPU parity of ccq_decode_step (Algorithm 2, one token, cache updated in
place) and of ccq_gdn_fwd against the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import (correction_bound, GDN, GLA, TOL, compare, gpu_forward, oracle_forward, rel_err, slice_bh,
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


@pytest.mark.parametrize("backbone", [GLA, GDN])
def test_repeated_in_place_decode_every_head(backbone):
    """Five decode steps in place on 64 batch rows x 16 heads (1024 CTAs, so the
    heads of one row run in different waves): the shared position count t must
    advance by exactly one per step for every head, whatever the CTA order."""
    B, H, d = 64, 16, 128
    steps = 5
    P = gen.make_inputs(backbone, B, 40 + steps, H, d, d, dtype=torch.bfloat16, seed=31, lam="high",
                        keys="structured")
    pre = {n: (None if x is None else x[:, :40].contiguous()) for n, x in P.items()}
    _, st = gpu_forward(backbone, pre)
    for s in range(steps):
        tok = {n: (None if x is None else x[:, 40 + s].contiguous().cuda()) for n, x in P.items()}
        o = ccq.decode_step(backbone, tok["q"], tok["k"], tok["v"], tok["gate"], tok["lam"], st,
                            beta=tok["beta"])
        torch.cuda.synchronize()
        assert (st.t.cpu() == 41 + s).all()
    full = oracle_forward(backbone, P)
    assert rel_err(o, full["o"][:, -1]) <= TOL[torch.bfloat16]
    for n in ("S", "C", "m"):
        assert rel_err(getattr(st, n), full[n]) <= TOL[torch.bfloat16], n


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


@pytest.mark.parametrize("lam", ["init", "trained", "high"])
@pytest.mark.parametrize("keys", ["iso", "structured", "lowrank"])
def test_gdn_chunkwise_ragged(lam, keys):
    """Chunkwise tensor-core GDN (WY/UT kernel + sequential kernel), T = 200."""
    P = gen.make_inputs(GDN, 2, 200, 3, 128, 128, dtype=torch.bfloat16, seed=31, lam=lam, keys=keys)
    o, fs = gpu_forward(GDN, P, algo="chunkwise")
    compare(o, fs, oracle_forward(GDN, P), TOL[torch.bfloat16], f"gdn chunkwise {lam} {keys}")


@pytest.mark.parametrize("T", [1, 63, 64, 65, 129])
def test_gdn_chunk_boundaries(T):
    P = gen.make_inputs(GDN, 1, T, 2, 128, 128, dtype=torch.bfloat16, seed=200 + T, lam="trained",
                        keys="structured")
    o, fs = gpu_forward(GDN, P, algo="chunkwise")
    compare(o, fs, oracle_forward(GDN, P), TOL[torch.bfloat16], f"gdn T={T}")


def test_gdn_chunkwise_correction_isolated():
    P = gen.make_inputs(GDN, 1, 192, 2, 128, 128, dtype=torch.bfloat16, seed=32, lam="high", keys="lowrank")
    P0 = dict(P, lam=torch.zeros_like(P["lam"]))
    o1, _ = gpu_forward(GDN, P, algo="chunkwise")
    o0, _ = gpu_forward(GDN, P0, algo="chunkwise")
    ref1 = oracle_forward(GDN, P)["o"]
    d_ref = ref1 - oracle_forward(GDN, P0)["o"]
    d = o1.double().cpu().numpy() - o0.double().cpu().numpy()
    assert np.abs(d_ref).max() > 0.1 * np.abs(ref1).max()
    bound, err = correction_bound(ref1, d_ref, torch.bfloat16), rel_err(d, d_ref)
    assert err <= bound, f"isolated CCQ term: error {err:.3e} above its bound {bound:.3e}"


def test_gdn_correction_dominant():
    """Keys and queries in one two-dimensional subspace with lambda = 0.9: the CCQ term is more than
    half of the output (rounding floor of the bound below 1 %)."""
    P = gen.make_inputs(GDN, 1, 192, 2, 128, 128, dtype=torch.bfloat16, seed=15, lam="high", keys="rank2",
                        queries="lowrank")
    P0 = dict(P, lam=torch.zeros_like(P["lam"]))
    o1, _ = gpu_forward(GDN, P)
    o0, _ = gpu_forward(GDN, P0)
    ref1 = oracle_forward(GDN, P)["o"]
    d_ref = ref1 - oracle_forward(GDN, P0)["o"]
    d = o1.double().cpu().numpy() - o0.double().cpu().numpy()
    assert np.abs(d_ref).max() >= 0.5 * np.abs(ref1).max()
    bound, err = correction_bound(ref1, d_ref, torch.bfloat16), rel_err(d, d_ref)
    assert bound <= TOL[torch.bfloat16] + 0.008
    assert err <= bound, f"isolated CCQ term: error {err:.3e} above its bound {bound:.3e}"


@pytest.mark.parametrize("opts", [dict(l2norm=False), dict(scale=0.37), dict(l2norm=False, centered=False)])
def test_gdn_forward_options(opts):
    """Chunkwise Gated DeltaNet without in-kernel normalisation (the generator's unit q, k)
    and with a read scale other than 1/sqrt(d_k)."""
    P = gen.make_inputs(GDN, 2, 200, 2, 128, 128, dtype=torch.bfloat16, seed=16, lam="trained",
                        keys="structured")
    o, fs = gpu_forward(GDN, P, **opts)
    ref = oracle_forward(GDN, P, **opts)
    compare(o, fs, ref, TOL[torch.bfloat16], f"GDN {opts}")


def test_gdn_chunkwise_resume_and_matches_recurrent():
    P = gen.make_inputs(GDN, 2, 230, 2, 128, 128, dtype=torch.bfloat16, seed=33, lam="trained",
                        keys="structured")
    head = {n: (None if x is None else x[:, :100].contiguous()) for n, x in P.items()}
    tail = {n: (None if x is None else x[:, 100:].contiguous()) for n, x in P.items()}
    o1, fs1 = gpu_forward(GDN, head, algo="chunkwise")
    o2, fs2 = gpu_forward(GDN, tail, fs1, algo="chunkwise")
    full = oracle_forward(GDN, P)
    assert rel_err(torch.cat([o1, o2], dim=1), full["o"]) <= TOL[torch.bfloat16]
    assert rel_err(fs2.S, full["S"]) <= TOL[torch.bfloat16]
    orr, _ = gpu_forward(GDN, P, algo="recurrent")
    oc, _ = gpu_forward(GDN, P, algo="chunkwise")
    assert rel_err(oc, orr.double().cpu().numpy()) <= TOL[torch.bfloat16]


def test_gdn_full_size_sampled():
    """B=8, H=16, T=4096 (the benchmark's launch); sampled pairs against the oracle."""
    w = dict(gen.WORKLOADS["gdn_bf16_4k"])
    backbone = w.pop("backbone")
    P = gen.make_inputs(backbone, **w)
    o, fs = gpu_forward(GDN, P)
    for b, h in [(0, 0), (5, 11), (7, 15)]:
        ref = oracle_forward(GDN, slice_bh(P, b, h))
        assert rel_err(o[b:b + 1, :, h:h + 1], ref["o"]) <= TOL[torch.bfloat16]
        assert rel_err(fs.S[b:b + 1, h:h + 1], ref["S"]) <= TOL[torch.bfloat16]
        assert rel_err(fs.C[b:b + 1, h:h + 1], ref["C"]) <= TOL[torch.bfloat16]


@pytest.mark.parametrize("split", [2, 3, 5])
@pytest.mark.parametrize("decay", ["drawn", "slow"])
def test_gdn_segmented_sequences(split, decay):
    """Sequences cut into segments (segment state and transition from zero, fp32
    combine, chunk kernel per segment) equal one sequential walk: T = 700 (11 chunks,
    ragged tail), resumed state.  "slow" divides the log decays by 100 so the segment
    transition P stays far from zero and every term of P H + Q is exercised."""
    P = gen.make_inputs(GDN, 2, 700, 2, 128, 128, dtype=torch.bfloat16, seed=60 + split, lam="trained",
                        keys="structured")
    prev = gen.make_inputs(GDN, 2, 90, 2, 128, 128, dtype=torch.bfloat16, seed=70, lam="trained")
    if decay == "slow":
        P["gate"] = P["gate"] / 100
        prev["gate"] = prev["gate"] / 100
    st = state_f32(oracle_forward(GDN, prev))
    o, fs = gpu_forward(GDN, P, state_to_dev(st), algo="chunkwise", seq_split=split)
    compare(o, fs, oracle_forward(GDN, P, st), TOL[torch.bfloat16], f"gdn split={split} {decay}")


def test_gdn_20k_sampled():
    """B=1, H=16, T=20480 (the long-context benchmark's launch, split into segments);
    sampled heads against the oracle."""
    w = dict(gen.WORKLOADS["gdn_bf16_20k"])
    backbone = w.pop("backbone")
    P = gen.make_inputs(backbone, **w)
    o, fs = gpu_forward(GDN, P)
    for b, h in [(0, 0), (0, 9)]:
        ref = oracle_forward(GDN, slice_bh(P, b, h))
        assert rel_err(o[b:b + 1, :, h:h + 1], ref["o"]) <= TOL[torch.bfloat16]
        assert rel_err(fs.S[b:b + 1, h:h + 1], ref["S"]) <= TOL[torch.bfloat16]
        assert rel_err(fs.C[b:b + 1, h:h + 1], ref["C"]) <= TOL[torch.bfloat16]
        assert rel_err(fs.m[b:b + 1, h:h + 1], ref["m"]) <= TOL[torch.bfloat16]
