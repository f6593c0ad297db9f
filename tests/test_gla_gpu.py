"""GPU parity of ccq_gla_fwd against the fp64 oracle (element by element).

Bounds (max|x - ref| / max|ref| for o and the final S, C, m; t exact):
1e-4 for fp32 inputs, 2e-2 for bf16 inputs with fp32 accumulation.
"""
import numpy as np
import pytest
import torch

from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import (correction_bound, GLA, TOL, compare, gpu_forward, oracle_forward, rel_err, slice_bh,
                           state_f32, state_to_dev)

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _status():
    yield
    ccq.device_status()


@pytest.mark.parametrize("lam", ["init", "trained", "high"])
@pytest.mark.parametrize("keys", ["iso", "structured"])
def test_fp32_small_workload(lam, keys):
    """fp32, B=1, H=2, T=256, Dk=Dv=64 (recurrent CUDA-core kernel)."""
    P = gen.make_inputs(GLA, 1, 256, 2, 64, 64, dtype=torch.float32, seed=1235, lam=lam, keys=keys)
    o, fs = gpu_forward(GLA, P)
    compare(o, fs, oracle_forward(GLA, P), TOL[torch.float32], f"fp32 {lam} {keys}")


@pytest.mark.parametrize("lam", ["init", "trained", "high"])
@pytest.mark.parametrize("keys", ["iso", "structured", "lowrank"])
def test_bf16_chunkwise_ragged(lam, keys):
    """bf16, Dk=Dv=128, T=200: three full chunks and an 8-token tail."""
    P = gen.make_inputs(GLA, 2, 200, 3, 128, 128, dtype=torch.bfloat16, seed=11, lam=lam, keys=keys)
    o, fs = gpu_forward(GLA, P, algo="chunkwise")
    compare(o, fs, oracle_forward(GLA, P), TOL[torch.bfloat16], f"bf16 {lam} {keys}")


@pytest.mark.parametrize("algo,dtype", [("chunkwise", torch.bfloat16), ("recurrent", torch.float32)])
def test_correction_isolated(algo, dtype):
    """The CCQ term alone: o(lambda) - o(0) against the oracle's difference."""
    P = gen.make_inputs(GLA, 1, 192, 2, 128, 128, dtype=dtype, seed=12, lam="high", keys="lowrank")
    P0 = dict(P, lam=torch.zeros_like(P["lam"]))
    o1, _ = gpu_forward(GLA, P, algo=algo)
    o0, _ = gpu_forward(GLA, P0, algo=algo)
    ref1 = oracle_forward(GLA, P)["o"]
    d_ref = ref1 - oracle_forward(GLA, P0)["o"]
    d = o1.double().cpu().numpy() - o0.double().cpu().numpy()
    assert np.abs(d_ref).max() > 0.1 * np.abs(ref1).max()
    bound, err = correction_bound(ref1, d_ref, dtype), rel_err(d, d_ref)
    assert err <= bound, f"isolated CCQ term: error {err:.3e} above its bound {bound:.3e}"


@pytest.mark.parametrize("algo", ["chunkwise", "recurrent"])
def test_correction_dominant(algo):
    """Keys and queries in one two-dimensional subspace with lambda = 0.9: the CCQ term is more than
    half of the output, so the rounding floor of the isolated-term bound stays below 1 %."""
    P = gen.make_inputs(GLA, 1, 192, 2, 128, 128, dtype=torch.bfloat16, seed=13, lam="high", keys="rank2",
                        queries="lowrank")
    P0 = dict(P, lam=torch.zeros_like(P["lam"]))
    o1, _ = gpu_forward(GLA, P, algo=algo)
    o0, _ = gpu_forward(GLA, P0, algo=algo)
    ref1 = oracle_forward(GLA, P)["o"]
    d_ref = ref1 - oracle_forward(GLA, P0)["o"]
    d = o1.double().cpu().numpy() - o0.double().cpu().numpy()
    assert np.abs(d_ref).max() >= 0.5 * np.abs(ref1).max()
    bound, err = correction_bound(ref1, d_ref, torch.bfloat16), rel_err(d, d_ref)
    assert bound <= TOL[torch.bfloat16] + 0.008
    assert err <= bound, f"isolated CCQ term: error {err:.3e} above its bound {bound:.3e}"


@pytest.mark.parametrize("opts", [dict(l2norm=False), dict(scale=0.37), dict(l2norm=False, centered=False)])
@pytest.mark.parametrize("algo", ["chunkwise", "recurrent"])
def test_forward_options(opts, algo):
    """The forward without in-kernel normalisation (unit keys from the generator, raw queries)
    and with a read scale other than 1/sqrt(d_k)."""
    P = gen.make_inputs(GLA, 2, 200, 2, 128, 128, dtype=torch.bfloat16, seed=14, lam="trained",
                        keys="structured")
    o, fs = gpu_forward(GLA, P, algo=algo, **opts)
    ref = oracle_forward(GLA, P, **opts)
    compare(o, fs, ref, TOL[torch.bfloat16], f"GLA {algo} {opts}")


def test_chunkwise_matches_recurrent_gpu():
    P = gen.make_inputs(GLA, 2, 300, 2, 128, 128, dtype=torch.bfloat16, seed=13, lam="trained",
                        keys="structured")
    oc, sc = gpu_forward(GLA, P, algo="chunkwise")
    orr, sr = gpu_forward(GLA, P, algo="recurrent")
    assert rel_err(oc, orr.double().cpu().numpy()) <= TOL[torch.bfloat16]
    assert rel_err(sc.S, sr.S.double().cpu().numpy()) <= TOL[torch.bfloat16]
    assert rel_err(sc.C, sr.C.double().cpu().numpy()) <= 1e-3


@pytest.mark.parametrize("T", [1, 63, 64, 65, 129])
def test_chunk_boundaries(T):
    P = gen.make_inputs(GLA, 1, T, 2, 128, 128, dtype=torch.bfloat16, seed=100 + T, lam="trained",
                        keys="structured")
    o, fs = gpu_forward(GLA, P, algo="chunkwise")
    compare(o, fs, oracle_forward(GLA, P), TOL[torch.bfloat16], f"T={T}")


@pytest.mark.parametrize("algo", ["chunkwise", "recurrent"])
def test_resume_from_state(algo):
    """A second call started from the first call's final state equals one call."""
    P = gen.make_inputs(GLA, 2, 230, 2, 128, 128, dtype=torch.bfloat16, seed=14, lam="trained",
                        keys="structured")
    cut = 100
    head = {n: (None if x is None else x[:, :cut].contiguous()) for n, x in P.items()}
    tail = {n: (None if x is None else x[:, cut:].contiguous()) for n, x in P.items()}
    ref_head = oracle_forward(GLA, head)
    st = state_f32(ref_head)
    o, fs = gpu_forward(GLA, tail, state_to_dev(st), algo=algo)
    compare(o, fs, oracle_forward(GLA, tail, st), TOL[torch.bfloat16], "resumed")
    # and chaining two GPU calls
    o1, fs1 = gpu_forward(GLA, head, algo=algo)
    o2, fs2 = gpu_forward(GLA, tail, fs1, algo=algo)
    full = oracle_forward(GLA, P)
    assert rel_err(torch.cat([o1, o2], dim=1), full["o"]) <= TOL[torch.bfloat16]
    assert rel_err(fs2.S, full["S"]) <= TOL[torch.bfloat16]


def test_fp32_gate_and_uncentred():
    P = gen.make_inputs(GLA, 1, 150, 2, 128, 128, dtype=torch.bfloat16, gate_dtype=torch.float32,
                        seed=15, lam="high", keys="structured")
    o, fs = gpu_forward(GLA, P, algo="chunkwise", centered=False)
    compare(o, fs, oracle_forward(GLA, P, centered=False), TOL[torch.bfloat16], "uncentred")


def test_zero_length_passes_states_through():
    P = gen.make_inputs(GLA, 2, 70, 2, 128, 128, dtype=torch.bfloat16, seed=16)
    ref = oracle_forward(GLA, P)
    st = state_to_dev(state_f32(ref))
    e = {n: (None if x is None else x[:, :0].contiguous()) for n, x in P.items()}
    o, fs = gpu_forward(GLA, e, st)
    assert o.shape[1] == 0
    for n in ("S", "C", "m", "t"):
        assert torch.equal(getattr(fs, n), getattr(st, n))


def test_zero_rows_stay_finite():
    P = gen.make_inputs(GLA, 1, 130, 1, 128, 128, dtype=torch.bfloat16, seed=17, lam="high")
    P["q"][:, 5:9] = 0
    P["k"][:, 70:75] = 0
    o, fs = gpu_forward(GLA, P, algo="chunkwise")
    assert torch.isfinite(o.float()).all() and torch.isfinite(fs.S).all()
    compare(o, fs, oracle_forward(GLA, P), TOL[torch.bfloat16], "zero rows")


@pytest.mark.parametrize("name,pairs", [("gla_bf16_4k", [(0, 0), (3, 7), (7, 15)]),
                                        ("gla_bf16_20k", [(0, 0), (0, 9)])])
def test_full_size_sampled(name, pairs):
    """The benchmark's launch (all heads and batch rows at full size); the
    oracle checks sampled (batch, head) pairs element by element."""
    w = dict(gen.WORKLOADS[name])
    backbone = w.pop("backbone")
    P = gen.make_inputs(backbone, **w)
    o, fs = gpu_forward(GLA, P)
    for b, h in pairs:
        ref = oracle_forward(GLA, slice_bh(P, b, h))
        errs = {"o": rel_err(o[b:b + 1, :, h:h + 1], ref["o"]),
                "S": rel_err(fs.S[b:b + 1, h:h + 1], ref["S"]),
                "C": rel_err(fs.C[b:b + 1, h:h + 1], ref["C"]),
                "m": rel_err(fs.m[b:b + 1, h:h + 1], ref["m"])}
        assert max(errs.values()) <= TOL[torch.bfloat16], (b, h, errs)
        assert int(fs.t[b]) == P["q"].shape[1]


@pytest.mark.parametrize("split", [2, 3, 5])
def test_segmented_sequences(split):
    """Sequences cut into segments (state deltas, exclusive combine, recompute)
    equal one sequential walk: T = 700 (11 chunks, ragged tail), resumed state."""
    P = gen.make_inputs(GLA, 2, 700, 2, 128, 128, dtype=torch.bfloat16, seed=40 + split, lam="trained",
                        keys="structured")
    prev = gen.make_inputs(GLA, 2, 90, 2, 128, 128, dtype=torch.bfloat16, seed=50, lam="trained")
    st = state_f32(oracle_forward(GLA, prev))
    o, fs = gpu_forward(GLA, P, state_to_dev(st), algo="chunkwise", seq_split=split)
    compare(o, fs, oracle_forward(GLA, P, st), TOL[torch.bfloat16], f"split={split}")
