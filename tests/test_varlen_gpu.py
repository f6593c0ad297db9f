"""GPU parity of ccq_fwd_varlen (packed variable-length sequences): every sequence of the pack
against the oracle run on that sequence alone, both backbones, the chunkwise (bf16, d = 128) and
recurrent (fp32, d = 64) paths, empty and one-token sequences, resumed per-sequence states."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import GDN, GLA, TOL, rel_err

pytestmark = pytest.mark.gpu
LENS = [130, 1, 64, 0, 200, 65]


@pytest.fixture(autouse=True)
def _status():
    yield
    ccq.device_status()


@pytest.mark.parametrize("backbone", [GLA, GDN])
@pytest.mark.parametrize("dtype,D", [(torch.bfloat16, 128), (torch.float32, 64)])
@pytest.mark.parametrize("resumed", [False, True])
def test_varlen_matches_per_sequence_oracle(backbone, dtype, D, resumed):
    H = 4
    total = sum(LENS)
    cu = np.concatenate([[0], np.cumsum(LENS)]).tolist()
    P = gen.make_inputs(backbone, 1, total, H, D, D, dtype=dtype, seed=61, lam="trained", keys="structured")
    sq = {n: (None if x is None else x[0]) for n, x in P.items()}  # [total, H, ...]
    ns = len(LENS)
    st = None
    if resumed:
        G = gen.make_backward_inputs(ns, 1, H, D, D, seed=62, prefix=20, state_grads=False)["state"]
        st = ccq.CCQState(G["S"].float().cuda(), G["C"].float().cuda(), G["m"].float().cuda(), G["t"].cuda())
    d = lambda x: None if x is None else x.cuda().contiguous()  # noqa: E731
    o, fs = ccq.fwd_varlen(backbone, d(sq["q"]), d(sq["k"]), d(sq["v"]), d(sq["gate"]), d(sq["lam"]), cu,
                           beta=d(sq["beta"]), state=st)
    torch.cuda.synchronize()
    tol = TOL[dtype]
    for s in range(ns):
        a, b = cu[s], cu[s + 1]
        one = {n: (None if x is None else x[a:b].unsqueeze(0)) for n, x in sq.items()}
        kw = {}
        if resumed:
            kw = dict(S0=G["S"][s:s + 1].float(), C0=G["C"][s:s + 1].float(), m0=G["m"][s:s + 1].float(),
                      t0=G["t"][s:s + 1])
        ref = oracle.forward(backbone, one["q"], one["k"], one["v"], one["gate"], one["lam"], beta=one["beta"], **kw)
        if b > a:
            assert rel_err(o[a:b], ref["o"][0]) <= tol, (s, "o")
        for n in ("S", "C", "m"):
            assert rel_err(getattr(fs, n)[s], ref[n][0]) <= tol, (s, n)
        assert int(fs.t[s]) == int(ref["t"][0])


@pytest.mark.parametrize("backbone", [GLA, GDN])
def test_varlen_mix_of_64_sequences(backbone):
    """One launch over 64 sequences of 100-4000 tokens (H = 16, d = 128, bf16): sampled
    (sequence, head) pairs against the oracle run on that sequence and head alone, and every
    sequence's position count."""
    rng = np.random.default_rng(77)
    lens = rng.integers(100, 4001, size=64).tolist()
    H = 16
    total = sum(lens)
    cu = np.concatenate([[0], np.cumsum(lens)]).tolist()
    P = gen.make_inputs(backbone, 1, total, H, 128, 128, dtype=torch.bfloat16, seed=63, lam="trained",
                        keys="structured")
    sq = {n: (None if x is None else x[0]) for n, x in P.items()}
    d = lambda x: None if x is None else x.cuda().contiguous()  # noqa: E731
    o, fs = ccq.fwd_varlen(backbone, d(sq["q"]), d(sq["k"]), d(sq["v"]), d(sq["gate"]), d(sq["lam"]), cu,
                           beta=d(sq["beta"]))
    torch.cuda.synchronize()
    assert fs.t.cpu().tolist() == lens
    o = o.cpu()
    for s, h in ((0, 0), (17, 5), (40, 15), (63, 9), (int(np.argmin(lens)), 3)):
        a, b = cu[s], cu[s + 1]
        one = {n: (None if x is None else x[a:b, h:h + 1].unsqueeze(0)) for n, x in sq.items()}
        ref = oracle.forward(backbone, one["q"], one["k"], one["v"], one["gate"], one["lam"], beta=one["beta"])
        assert rel_err(o[a:b, h:h + 1], ref["o"][0]) <= TOL[torch.bfloat16], (s, h, "o")
        for n in ("S", "C", "m"):
            assert rel_err(getattr(fs, n)[s, h:h + 1].cpu(), ref[n][0]) <= TOL[torch.bfloat16], (s, h, n)
