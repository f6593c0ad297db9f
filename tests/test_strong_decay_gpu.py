"""GPU parity under strong forgetting (Sec. 2.2, the backbone write rules), element by element
against the oracle, on the whole-sequence and the segment-parallel paths.

Gated DeltaNet: every decay factor of the chunk kernels is an exponential of a non-positive
argument, so any decay is exact (where a factor underflows its contribution is exactly zero);
cases: -8 softplus(N(0,1)) and a constant -5 per token.
GLA (per key dimension gates): the factors are measured from reference tokens, one per chunk
in the default kernel and one per half chunk in the "wide" kernel; cases inside both ranges
(logsigmoid(N(0,1)) without the 1/16), inside only the wide kernel's (a constant -3 and -4.5,
where the default kernel must report CCQ_ERR_RANGE), and beyond both (-6, reported)."""
import numpy as np
import pytest
import torch

from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen
from tests.helpers import GDN, GLA, TOL, compare, gpu_forward, oracle_forward

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _status():
    yield
    ccq.device_status()


def _finite(o, fs):
    for x in (o, fs.S, fs.C, fs.m):
        assert torch.isfinite(x.float()).all()


@pytest.mark.parametrize("algo", ["chunkwise", "wide"])
@pytest.mark.parametrize("split", [1, 2])
def test_gla_strong_gates(algo, split):
    """logsigmoid(N(0,1)) per token and key dimension, without the 1/16: inside both kernels'
    range."""
    P = gen.make_inputs(GLA, 1, 300, 2, 128, 128, dtype=torch.bfloat16, seed=71, lam="trained",
                        keys="structured", gates="strong")
    o, fs = gpu_forward(GLA, P, algo=algo, seq_split=split)
    _finite(o, fs)
    compare(o, fs, oracle_forward(GLA, P), TOL[torch.bfloat16], f"GLA {algo} strong split={split}")


@pytest.mark.parametrize("gates", [-3.0, -4.5])
@pytest.mark.parametrize("split", [1, 2])
def test_gla_wide_range(gates, split):
    """A constant log gate of -3 or -4.5 per token and key dimension: beyond the midpoint
    kernel's range (a 32-token half sums to -93 or worse), which reports CCQ_ERR_RANGE, and
    inside the two-reference kernel's, which matches the oracle."""
    P = gen.make_inputs(GLA, 1, 300, 2, 128, 128, dtype=torch.bfloat16, seed=71, lam="trained",
                        keys="structured", gates=gates)
    gpu_forward(GLA, P, algo="chunkwise", seq_split=split)
    with pytest.raises(ccq.CCQError) as ex:
        ccq.device_status()
    assert ex.value.status == ccq.CCQ_ERR_RANGE
    o, fs = gpu_forward(GLA, P, algo="wide", seq_split=split)
    _finite(o, fs)
    compare(o, fs, oracle_forward(GLA, P), TOL[torch.bfloat16], f"GLA wide gates={gates} split={split}")


def test_gla_beyond_wide_range_is_reported():
    """-6 per token: a 16-token quarter sums to -96, beyond the two-reference kernel too."""
    P = gen.make_inputs(GLA, 1, 130, 1, 128, 128, dtype=torch.bfloat16, seed=74, gates=-6.0)
    gpu_forward(GLA, P, algo="wide")
    with pytest.raises(ccq.CCQError) as ex:
        ccq.device_status()
    assert ex.value.status == ccq.CCQ_ERR_RANGE


@pytest.mark.parametrize("gates", ["strong", -5.0])
@pytest.mark.parametrize("split", [1, 2, 3])
def test_gdn_strong_decay(gates, split):
    P = gen.make_inputs(GDN, 1, 600, 2, 128, 128, dtype=torch.bfloat16, seed=72, lam="trained",
                        keys="structured", gates=gates)
    o, fs = gpu_forward(GDN, P, algo="chunkwise", seq_split=split)
    _finite(o, fs)
    compare(o, fs, oracle_forward(GDN, P), TOL[torch.bfloat16], f"GDN gates={gates} split={split}")


@pytest.mark.parametrize("backbone", [GLA, GDN])
def test_decode_strong_decay(backbone):
    """The recurrent path (fp32 arithmetic per token) under the same gates."""
    P = gen.make_inputs(backbone, 1, 130, 2, 64, 64, dtype=torch.float32, seed=73, lam="trained",
                        gates="strong")
    o, fs = gpu_forward(backbone, P)
    _finite(o, fs)
    compare(o, fs, oracle_forward(backbone, P), TOL[torch.float32], "recurrent strong gates")
