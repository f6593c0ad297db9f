"""Host logic of bench.py, checked without a GPU.

The roofline fraction bench.py reports divides an algorithmic byte count by a kernel's
time, so that count is pinned here to the tensors one step actually moves: the bytes of
the inputs the seeded generator draws, of the outputs the library writes and of the
states it reads or writes, counted from tensor shapes and dtypes rather than from the
formula. bench.py's copy of the library's segment split is checked against the split
the library itself reports (through the workspace size it asks for)."""
import ctypes

import pytest
import torch

import bench
from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen


def nbytes(*ts):
    return sum(t.numel() * t.element_size() for t in ts if t is not None)


def final_states(B, H, D):
    # S [B,H,Dk,Dv], C [B,H,Dk,Dk], m [B,H,Dk] fp32 and the position count t [B] int64
    return (torch.empty(B, H, D, D), torch.empty(B, H, D, D), torch.empty(B, H, D),
            torch.empty(B, dtype=torch.int64))


@pytest.mark.parametrize("kind,bb", [("gla", gen.GLA), ("gdn", gen.GDN)])
def test_forward_bytes_are_the_tensors_a_step_moves(kind, bb):
    B, H, T, D = 2, 3, 80, 128
    P = gen.make_inputs(bb, B, T, H, D, D, dtype=torch.bfloat16, seed=1)
    o = torch.empty_like(P["v"])
    moved = nbytes(P["q"], P["k"], P["v"], P["gate"], P["beta"], P["lam"], o,
                   *final_states(B, H, D))
    assert bench.algorithmic_bytes(kind, B, H, T, D) == moved


def test_decode_bytes_are_the_token_and_the_cache_read_and_written():
    B, H, D = 5, 2, 128
    Dd = gen.make_decode_inputs(gen.GLA, B, H, D, D, prefix=3)
    tk = Dd["token"]
    o = torch.empty_like(tk["v"])
    cache = final_states(B, H, D)
    moved = nbytes(tk["q"], tk["k"], tk["v"], tk["gate"], tk["lam"], o) + 2 * nbytes(*cache)
    assert bench.algorithmic_bytes("decode", B, H, 1, D) == moved


def test_training_step_bytes_are_forward_plus_backward_tensors():
    B, H, T, D = 2, 2, 70, 128
    P = gen.make_inputs(gen.GLA, B, T, H, D, D, dtype=torch.bfloat16, seed=2)
    G = gen.make_backward_inputs(B, T, H, D, D, seed=3, state_grads=False)
    fwd = nbytes(P["q"], P["k"], P["v"], P["gate"], P["lam"], torch.empty_like(P["v"]),
                 *final_states(B, H, D))
    grads = [torch.empty_like(P[n]) for n in ("q", "k", "v", "gate", "lam")]
    # initial-state gradients dS0, dC0, dm0 (fp32); no position count
    init = final_states(B, H, D)[:3]
    bwd = nbytes(P["q"], P["k"], P["v"], P["gate"], P["lam"], G["dout"], *grads, *init)
    assert bench.algorithmic_bytes("glabwd", B, H, T, D) == fwd + bwd


@pytest.fixture(scope="module")
def lib():
    try:
        return ccq.load_library()
    except (OSError, RuntimeError) as e:
        pytest.skip(f"libccq.so not built: {e}")


@pytest.mark.parametrize("B,H,T", [(8, 16, 4096), (1, 16, 20480), (4, 16, 4096), (1, 1, 640),
                                   (1, 2, 300), (2, 8, 8192), (1, 4, 100000), (3, 5, 1)])
def test_segment_split_mirrors_the_library(lib, B, H, T):
    # Without a device the library assumes 148 SMs; the split it picks shows in the
    # workspace it asks for (one slot of per-segment states per segment, none unsplit).
    sms = 148
    n = ctypes.c_size_t(0)
    assert lib.ccq_gla_workspace_size(B, T, H, 128, 128, 0, ctypes.byref(ccq.params()),
                                      ctypes.byref(n)) == 0
    seg_bytes = (2 * 128 * 128 + 2 * 128) * 4
    nseg = bench.gla_segments(B, H, T, sms)
    assert n.value == (B * H * nseg * seg_bytes if nseg > 1 else 0)
