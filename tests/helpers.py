"""Shared helpers of the GPU parity tests: move seeded inputs to the device,
call the library through its binding, call the oracle, and measure the
relative error max|x - ref| / max|ref| that the tolerances are stated in."""
import numpy as np
import torch

import oracle
from paper_2606_01294_gb300 import ccq
from paper_2606_01294_gb300 import inputs as gen

GLA, GDN = gen.GLA, gen.GDN
# max|x - ref| / max|ref| bounds for o and the final states
TOL = {torch.float32: 1e-4, torch.bfloat16: 2e-2}


def rel_err(x, ref) -> float:
    if isinstance(x, torch.Tensor):
        x = x.detach().float().cpu().double().numpy()
    ref = np.asarray(ref, dtype=np.float64)
    denom = np.abs(ref).max()
    return float(np.abs(x - ref).max() / max(denom, 1e-30))


def to_dev(P, device="cuda"):
    return {n: (None if x is None else x.to(device)) for n, x in P.items()}


def state_to_dev(st, device="cuda"):
    if st is None:
        return None
    return ccq.CCQState(torch.as_tensor(st["S"], dtype=torch.float32, device=device).contiguous(),
                        torch.as_tensor(st["C"], dtype=torch.float32, device=device).contiguous(),
                        torch.as_tensor(st["m"], dtype=torch.float32, device=device).contiguous(),
                        torch.as_tensor(st["t"], dtype=torch.int64, device=device).contiguous())


def state_f32(st):
    """Round an oracle state to the fp32 the library stores (for a resumed call)."""
    return {n: (np.asarray(v, dtype=np.float32).astype(np.float64) if n != "t" else v)
            for n, v in st.items()}


def gpu_forward(backbone, P, state=None, **kw):
    D = to_dev(P)
    if backbone == GLA:
        o, fs = ccq.gla_fwd(D["q"], D["k"], D["v"], D["gate"], D["lam"], state, **kw)
    else:
        o, fs = ccq.gdn_fwd(D["q"], D["k"], D["v"], D["gate"], D["beta"], D["lam"], state, **kw)
    torch.cuda.synchronize()
    return o, fs


def oracle_forward(backbone, P, state=None, **kw):
    st = state or {}
    return oracle.forward(backbone, P["q"], P["k"], P["v"], P["gate"], P["lam"], beta=P["beta"],
                          S0=st.get("S"), C0=st.get("C"), m0=st.get("m"), t0=st.get("t"), **kw)


def compare(o, fs, ref, tol, what=""):
    errs = {"o": rel_err(o, ref["o"]), "S": rel_err(fs.S, ref["S"]),
            "C": rel_err(fs.C, ref["C"]), "m": rel_err(fs.m, ref["m"])}
    bad = {k: v for k, v in errs.items() if not v <= tol}
    assert not bad, f"{what}: relative errors above {tol}: {errs}"
    np.testing.assert_array_equal(fs.t.cpu().numpy(), ref["t"])
    return errs


def slice_bh(P, b, h):
    """Inputs of one (batch row, head) pair, kept 4-D."""
    return {n: (None if x is None else x[b:b + 1, :, h:h + 1].contiguous()) for n, x in P.items()}


def correction_bound(o1_ref, d_ref, dtype) -> float:
    """Bound for the isolated CCQ term o(lambda) - o(0): the stated output
    tolerance plus the floor of differencing two outputs rounded to the output
    dtype (each carries up to half an ulp, 2^-9 of its magnitude for bf16)."""
    half_ulp = {torch.float32: 2.0 ** -24, torch.bfloat16: 2.0 ** -9}[dtype]
    return TOL[dtype] + 2 * half_ulp * float(np.abs(o1_ref).max()) / float(np.abs(d_ref).max())
