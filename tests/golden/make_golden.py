"""Write tests/golden/oracle_small.json: small fixed problems and the oracle's answers.

The paper prints no worked numerical example, so these fixtures are not the paper's
numbers: they are the fp64 oracle's results on tiny seeded problems, stored so that any
later change to the oracle's arithmetic shows up as a failing comparison
(tests/test_golden.py) and has to be justified by the passage it follows. The oracle
itself is pinned by brute force, closed forms and finite differences elsewhere in tests/.

Inputs are drawn here with numpy (seed per case) and stored with the answers, so the
fixture does not depend on any generator outside this file. Only ``oracle`` is called.

Run from the repository root:  python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)
import oracle  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_small.json")
B, T, H, DK, DV = 1, 8, 2, 4, 3


def rounded(d):
    """Inputs rounded to 5 decimals, so the stored text is exactly what the oracle saw."""
    return {n: (None if x is None else np.round(x, 5)) for n, x in d.items()}


def draw(seed, gdn):
    rng = np.random.RandomState(seed)
    q = rng.standard_normal((B, T, H, DK))
    k = rng.standard_normal((B, T, H, DK))
    v = rng.standard_normal((B, T, H, DV))
    if gdn:
        gate = -np.log1p(np.exp(rng.standard_normal((B, T, H))))          # log alpha = -softplus(N)
        beta = 1.0 / (1.0 + np.exp(-rng.standard_normal((B, T, H))))      # sigmoid(N)
    else:
        z = rng.standard_normal((B, T, H, DK))
        gate = -np.log1p(np.exp(-z)) / 16.0                                  # logsigmoid(N) / 16
        beta = None
    lam = 1.0 / (1.0 + np.exp(-(np.log(0.29 / 0.71) + 0.5 * rng.standard_normal((B, T, H)))))
    return rounded({"q": q, "k": k, "v": v, "gate": gate, "beta": beta, "lam": lam})


def initial_state(seed):
    rng = np.random.RandomState(seed)
    hist = rng.standard_normal((B, H, 5, DK))
    hist /= np.linalg.norm(hist, axis=-1, keepdims=True)
    st = rounded({"S": rng.standard_normal((B, H, DK, DV)) / DK,
                  "C": np.einsum("bhti,bhtj->bhij", hist, hist), "m": hist.sum(axis=2)})
    st["t"] = np.full((B,), 5, dtype=np.int64)
    return st


def listify(d, digits=None):
    """Nested lists for JSON; expected values are kept to 13 significant digits."""
    out = {}
    for n, x in d.items():
        if x is None:
            out[n] = None
            continue
        x = np.asarray(x)
        if digits is not None and x.dtype.kind == "f":
            x = np.vectorize(lambda e: float("%.*g" % (digits, e)))(x)
        out[n] = x.tolist()
    return out


def main():
    cases = []
    for name, backbone, centered, seed in (("gla_centred", oracle.GLA, True, 11),
                                           ("gla_uncentred", oracle.GLA, False, 12),
                                           ("gdn_centred", oracle.GDN, True, 13)):
        P = draw(seed, backbone == oracle.GDN)
        st = initial_state(seed + 100)
        r = oracle.forward(backbone, P["q"], P["k"], P["v"], P["gate"], P["lam"], beta=P["beta"],
                           S0=st["S"], C0=st["C"], m0=st["m"], t0=st["t"], centered=centered)
        cases.append({"name": name, "kind": "forward", "backbone": int(backbone), "centered": centered,
                      "cite": "Algorithm 2; Eq. clean; Eq. read; Sec. 2.2 write rules",
                      "inputs": listify(P), "state": listify(st), "expected": listify(r, 13)})
    for name, backbone, seed in (("decode_gla", oracle.GLA, 21), ("decode_gdn", oracle.GDN, 22)):
        P = draw(seed, backbone == oracle.GDN)
        st = initial_state(seed + 100)
        one = {n: (None if x is None else x[:, 0]) for n, x in P.items()}
        r = oracle.decode_step(backbone, one["q"], one["k"], one["v"], one["gate"], one["lam"],
                               st["S"], st["C"], st["m"], st["t"], beta=one["beta"])
        cases.append({"name": name, "kind": "decode", "backbone": int(backbone), "centered": True,
                      "cite": "Algorithm 2 (one token)", "inputs": listify(one), "state": listify(st),
                      "expected": listify(r, 13)})
    P = draw(31, False)
    st = initial_state(131)
    rng = np.random.RandomState(231)
    grads_in = rounded({"dout": rng.standard_normal((B, T, H, DV)), "dST": rng.standard_normal((B, H, DK, DV)),
                "dCT": rng.standard_normal((B, H, DK, DK)), "dmT": rng.standard_normal((B, H, DK))})
    r = oracle.gla_backward(P["q"], P["k"], P["v"], P["gate"], P["lam"], grads_in["dout"],
                            S0=st["S"], C0=st["C"], m0=st["m"], t0=st["t"], dST=grads_in["dST"],
                            dCT=grads_in["dCT"], dmT=grads_in["dmT"])
    cases.append({"name": "gla_backward", "kind": "gla_backward", "backbone": 0, "centered": True,
                  "cite": "reverse mode of Eq. clean, Eq. read and the GLA write",
                  "inputs": listify({**P, **grads_in}), "state": listify(st), "expected": listify(r, 13)})
    P = draw(41, True)
    rng = np.random.RandomState(241)
    dout = np.round(rng.standard_normal((B, T, H, DV)), 5)
    r = oracle.gdn_backward(P["q"], P["k"], P["v"], P["gate"], P["beta"], P["lam"], dout)
    cases.append({"name": "gdn_backward", "kind": "gdn_backward", "backbone": 1, "centered": True,
                  "cite": "reverse mode of Eq. clean, Eq. read and the gated delta rule",
                  "inputs": listify({**P, "dout": dout}), "state": None, "expected": listify(r, 13)})
    doc = {"about": "fp64 oracle answers on tiny seeded problems (B=1, T=8, H=2, Dk=4, Dv=3); "
                    "written by tests/golden/make_golden.py, which calls only oracle/. The paper "
                    "prints no worked example; these guard the oracle against unjustified change.",
           "cases": cases}
    with open(OUT, "w") as f:
        json.dump(doc, f, indent=None, separators=(",", ":"))
        f.write("\n")


if __name__ == "__main__":
    main()
