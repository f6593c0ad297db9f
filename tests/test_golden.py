"""The oracle against its stored answers (tests/golden/oracle_small.json).

The paper prints no worked numerical example, so the stored answers are the oracle's own,
written by tests/golden/make_golden.py on tiny problems whose inputs are stored with them.
This guards the oracle against silent change: a change to its arithmetic that moves any
of these numbers must regenerate the file in a commit that names the passage of the paper
(or the reading of it) that justifies the change. What pins the oracle to the paper and
to mathematics is the rest of the CPU suite (brute force, closed forms, finite differences)."""
import json
import os

import numpy as np
import pytest

import oracle

PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "oracle_small.json")
with open(PATH) as f:
    CASES = json.load(f)["cases"]


def arr(x, dtype=np.float64):
    return None if x is None else np.asarray(x, dtype=dtype)


def run(case):
    P = {n: arr(x) for n, x in case["inputs"].items()}
    st = case["state"]
    st = None if st is None else {n: arr(x, np.int64 if n == "t" else np.float64) for n, x in st.items()}
    kind, backbone = case["kind"], case["backbone"]
    if kind == "forward":
        return oracle.forward(backbone, P["q"], P["k"], P["v"], P["gate"], P["lam"], beta=P["beta"],
                              S0=st["S"], C0=st["C"], m0=st["m"], t0=st["t"], centered=case["centered"])
    if kind == "decode":
        return oracle.decode_step(backbone, P["q"], P["k"], P["v"], P["gate"], P["lam"], st["S"], st["C"],
                                  st["m"], st["t"], beta=P["beta"])
    if kind == "gla_backward":
        return oracle.gla_backward(P["q"], P["k"], P["v"], P["gate"], P["lam"], P["dout"], S0=st["S"],
                                   C0=st["C"], m0=st["m"], t0=st["t"], dST=P["dST"], dCT=P["dCT"],
                                   dmT=P["dmT"])
    if kind == "gdn_backward":
        return oracle.gdn_backward(P["q"], P["k"], P["v"], P["gate"], P["beta"], P["lam"], P["dout"])
    raise AssertionError(kind)


@pytest.mark.parametrize("case", CASES, ids=[c["name"] for c in CASES])
def test_oracle_matches_stored_answers(oracle_mod, case):
    got = run(case)
    assert set(got) == set(case["expected"]), case["name"]
    for name, want in case["expected"].items():
        want = np.asarray(want)
        have = np.asarray(got[name])
        assert have.shape == want.shape, (case["name"], name)
        if want.dtype.kind in "iu":
            np.testing.assert_array_equal(have, want, err_msg=f"{case['name']}.{name}")
        else:
            # stored to 13 significant digits
            np.testing.assert_allclose(have, want, rtol=1e-11, atol=1e-12 * max(1.0, np.abs(want).max()),
                                       err_msg=f"{case['name']}.{name}")


def test_fixture_covers_every_oracle_entry_point():
    kinds = {c["kind"] for c in CASES}
    assert kinds == {"forward", "decode", "gla_backward", "gdn_backward"}
    assert {c["backbone"] for c in CASES if c["kind"] == "forward"} == {0, 1}
    assert any(not c["centered"] for c in CASES)
