"""The fixtures in tests/golden/ (written from the oracle by
tests/golden/make_golden.py) checked on the CPU: every stored expected value
is re-derived here with exact rational arithmetic from the stored inputs and
the definitions of Table 1's kernels, is exact in its output type, and is
what the oracle still returns."""
import glob
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))
FIXTURES = sorted(glob.glob(os.path.join(HERE, "golden", "*.json")))
NP = {"f32": np.float32, "f64": np.float64, "i32": np.int32}


def load(path):
    with open(path) as f:
        return json.load(f)


def F(v):
    return Fraction(v) if not isinstance(v, list) else [F(x) for x in v]


def matvec(A, x):
    return [sum((a * b for a, b in zip(row, x)), Fraction(0)) for row in A]


def exact(fx):
    """Expected outputs of a fixture from its inputs, as Fractions."""
    if fx["op"] == "bicg":
        A = [row[: fx["N"]] for row in F(fx["A"])]
        At = [list(c) for c in zip(*A)]
        return {"q": matvec(A, F(fx["p"])), "s": matvec(At, F(fx["r"]))}
    A = F(fx["A"])
    if fx["op"] == "gesummv":
        a, b = Fraction(fx["alpha"]), Fraction(fx["beta"])
        ta, tb = matvec(A, F(fx["x"])), matvec(F(fx["B"]), F(fx["x"]))
        return {"y": [a * u + b * v for u, v in zip(ta, tb)]}
    if fx["op"] == "atax":
        t = matvec(A, F(fx["x"]))
        return {"y": matvec([list(c) for c in zip(*A)], t)}
    u1, v1, u2, v2 = F(fx["u1"]), F(fx["v1"]), F(fx["u2"]), F(fx["v2"])
    ah = [[A[i][j] + u1[i] * v1[j] + u2[i] * v2[j] for j in range(fx["N"])]
          for i in range(fx["M"])]
    x = [xi + Fraction(fx["beta"]) * s + zi
         for xi, s, zi in zip(F(fx["x"]), matvec([list(c) for c in zip(*ah)], F(fx["y"])),
                              F(fx["z"]))]
    w = [wi + Fraction(fx["alpha"]) * t for wi, t in zip(F(fx["w"]), matvec(ah, x))]
    return {"A_hat": ah, "x_out": x, "w_out": w}


def flat(v):
    return [y for x in v for y in (flat(x) if isinstance(x, list) else [x])]


def test_fixtures_exist():
    assert len(FIXTURES) >= 6


@pytest.mark.parametrize("path", FIXTURES, ids=os.path.basename)
def test_fixture_matches_exact_arithmetic(path):
    fx = load(path)
    for key, want in exact(fx).items():
        stored = flat(fx[key])
        want = flat(want)
        assert len(stored) == len(want)
        for got, w in zip(stored, want):
            assert Fraction(got) == w, (key, got, w)   # exact, so also representable


@pytest.mark.parametrize("path", FIXTURES, ids=os.path.basename)
def test_oracle_reproduces_fixture(path):
    fx = load(path)
    t = NP[fx["dtype"]]
    if fx["op"] == "bicg":
        q, s = oracle.dualmv(np.array(fx["A"], dtype=t), np.array(fx["p"], dtype=t),
                             np.array(fx["r"], dtype=t), N=fx["N"])
        got = {"q": q, "s": s}
    elif fx["op"] == "gesummv":
        got = {"y": oracle.gesummv(np.array(fx["A"], dtype=t), np.array(fx["B"], dtype=t),
                                   np.array(fx["x"], dtype=t), fx["alpha"], fx["beta"])}
    elif fx["op"] == "atax":
        got = {"y": oracle.atax(np.array(fx["A"], dtype=t), np.array(fx["x"], dtype=t))}
    else:
        args = [np.array(fx[k], dtype=t) for k in ("A", "u1", "v1", "u2", "v2", "w", "x", "y",
                                                  "z")]
        ah, wo, xo = oracle.gemver(*args, fx["alpha"], fx["beta"])
        got = {"A_hat": ah, "w_out": wo, "x_out": xo}
    for key, val in got.items():
        assert flat(np.asarray(val).tolist()) == flat(fx[key]), key
