"""Writes the small text fixtures in this folder from the CPU oracle.

The paper prints no worked example for these kernels, so the expected values
here are not the paper's: they are the oracle's, for the operations of
Table 1 (BICG q = A p, s = A^T r; GESUMMV; ATAX; GEMVER) on small seeded
inputs whose entries are small integers or dyadic rationals, so that every
expected value is exact in its output type.  The tests re-derive each one
with exact rational arithmetic, independently of the oracle.

    python tests/golden/make_golden.py        (from the repository root)
"""
from __future__ import annotations

import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402

INT32_MIN = -(2 ** 31)


def _ints(rng, shape, lo=-8, hi=8):
    return rng.integers(lo, hi + 1, size=shape)


def _dyadic(rng, shape):
    """k / 2^e with |k| < 64 and e in [0, 3]: products are multiples of 2^-6
    below 2^12, so a sum of up to 16 of them needs at most 22 significant
    bits and is exact in fp32, in any order."""
    return rng.integers(-63, 64, size=shape) / 2.0 ** rng.integers(0, 4, size=shape)


def bicg_cases():
    rng = np.random.default_rng(20251222)
    out = []
    # int32, padded rows (the padding holds INT32_MIN and is never read)
    M, N, lda = 7, 11, 13
    A = np.full((M, lda), INT32_MIN, dtype=np.int32)
    A[:, :N] = _ints(rng, (M, N))
    p, r = _ints(rng, N).astype(np.int32), _ints(rng, M).astype(np.int32)
    q, s = oracle.dualmv(A, p, r, N=N)
    out.append(("bicg_i32_7x11_lda13", "i32", A, N, p, r, q, s))
    # fp64 and fp32 with dyadic entries: every product and sum is exact
    for tag, dt in (("f64", np.float64), ("f32", np.float32)):
        M, N = 5, 9
        A = _dyadic(rng, (M, N)).astype(dt)
        p, r = _dyadic(rng, N).astype(dt), _dyadic(rng, M).astype(dt)
        q, s = oracle.dualmv(A, p, r, N=N)
        out.append((f"bicg_{tag}_5x9_dyadic", tag, A, N, p, r, q, s))
    return out


def write(name, payload):
    with open(os.path.join(HERE, name + ".json"), "w") as f:
        json.dump(payload, f, indent=None, separators=(",", ":"))
        f.write("\n")


def main():
    for name, tag, A, N, p, r, q, s in bicg_cases():
        write(name, {"op": "bicg", "dtype": tag, "M": int(A.shape[0]), "N": int(N),
                     "lda": int(A.shape[1]), "A": A.tolist(), "p": p.tolist(),
                     "r": r.tolist(), "q": q.tolist(), "s": s.tolist(),
                     "source": "oracle.dualmv (oracle/oracle.c), BICG of Table 1"})
    rng = np.random.default_rng(7)
    M, N = 6, 10
    A = _ints(rng, (M, N)).astype(np.float64)
    B = _ints(rng, (M, N)).astype(np.float64)
    x = _ints(rng, N).astype(np.float64)
    y = oracle.gesummv(A, B, x, 3.0, -2.0)
    write("gesummv_f64_6x10", {"op": "gesummv", "dtype": "f64", "M": M, "N": N,
                               "alpha": 3.0, "beta": -2.0, "A": A.tolist(), "B": B.tolist(),
                               "x": x.tolist(), "y": y.tolist(),
                               "source": "oracle.gesummv, GESUMMV of Table 1"})
    y = oracle.atax(A, x)
    write("atax_f64_6x10", {"op": "atax", "dtype": "f64", "M": M, "N": N, "A": A.tolist(),
                            "x": x.tolist(), "y": y.tolist(),
                            "source": "oracle.atax, ATAX of Table 1"})
    u1, u2, w, yv = (_ints(rng, M).astype(np.float64) for _ in range(4))
    v1, v2, xv, z = (_ints(rng, N).astype(np.float64) for _ in range(4))
    ah, wo, xo = oracle.gemver(A, u1, v1, u2, v2, w, xv, yv, z, 2.0, 0.5)
    write("gemver_f64_6x10", {"op": "gemver", "dtype": "f64", "M": M, "N": N, "alpha": 2.0,
                              "beta": 0.5, "A": A.tolist(), "u1": u1.tolist(),
                              "v1": v1.tolist(), "u2": u2.tolist(), "v2": v2.tolist(),
                              "w": w.tolist(), "x": xv.tolist(), "y": yv.tolist(),
                              "z": z.tolist(), "A_hat": ah.tolist(), "w_out": wo.tolist(),
                              "x_out": xo.tolist(),
                              "source": "oracle.gemver, GEMVER of Table 1"})


if __name__ == "__main__":
    main()
