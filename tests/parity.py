"""Parity helpers: run the CUDA path and the CPU oracle on the same inputs and
compare.  The bar (the functional-equivalence check of Eq. 4, made
quantitative): int32 results bit-exact; floating-point results within
max_i |got_i - want_i| / sum_j |A_ij||x_j| <= 1e-5 (f32) or 1e-12 (f64),
the denominators computed by the oracle."""
from __future__ import annotations

import numpy as np
import torch

import oracle
import paper_2512_22147_gb300 as dm

TOL = {"f32": 1e-5, "f64": 1e-12, "i32": 0.0}
TAG = {torch.float32: "f32", torch.float64: "f64", torch.int32: "i32"}


def scaled_error(got: np.ndarray, want: np.ndarray, denom: np.ndarray) -> float:
    """max |got - want| / denom; where denom is 0 the values must be equal."""
    got = got.astype(np.float64)
    diff = np.abs(got - want)
    zero = denom == 0
    if zero.any() and (diff[zero] != 0).any():
        return float("inf")
    if (~zero).any():
        return float((diff[~zero] / denom[~zero]).max())
    return 0.0


def oracle_outputs(A_store: np.ndarray, p: np.ndarray, r: np.ndarray, N: int):
    """Oracle (q, s) and denominators for one problem (A_store is M x lda)."""
    q, s = oracle.dualmv(A_store, p, r, N=N)
    if A_store.dtype == np.int32:
        return q, s, None, None
    qa, sa = oracle.absdot(A_store, p, r, N=N)
    return q, s, qa, sa


def compare_problem(tag, qg, sg, A_store, p, r, N):
    """Returns the scaled error (0.0 means bit-exact for i32)."""
    q, s, qa, sa = oracle_outputs(A_store, p, r, N)
    if tag == "i32":
        if not (np.array_equal(qg, q) and np.array_equal(sg, s)):
            bad_q = np.flatnonzero(qg != q)[:5]
            bad_s = np.flatnonzero(sg != s)[:5]
            raise AssertionError(f"i32 mismatch: q idx {bad_q}, s idx {bad_s}")
        return 0.0
    return max(scaled_error(qg, q, qa), scaled_error(sg, s, sa))


def run_and_compare(A_store: torch.Tensor, p: torch.Tensor, r: torch.Tensor, N: int,
                    check_fault: bool = True) -> float:
    """A_store is (M, lda) or (B, M, lda) on the GPU; the matrix is its first
    N columns.  Runs dualmv through the C ABI and compares every output with
    the oracle.  Returns the largest scaled error."""
    tag = TAG[A_store.dtype]
    q, s = dm.dualmv(A_store[..., :N], p, r)
    torch.cuda.synchronize()
    if check_fault:
        assert dm.device_fault() == dm.DUALMV_SUCCESS
    An = A_store.cpu().numpy()
    pn, rn = p.cpu().numpy(), r.cpu().numpy()
    qg, sg = q.cpu().numpy(), s.cpu().numpy()
    if A_store.dim() == 2:
        err = compare_problem(tag, qg, sg, An, pn, rn, N)
    else:
        err = 0.0
        for b in range(An.shape[0]):
            pb = pn[b] if pn.ndim == 2 else pn
            rb = rn[b] if rn.ndim == 2 else rn
            err = max(err, compare_problem(tag, qg[b], sg[b], An[b], pb, rb, N))
    assert err <= TOL[tag], f"{tag}: scaled error {err:.3e} > {TOL[tag]:.0e}"
    return err
