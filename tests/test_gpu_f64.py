"""fp64 on the FP32 pipes (double-float emulation) against the oracle and
against native fp64 FMA, including the rows that must fall back to native
fp64: zeros, values outside [2^-40, 2^40), subnormals and large ranges."""
import numpy as np
import pytest
import torch

import paper_2512_22147_gb300 as dm
from parity import TOL, run_and_compare

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _rand(shape, seed, scale_exp=0):
    g = torch.Generator(device=DEV).manual_seed(seed)
    x = torch.empty(shape, dtype=torch.float64, device=DEV).normal_(0, 1, generator=g)
    return x * (2.0 ** scale_exp)


@pytest.fixture
def native_f64():
    def run(fn):
        old = dm.dualmv_set_path(dm.DUALMV_PATH_TMA_NATIVE_F64)
        try:
            return fn()
        finally:
            dm.dualmv_set_path(old)
    return run


@pytest.mark.parametrize("M,N", [(1000, 4096), (4099, 777), (33, 100000)])
def test_emulated_matches_oracle(M, N):
    A = _rand((M, N), 1)
    run_and_compare(A, _rand((N,), 2), _rand((M,), 3), N)


def test_emulated_and_native_agree(native_f64):
    M, N = 3000, 5000
    A, p, r = _rand((M, N), 4), _rand((N,), 5), _rand((M,), 6)
    q1, s1 = dm.dualmv(A, p, r)
    q2, s2 = native_f64(lambda: dm.dualmv(A, p, r))
    den_q = (A.abs() @ p.abs())
    den_s = (r.abs() @ A.abs())
    assert float(((q1 - q2).abs() / den_q).max()) <= 2 * TOL["f64"]
    assert float(((s1 - s2).abs() / den_s).max()) <= 2 * TOL["f64"]


def test_native_path_matches_oracle(native_f64):
    M, N = 700, 1300
    A = _rand((M, N), 7)
    native_f64(lambda: run_and_compare(A, _rand((N,), 8), _rand((M,), 9), N))


@pytest.mark.parametrize("density", [0.0, 0.01, 0.5])
def test_zero_heavy_matrices(density):
    """Zeros trip the cheap range bound; the exact re-check keeps the
    emulated result."""
    M, N = 900, 2100
    A = _rand((M, N), 10)
    g = torch.Generator(device=DEV).manual_seed(11)
    keep = torch.rand((M, N), generator=g, device=DEV) < density
    A = torch.where(keep, A, torch.zeros_like(A))
    p, r = _rand((N,), 12), _rand((M,), 13)
    p[::7] = 0.0
    r[::5] = 0.0
    run_and_compare(A, p, r, N)


@pytest.mark.parametrize("kind", ["huge", "tiny", "subnormal", "mixed_rows", "big_p", "small_r"])
def test_out_of_range_values_fall_back(kind):
    """Rows with values outside [2^-40, 2^40) are computed in native fp64;
    all other rows keep the emulated path; every output within tolerance."""
    M, N = 640, 1536
    A, p, r = _rand((M, N), 20), _rand((N,), 21), _rand((M,), 22)
    if kind == "huge":
        A[5, 100] = 3.0e100
        A[300, :] *= 2.0 ** 60
    elif kind == "tiny":
        A[7, 7] = 1.0e-200
        A[400, :] *= 2.0 ** -70
    elif kind == "subnormal":
        A[9, 1000] = 5e-324
        A[10, :17] = 2.2e-310
    elif kind == "mixed_rows":
        A[::37, :] *= 1.0e60
        A[1::41, :] *= 1.0e-60
    elif kind == "big_p":
        p[1234] = 1.0e30
    elif kind == "small_r":
        r[77] = 1.0e-30
    run_and_compare(A, p, r, N)


def test_ill_conditioned_rows():
    """Heavy cancellation: exact sums near zero while sum |a x| is large."""
    M, N = 512, 4096
    base = _rand((M, N // 2), 30)
    A = torch.cat([base, -base], dim=1).contiguous()
    p = torch.ones(N, dtype=torch.float64, device=DEV)
    r = _rand((M,), 31)
    run_and_compare(A, p, r, N)
