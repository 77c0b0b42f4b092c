"""fp64 on the FP32 pipes against the oracle, on inputs built to make its
rounding errors as large as they can be, and all of one sign.

The double-float kernels split every double into a high float (the top
significant bits) and a low float (the rest), form each product from three of
the four partial products, and sum in (high, low) float pairs.  Their error
grows with the size of the low parts, so the worst inputs have the low
mantissa bits all set and the high bits nearly zero: a = 2^e (1 + k 2^-t +
(2^(52-t) - 1) 2^-52) for small k, where t is the split point.  With all of
A, p and r positive every product errs the same way, so nothing cancels.
Two families cover a split after 20 and after 23 stored bits; a third mixes
exponents across the accepted range [2^-40, 2^40).  Each test prints its
measured maximum scaled error (``pytest -s``) and holds it to 1e-12.

The same inputs go through every operation that uses the split: the dual
product (at the full 65536 x 4096 workload shape, for the 65536-term column
sums, and on a 2^20-column matrix for long row sums), ATAX, GESUMMV and
GEMVER (factorised: its passes are the double-float kernels)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2512_22147_gb300 as dm
from parity import TOL, run_and_compare, scaled_error

pytestmark = pytest.mark.gpu
DEV = "cuda:0"

# (split point t in stored mantissa bits, exponent range [lo, hi))
FAMILIES = {
    "low32_set": (20, 0, 1),
    "low29_set": (23, 0, 1),
    "low32_set_mixed_exponents": (20, -20, 20),
}


def adversarial(shape, seed, family):
    """Positive doubles 2^e (1 + k 2^-t + (2^(52-t) - 1) 2^-52), k < 16,
    e uniform in the family's range."""
    t, e_lo, e_hi = FAMILIES[family]
    g = torch.Generator(device=DEV).manual_seed(seed)
    k = torch.randint(0, 16, shape, generator=g, device=DEV, dtype=torch.int64)
    e = torch.randint(e_lo, e_hi, shape, generator=g, device=DEV, dtype=torch.int64)
    low = (1 << (52 - t)) - 1
    bits = ((e + 1023) << 52) | (k << (52 - t)) | low
    return bits.view(torch.float64)


def _report(name, err):
    print(f"adversarial {name}: max scaled error {err:.3e} (bar {TOL['f64']:.0e})")


@pytest.mark.parametrize("family", list(FAMILIES))
def test_dual_product_full_workload_shape(family):
    """65536 x 4096: every s_j sums 65536 same-signed products."""
    M, N = 65536, 4096
    A = adversarial((M, N), 1, family)
    p, r = adversarial((N,), 2, family), adversarial((M,), 3, family)
    err = run_and_compare(A, p, r, N)
    _report(f"dualmv 65536x4096 {family}", err)
    del A
    torch.cuda.empty_cache()


@pytest.mark.parametrize("family", ["low32_set", "low29_set"])
def test_dual_product_long_rows(family):
    """2^20 columns: every q_i sums 2^20 same-signed products over 4096 bands."""
    M, N = 48, 1 << 20
    A = adversarial((M, N), 4, family)
    err = run_and_compare(A, adversarial((N,), 5, family), adversarial((M,), 6, family), N)
    _report(f"dualmv 48x1048576 {family}", err)


@pytest.mark.parametrize("family", ["low32_set", "low29_set"])
def test_atax(family):
    M, N = 8192, 4096
    A, x = adversarial((M, N), 7, family), adversarial((N,), 8, family)
    y = dm.atax(A, x)
    torch.cuda.synchronize()
    assert dm.device_fault() == dm.DUALMV_SUCCESS
    An, xn = A.cpu().numpy(), x.cpu().numpy()
    want = oracle.atax(An, xn, N=N)
    qa, _ = oracle.absdot(An, xn, np.zeros(M), N=N)
    _, den = oracle.absdot(An, np.zeros(N), qa, N=N)
    err = scaled_error(y.cpu().numpy(), want, den)
    _report(f"atax {M}x{N} {family}", err)
    assert err <= TOL["f64"], err


@pytest.mark.parametrize("family", ["low32_set", "low29_set"])
def test_gesummv(family):
    M, N = 4096, 4096
    A, B = adversarial((M, N), 9, family), adversarial((M, N), 10, family)
    x = adversarial((N,), 11, family)
    alpha, beta = 1.5, 0.75
    y = dm.gesummv(A, B, x, alpha=alpha, beta=beta)
    torch.cuda.synchronize()
    An, Bn, xn = A.cpu().numpy(), B.cpu().numpy(), x.cpu().numpy()
    want = oracle.gesummv(An, Bn, xn, alpha, beta, N=N)
    qa, _ = oracle.absdot(An, xn, np.zeros(M), N=N)
    qb, _ = oracle.absdot(Bn, xn, np.zeros(M), N=N)
    err = scaled_error(y.cpu().numpy(), want, alpha * qa + beta * qb)
    _report(f"gesummv {M}x{N} {family}", err)
    assert err <= TOL["f64"], err


@pytest.mark.parametrize("family", ["low32_set", "low29_set"])
def test_gemver_factorised(family):
    M, N = 4096, 4096
    A = adversarial((M, N), 12, family)
    vecs = [adversarial((n,), 13 + i, family)
            for i, n in enumerate((M, N, M, N, M, N, M, N))]   # u1 v1 u2 v2 w x y z
    u1, v1, u2, v2, w, x, y, z = vecs
    host = [t.cpu().numpy() for t in (A, u1, v1, u2, v2, w, x, y, z)]
    alpha, beta = 1.5, 0.75
    old = dm.dualmv_gemver_set_onthefly(0)
    try:
        dm.gemver(A, u1, v1, u2, v2, w, x, y, z, alpha=alpha, beta=beta)
        torch.cuda.synchronize()
    finally:
        dm.dualmv_gemver_set_onthefly(old)
    An, hu1, hv1, hu2, hv2, hw, hx, hy, hz = host
    _, wo, xo = oracle.gemver(An.copy(), hu1, hv1, hu2, hv2, hw.copy(), hx.copy(), hy, hz,
                              alpha, beta, N=N)
    # Denominators: the magnitude of every term of each output (all inputs
    # are positive, so the magnitudes are the values themselves).
    _, sa = oracle.absdot(An, np.zeros(N), hy)
    Xm = hx + beta * (sa + hv1 * (hu1 @ hy) + hv2 * (hu2 @ hy)) + hz
    qa, _ = oracle.absdot(An, Xm, np.zeros(M))
    Wm = hw + alpha * (qa + hu1 * (hv1 @ Xm) + hu2 * (hv2 @ Xm))
    err = max(scaled_error(x.cpu().numpy(), xo, Xm), scaled_error(w.cpu().numpy(), wo, Wm))
    _report(f"gemver {M}x{N} {family}", err)
    assert err <= TOL["f64"], err
