"""GEMVER with update_A: the rows pass that writes A_hat
(dualmv_gemver_update.cuh) against the oracle.

With A 16-byte aligned and a row stride that is a multiple of 16 bytes, a
call with update_A runs the factorised columns pass and x update, then one
kernel that writes A_hat = fma(u2_i, v2_j, fma(u1_i, v1_j, a)) over A and
forms A x from the original A (fp64: in double-float arithmetic).  These
tests check, element by element against the oracle within the dtype's bar
(A_hat, x and w):

  * the path taken (and the fallbacks: a row stride off the 16-byte grid, a
    base off it, the on-the-fly setting);
  * widths around the kernels' bands (fp64: 512 columns, fp32: 1024; ragged
    last band, one column, a band and one);
  * values outside [2^-40, 2^40) in rows of A and in the new x (native fp64
    for those rows or that band), and zero rows;
  * repeated calls giving the same bits, and the padding columns untouched;
  * the adversarial all-positive inputs of the fp64 error-bound tests;
  * vectors long enough for the dot products' compensated thread sums.
The full-size workload (gemver_update_f64_8192x8192) runs in
test_gpu_ops.py with the other operation workloads."""
import numpy as np
import pytest
import torch

import oracle
import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import inputs
from parity import TOL, scaled_error
from test_gpu_f64_adversarial import adversarial
from test_gpu_ops import _w, check_gemver

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _ops(M, N, lda, seed, dtype="f64"):
    return inputs.generate_gemver(_w("gemver", dtype, M, N, lda, seed), DEV)


@pytest.mark.parametrize("M,N,pad", [(300, 512, 0), (300, 511, 1), (300, 513, 1), (64, 1, 1),
                                     (200, 1025, 1), (2, 4096, 0), (4097, 300, 2)])
def test_update_split_matches_oracle(M, N, pad):
    err = check_gemver(_ops(M, N, N + pad, M * 7 + N), N, 1.5, -0.75, True, "f64")
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_UPDATE_SPLIT
    print(f"gemver update_A {M}x{N}+{pad}: {err:.3e}")


@pytest.mark.parametrize("M,N,pad", [(300, 1024, 0), (300, 1023, 1), (300, 1025, 3), (64, 1, 3),
                                     (200, 2049, 3), (2, 8192, 0), (4097, 300, 0)])
def test_update_f32_matches_oracle(M, N, pad):
    err = check_gemver(_ops(M, N, N + pad, M * 5 + N, "f32"), N, 1.5, -0.75, True, "f32")
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_UPDATE_SPLIT
    print(f"gemver f32 update_A {M}x{N}+{pad}: {err:.3e}")


def test_path_taken_and_fallbacks():
    A, u1, v1, u2, v2, w, x, y, z = _ops(100, 300, 301, 3)
    args = (u1, v1, u2, v2, w.clone(), x.clone(), y, z)
    dm.gemver(A.clone()[:, :300], *args, update_A=True)          # lda 301: odd
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_ONTHEFLY
    B = torch.empty(100, 303, dtype=torch.float64, device=DEV)
    B[:, 1:301] = A[:, :300]
    dm.gemver(B[:, 1:301], *args, update_A=True)                  # base 8 bytes off the grid
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_ONTHEFLY
    C = torch.empty(100, 302, dtype=torch.float64, device=DEV)
    C[:, :300] = A[:, :300]
    dm.gemver(C[:, :300], *args, update_A=True)                   # lda 302: even
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_UPDATE_SPLIT
    dm.gemver(C[:, :300], *args, update_A=False)
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_FACTORED
    old = dm.dualmv_gemver_set_onthefly(1)
    try:
        dm.gemver(C[:, :300], *args, update_A=True)
        assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_ONTHEFLY
    finally:
        dm.dualmv_gemver_set_onthefly(old)
    f = [t.float() for t in (C[:, :300],) + args]
    dm.gemver(f[0], *f[1:], update_A=True)                       # fp32, 1200-byte rows
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_UPDATE_SPLIT
    F = torch.empty(100, 302, dtype=torch.float32, device=DEV)   # 1208-byte rows
    F[:, :300] = f[0]
    dm.gemver(F[:, :300], *f[1:], update_A=True)
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_ONTHEFLY
    dm.gemver(C[:0, :0], u1[:0], v1[:0], u2[:0], v2[:0], w[:0], x[:0], y[:0], z[:0],
              update_A=True)
    assert dm.dualmv_gemver_last_path() == -1


@pytest.mark.parametrize("case", ["huge_rows", "tiny_rows", "zero_rows", "x_out_of_range"])
def test_out_of_range_values(case):
    M, N = 700, 1100
    A, u1, v1, u2, v2, w, x, y, z = _ops(M, N, N, 11)
    if case == "huge_rows":
        A[10:13, :] *= 1.0e13          # |a| beyond 2^40
    elif case == "tiny_rows":
        A[500:504, 600:] *= 1.0e-14    # |a| below 2^-40 in the second and third bands
    elif case == "zero_rows":
        A[20:40, :] = 0.0              # zeros stay on the double-float path
    else:
        z[520:530] = 1.0e14            # the new x beyond 2^40 in the second band
    check_gemver((A, u1, v1, u2, v2, w, x, y, z), N, 1.5, -0.75, True, "f64")
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_UPDATE_SPLIT
    assert dm.device_fault() == dm.DUALMV_SUCCESS


@pytest.mark.parametrize("dtype", ["f64", "f32"])
def test_repeated_calls_are_bit_identical(dtype):
    M, N = 1500, 2000
    ops = _ops(M, N, N + 4, 5, dtype)
    outs = []
    for _ in range(2):
        A, u1, v1, u2, v2, w, x, y, z = (t.clone() for t in ops)
        dm.gemver(A[:, :N], u1, v1, u2, v2, w, x, y, z, alpha=0.5, beta=2.0, update_A=True)
        outs.append((A, w, x))
    torch.cuda.synchronize()
    A0, A1 = outs[0][0], outs[1][0]
    assert torch.equal(A0[:, :N], A1[:, :N])
    for a, b in zip(outs[0][1:], outs[1][1:]):
        assert torch.equal(a, b)
    # The padding columns (NaN in the generated storage) are untouched.
    assert torch.equal(A0[:, N:].isnan(), ops[0][:, N:].isnan())
    assert bool(A0[:, N:].isnan().all())


@pytest.mark.parametrize("dtype", ["f64", "f32"])
@pytest.mark.parametrize("M,N", [(1048600, 3), (3, 1048600)])
@pytest.mark.parametrize("update_A", [False, True])
def test_long_vectors(dtype, M, N, update_A):
    """Vectors past 64 x 256 x 64 elements: each thread of the dot-product
    kernels then has more than 64 elements of its chunk and sums them
    compensated (at most 64 it uses plain FMAs): u . y when M is long,
    v . x when N is long."""
    err = check_gemver(_ops(M, N, N + (1 if N == 3 else 0), M + N, dtype), N, 1.5, -0.75,
                       update_A, dtype)
    print(f"gemver {dtype} {M}x{N} update_A={update_A}: {err:.3e}")


@pytest.mark.parametrize("dtype", ["f64", "f32"])
def test_back_to_back_calls_see_the_previous_writes(dtype):
    """The columns pass reads A and y without waiting for the u . y kernel
    beside it (it waits for that grid only before it exits); every grid
    queued before the call has completed when it starts.  A call right after
    one that wrote A_hat over A, and after a kernel that rewrote y, gives
    the bits of the same calls with a synchronisation between them."""
    ops = _ops(1500, 2000, 2000, 77, dtype)

    def sequence(sync):
        A, u1, v1, u2, v2, w, x, y, z = (t.clone() for t in ops)
        torch.cuda.synchronize()
        dm.gemver(A, u1, v1, u2, v2, w, x, y, z, alpha=1.5, beta=0.5, update_A=True)
        if sync:
            torch.cuda.synchronize()
        y.mul_(-0.5)
        if sync:
            torch.cuda.synchronize()
        dm.gemver(A, u1, v1, u2, v2, w, x, y, z, alpha=1.5, beta=0.5)
        dm.gemver(A, u1, v1, u2, v2, w, x, y, z, alpha=0.5, beta=2.0, update_A=True)
        torch.cuda.synchronize()
        return A, w, x

    for _ in range(3):
        for t0, t1 in zip(sequence(False), sequence(True)):
            assert torch.equal(t0, t1)


@pytest.mark.parametrize("family", ["low32_set", "low29_set"])
def test_adversarial_inputs(family):
    """All inputs positive with the low mantissa bits set: the double-float
    errors all of one sign."""
    M, N = 2048, 4096
    A = adversarial((M, N), 21, family)
    vecs = [adversarial((n,), 22 + i, family) for i, n in enumerate((M, N, M, N, M, N, M, N))]
    u1, v1, u2, v2, w, x, y, z = vecs
    host = [t.cpu().numpy() for t in (A, u1, v1, u2, v2, w, x, y, z)]
    alpha, beta = 1.5, 0.75
    dm.gemver(A, u1, v1, u2, v2, w, x, y, z, alpha=alpha, beta=beta, update_A=True)
    torch.cuda.synchronize()
    assert dm.dualmv_gemver_last_path() == dm.DUALMV_GEMVER_UPDATE_SPLIT
    An, hu1, hv1, hu2, hv2, hw, hx, hy, hz = host
    ah, wo, xo = oracle.gemver(An.copy(), hu1, hv1, hu2, hv2, hw.copy(), hx.copy(), hy, hz,
                               alpha, beta, N=N)
    _, sa = oracle.absdot(An, np.zeros(N), hy)
    Xm = hx + beta * (sa + hv1 * (hu1 @ hy) + hv2 * (hu2 @ hy)) + hz
    qa, _ = oracle.absdot(An, Xm, np.zeros(M))
    Wm = hw + alpha * (qa + hu1 * (hv1 @ Xm) + hu2 * (hv2 @ Xm))
    Am = An + np.outer(hu1, hv1) + np.outer(hu2, hv2)
    err = max(scaled_error(x.cpu().numpy(), xo, Xm), scaled_error(w.cpu().numpy(), wo, Wm),
              scaled_error(A.cpu().numpy().ravel(), ah.ravel(), Am.ravel()))
    print(f"adversarial gemver update_A {family}: {err:.3e}")
    assert err <= TOL["f64"], err
