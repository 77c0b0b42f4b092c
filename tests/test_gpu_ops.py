"""GESUMMV, ATAX and GEMVER (Table 1 of the paper; GESUMMV and GEMVER also
Table 2) on the GPU through the C ABI, against the CPU oracle.

Tolerance, as for the dual product, relative to the magnitude of each
output's terms: GESUMMV |y_i - y^_i| <= tol (|alpha| sum_j |A_ij||x_j| +
|beta| sum_j |B_ij||x_j|); ATAX |y_j - y^_j| <= tol sum_i |A_ij| sum_k
|A_ik||x_k| (the error of tmp = A x propagates through A^T).  tol = 1e-5
(f32) and 1e-12 (f64)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import inputs
from parity import TOL, scaled_error

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
TAGS = {"f32": torch.float32, "f64": torch.float64}


@pytest.fixture(params=[dm.DUALMV_PATH_TMA, dm.DUALMV_PATH_DIRECT], ids=["tma", "direct"])
def path(request):
    old = dm.dualmv_set_path(request.param)
    yield request.param
    dm.dualmv_set_path(old)


@pytest.fixture(params=[0, 1], ids=["one_read", "two_pass"])
def atax_mode(request):
    old = dm.dualmv_atax_set_two_pass(request.param)
    yield request.param
    dm.dualmv_atax_set_two_pass(old)


def _w(op, dtype, M, N, lda, seed):
    dist = "uniform" if dtype == "f32" else "normal"
    return inputs.Workload(op, dtype, M, N, lda, dist, seed, op=op)


def check_gesummv(A, B, x, N, alpha, beta, dtype):
    y = dm.gesummv(A[:, :N], B[:, :N], x, alpha=alpha, beta=beta)
    torch.cuda.synchronize()
    An, Bn, xn = A.cpu().numpy(), B.cpu().numpy(), x.cpu().numpy()
    want = oracle.gesummv(An, Bn, xn, alpha, beta, N=N)
    qa, _ = oracle.absdot(An, xn, np.zeros(An.shape[0], An.dtype), N=N)
    qb, _ = oracle.absdot(Bn, xn, np.zeros(Bn.shape[0], Bn.dtype), N=N)
    den = abs(alpha) * qa + abs(beta) * qb
    err = scaled_error(y.cpu().numpy(), want, den)
    assert err <= TOL[dtype], err
    return err


def check_atax(A, x, N, dtype):
    y = dm.atax(A[:, :N], x)
    torch.cuda.synchronize()
    An, xn = A.cpu().numpy(), x.cpu().numpy()
    want = oracle.atax(An, xn, N=N)
    qa, _ = oracle.absdot(An, xn, np.zeros(An.shape[0], An.dtype), N=N)
    _, den = oracle.absdot(An.astype(np.float64), np.zeros(N), qa, N=N)
    err = scaled_error(y.cpu().numpy(), want, den)
    assert err <= TOL[dtype], err
    return err


@pytest.mark.parametrize("dtype", ["f32", "f64"])
@pytest.mark.parametrize("M,N,pad", [(1000, 3000, 0), (3001, 257, 5), (1, 1, 0), (77, 1000, 3),
                                     (2048, 64, 0)])
def test_gesummv_matches_oracle(dtype, M, N, pad, path):
    A, B, x = inputs.generate_gesummv(_w("gesummv", dtype, M, N, N + pad, M + N), DEV)
    check_gesummv(A, B, x, N, 0.75, -1.25, dtype)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
@pytest.mark.parametrize("M,N,pad", [(1000, 3000, 0), (3001, 257, 5), (1, 1, 0), (77, 1000, 3),
                                     (2048, 64, 0), (513, 5000, 4), (1030, 2048, 0)])
def test_atax_matches_oracle(dtype, M, N, pad, path, atax_mode):
    A, x = inputs.generate_atax(_w("atax", dtype, M, N, N + pad, 3 * M + N), DEV)
    check_atax(A, x, N, dtype)


# fp32 widths for the single-read path: clusters of 1, 2, 4, 5, 10 and 16
# CTAs (16 sub-bands of 256 columns per CTA), and one too wide for a cluster
# of 16 (two passes).
@pytest.mark.parametrize("M,N", [(4096, 16384), (300, 20000), (1000, 700), (1999, 4100),
                                 (33, 6144), (256, 40000), (9, 16384), (17, 65536),
                                 (40, 70000)])
def test_atax_one_read_widths(M, N, atax_mode):
    A, x = inputs.generate_atax(_w("atax", "f32", M, N, N, 7 * M + N), DEV)
    check_atax(A, x, N, "f32")


def test_atax_one_read_path_runs():
    """The single-read path adds the row sums in another order than the
    two-pass path, so on random data their bits differ: the cluster kernel
    really ran.  Both are checked against the oracle elsewhere."""
    A, x = inputs.generate_atax(_w("atax", "f32", 4096, 4096, 4096, 5), DEV)
    old = dm.dualmv_atax_set_two_pass(0)
    try:
        y1 = dm.atax(A, x)
        dm.dualmv_atax_set_two_pass(1)
        y2 = dm.atax(A, x)
        torch.cuda.synchronize()
    finally:
        dm.dualmv_atax_set_two_pass(old)
    assert not torch.equal(y1, y2)
    assert dm.device_fault() == dm.DUALMV_SUCCESS


# The one-read path's stated limits (include/dualmv.h): a cluster of at most
# 16 CTAs, each 4096 (fp32) or 2048 (fp64) columns wide, and TMA-aligned rows.
@pytest.mark.parametrize("dtype,limit", [("f32", 65536), ("f64", 32768)])
def test_atax_width_limit_chooses_the_path(dtype, limit):
    """Just inside the width limit the cluster kernel reads A once; one
    column past it (rows still 16-byte aligned), A is read twice."""
    per16 = 4 if dtype == "f32" else 2
    for N, want in ((limit, dm.DUALMV_ATAX_ONE_READ),
                    (limit + 1, dm.DUALMV_ATAX_TWO_PASS)):
        lda = (N + per16 - 1) // per16 * per16
        A, x = inputs.generate_atax(_w("atax", dtype, 9, N, lda, N), DEV)
        check_atax(A, x, N, dtype)
        assert dm.dualmv_atax_last_path() == want, (N, dm.dualmv_atax_last_path())


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_atax_alignment_and_override_choose_two_passes(dtype):
    """Rows whose stride or base is not 16-byte aligned, and the two-pass
    override, take two passes; the aligned problem takes one read."""
    M, N = 300, 1000
    A, x = inputs.generate_atax(_w("atax", dtype, M, N + 8, N + 8, 17), DEV)
    check_atax(A, x[:N].contiguous(), N, dtype)
    assert dm.dualmv_atax_last_path() == dm.DUALMV_ATAX_ONE_READ
    A1, x1 = inputs.generate_atax(_w("atax", dtype, M, N, N + 1, 18), DEV)
    check_atax(A1, x1, N, dtype)                      # odd row stride
    assert dm.dualmv_atax_last_path() == dm.DUALMV_ATAX_TWO_PASS
    y = dm.atax(A[:, 1:N + 1], x[:N].contiguous())    # base one element in
    torch.cuda.synchronize()
    assert dm.dualmv_atax_last_path() == dm.DUALMV_ATAX_TWO_PASS
    old = dm.dualmv_atax_set_two_pass(1)
    try:
        check_atax(A, x[:N].contiguous(), N, dtype)
        assert dm.dualmv_atax_last_path() == dm.DUALMV_ATAX_TWO_PASS
    finally:
        dm.dualmv_atax_set_two_pass(old)
    assert y.shape == (N,)


def test_atax_one_read_is_deterministic():
    A, x = inputs.generate_atax(_w("atax", "f32", 3000, 9000, 9000, 6), DEV)
    y1 = dm.atax(A, x)
    y2 = dm.atax(A, x)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)


# fp64 widths for the single-read path (8 sub-bands of 256 columns per CTA):
# clusters of 1, 2, 3, 4, 8 and 10 CTAs, and one too wide for a cluster of
# 16 (two passes).
@pytest.mark.parametrize("M,N", [(1000, 700), (2049, 3000), (301, 5000), (4096, 8192),
                                 (517, 16384), (64, 20000), (40, 40000)])
def test_atax_f64_one_read_widths(M, N, atax_mode):
    A, x = inputs.generate_atax(_w("atax", "f64", M, N, N, 11 * M + N), DEV)
    check_atax(A, x, N, "f64")


def test_atax_f64_one_read_path_runs():
    """As for fp32: the cluster kernel's summation order differs from the
    two-pass path's, so its bits differ on random data."""
    A, x = inputs.generate_atax(_w("atax", "f64", 2048, 4096, 4096, 15), DEV)
    old = dm.dualmv_atax_set_two_pass(0)
    try:
        y1 = dm.atax(A, x)
        dm.dualmv_atax_set_two_pass(1)
        y2 = dm.atax(A, x)
        torch.cuda.synchronize()
    finally:
        dm.dualmv_atax_set_two_pass(old)
    assert not torch.equal(y1, y2)
    assert dm.device_fault() == dm.DUALMV_SUCCESS


def test_atax_f64_one_read_is_deterministic():
    A, x = inputs.generate_atax(_w("atax", "f64", 3000, 5000, 5000, 16), DEV)
    y1 = dm.atax(A, x)
    y2 = dm.atax(A, x)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)


@pytest.mark.parametrize("case", ["zeros", "a_huge_tiny", "x_zero_huge", "t_out_of_range",
                                  "zero_rows"])
def test_atax_f64_one_read_range(case, atax_mode):
    """The double-float cluster kernel is exact only for |a|, |x|, |t| in
    [2^-40, 2^40) or zero: zeros stay on the fast path, anything else sends
    the stripe (or the warp) to native fp64.  Every case matches the
    oracle."""
    M, N = 1500, 3000
    A, x = inputs.generate_atax(_w("atax", "f64", M, N, N + 2, 17), DEV)
    if case == "zeros":
        A[:, ::3] = 0.0
        A[::5, :] = 0.0
        x[::7] = 0.0
    elif case == "a_huge_tiny":
        A[13, 100] = 3.0e20
        A[700, 2500] = -2.5e-20
        A[1499, 2999] = 1.0e100     # t of row 1499 ~ 1e100; y stays finite
    elif case == "x_zero_huge":
        x[::11] = 0.0
        x[1024] = 7.0e15
    elif case == "t_out_of_range":
        # a stays in range; t does not.  Rows 40-43: |a| ~ 1e11, so t is near
        # 1e11 * sqrt(N) > 2^40.  Row 900: two entries whose products cancel
        # to a rounding residue, t ~ 1e-16 < 2^-40.
        A[40:44, :] *= 1.0e11
        A[900, :] = 0.0
        A[900, 0] = 1.0
        A[900, 1] = -(x[0] / x[1])
    elif case == "zero_rows":
        A[200:208, :] = 0.0         # t exactly zero
    check_atax(A, x, N, "f64")
    assert dm.device_fault() == dm.DUALMV_SUCCESS


def check_gemver(ops, N, alpha, beta, update_A, dtype):
    """GEMVER on the GPU vs the oracle.  Denominators (terms' magnitudes):
    A_hat: |A| + |u1 v1| + |u2 v2|;  x: |x| + |beta| sum_i Am_ij |y_i| + |z|;
    w: |w| + |alpha| sum_j Am_ij Xm_j (the new x's error carried into w)."""
    A, u1, v1, u2, v2, w, x, y, z = ops
    host = [t.cpu().numpy() for t in (A, u1, v1, u2, v2, w, x, y, z)]
    wg, xg = w.clone(), x.clone()
    Ag = A.clone()
    dm.gemver(Ag[:, :N], u1, v1, u2, v2, wg, xg, y, z, alpha=alpha, beta=beta,
              update_A=update_A)
    torch.cuda.synchronize()
    ah, wo, xo = oracle.gemver(host[0], *host[1:], alpha, beta, N=N)
    An = host[0].astype(np.float64)[:, :N]
    au1, av1, au2, av2, aw, ax, ay, az = (np.abs(v.astype(np.float64)) for v in host[1:])
    zeros_m = np.zeros(An.shape[0])
    _, sa = oracle.absdot(np.ascontiguousarray(An), np.zeros(N), ay)
    Xm = ax + abs(beta) * (sa + av1 * (au1 @ ay) + av2 * (au2 @ ay)) + az
    qa, _ = oracle.absdot(np.ascontiguousarray(An), Xm, zeros_m)
    Wm = aw + abs(alpha) * (qa + au1 * (av1 @ Xm) + au2 * (av2 @ Xm))
    err = max(scaled_error(xg.cpu().numpy(), xo, Xm), scaled_error(wg.cpu().numpy(), wo, Wm))
    if update_A:
        Am = np.abs(An) + np.outer(au1, av1) + np.outer(au2, av2)
        got = Ag[:, :N].cpu().numpy()
        err = max(err, scaled_error(got.ravel(), ah.ravel(), Am.ravel()))
        assert torch.equal(Ag[:, N:].cpu().isnan(), A[:, N:].cpu().isnan())  # padding untouched
    assert err <= TOL[dtype], err
    return err


@pytest.fixture(params=[0, 1], ids=["factored", "onthefly"])
def gemver_mode(request):
    old = dm.dualmv_gemver_set_onthefly(request.param)
    yield request.param
    dm.dualmv_gemver_set_onthefly(old)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
@pytest.mark.parametrize("M,N,pad", [(1000, 3000, 0), (3001, 257, 5), (1, 1, 0), (77, 1000, 3),
                                     (1, 5000, 0), (5000, 1, 0)])
@pytest.mark.parametrize("update_A", [False, True])
def test_gemver_matches_oracle(dtype, M, N, pad, update_A, path, gemver_mode):
    w = _w("gemver", dtype, M, N, N + pad, 5 * M + N)
    check_gemver(inputs.generate_gemver(w, DEV), N, 1.5, -0.75, update_A, dtype)


@pytest.mark.parametrize("name", list(inputs.OP_WORKLOADS))
def test_op_workloads_full_size(name):
    w = inputs.OP_WORKLOADS[name]
    if w.op == "gesummv":
        A, B, x = inputs.generate_gesummv(w, DEV)
        err = check_gesummv(A, B, x, w.N, 1.5, 1.2, w.dtype)
        del B
    elif w.op == "atax":
        A, x = inputs.generate_atax(w, DEV)
        err = check_atax(A, x, w.N, w.dtype)
    else:
        ops = inputs.generate_gemver(w, DEV)
        err = check_gemver(ops, w.N, 1.5, 1.2, w.update_a, w.dtype)
        A = x = ops
    print(f"{name}: max scaled error {err:.3e}")
    del A, x
    torch.cuda.empty_cache()


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_gesummv_closed_forms(dtype, path):
    """Both row passes are deterministic, so with B = A and alpha = beta = 1
    the result is exactly twice the alpha = 1, B = 0 result, and alpha = 4
    gives exactly four times it (powers of two scale exactly)."""
    M, N = 513, 1300
    A, _, x = inputs.generate_gesummv(_w("gesummv", dtype, M, N, N, 3), DEV)
    Z = torch.zeros_like(A)
    y_one = dm.gesummv(A, Z, x, alpha=1.0, beta=0.0)
    y_two = dm.gesummv(A, A, x, alpha=1.0, beta=1.0)
    y_four = dm.gesummv(A, Z, x, alpha=4.0, beta=3.0)
    assert torch.equal(y_two, 2 * y_one) and torch.equal(y_four, 4 * y_one)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_atax_permutation_is_exact(dtype, atax_mode):
    n = 900
    g = torch.Generator(device="cpu").manual_seed(9)
    perm = torch.randperm(n, generator=g)
    P = torch.zeros(n, n, dtype=TAGS[dtype])
    P[torch.arange(n), perm] = 1.0
    x = torch.empty(n, dtype=TAGS[dtype]).uniform_(-1, 1, generator=g)
    y = dm.atax(P.to(DEV), x.to(DEV))
    if dtype == "f64":
        assert float(((y.cpu() - x).abs() / x.abs()).max()) <= 2.0 ** -43
    else:
        assert torch.equal(y.cpu(), x)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_empty_shapes(dtype):
    t = TAGS[dtype]
    A = torch.empty(4, 0, dtype=t, device=DEV)
    y = dm.gesummv(A, A, torch.empty(0, dtype=t, device=DEV))
    assert (y.cpu() == 0).all() and y.shape == (4,)
    A = torch.empty(0, 6, dtype=t, device=DEV)
    y = dm.atax(A, torch.ones(6, dtype=t, device=DEV))
    assert (y.cpu() == 0).all() and y.shape == (6,)


def test_no_device_fault_recorded():
    assert dm.device_fault() == dm.DUALMV_SUCCESS


# ---------------------------------------------------------- golden fixtures ---

import glob as _glob
import json as _json
import os as _os

_GOLDEN = sorted(_glob.glob(_os.path.join(_os.path.dirname(_os.path.abspath(__file__)),
                                          "golden", "*.json")))
_T = {"f32": torch.float32, "f64": torch.float64, "i32": torch.int32}


@pytest.mark.parametrize("fixture", _GOLDEN, ids=_os.path.basename)
def test_golden_fixture_exact(fixture, path):
    """Every stored value is exact in its type, so any summation order gives
    it: the CUDA path must reproduce the fixture exactly, on both paths."""
    with open(fixture) as f:
        fx = _json.load(f)
    t = _T[fx["dtype"]]

    def dev(key):
        return torch.tensor(fx[key], dtype=t, device=DEV)

    if fx["op"] == "bicg":
        q, s = dm.dualmv(dev("A")[:, : fx["N"]], dev("p"), dev("r"))
        got = {"q": q, "s": s}
    elif fx["op"] == "gesummv":
        got = {"y": dm.gesummv(dev("A"), dev("B"), dev("x"), alpha=fx["alpha"],
                               beta=fx["beta"])}
    elif fx["op"] == "atax":
        got = {"y": dm.atax(dev("A"), dev("x"))}
    else:  # with write-back (on the fly), then without (factorised)
        A, w, x = dev("A"), dev("w"), dev("x")
        dm.gemver(A, dev("u1"), dev("v1"), dev("u2"), dev("v2"), w, x, dev("y"), dev("z"),
                  alpha=fx["alpha"], beta=fx["beta"], update_A=True)
        w2, x2 = dev("w"), dev("x")
        dm.gemver(dev("A"), dev("u1"), dev("v1"), dev("u2"), dev("v2"), w2, x2, dev("y"),
                  dev("z"), alpha=fx["alpha"], beta=fx["beta"], update_A=False)
        got = {"A_hat": A, "w_out": w, "x_out": x}
        torch.cuda.synchronize()
        assert torch.equal(w2.cpu(), torch.tensor(fx["w_out"], dtype=t))
        assert torch.equal(x2.cpu(), torch.tensor(fx["x_out"], dtype=t))
    torch.cuda.synchronize()
    for key, val in got.items():
        want = torch.tensor(fx[key], dtype=val.dtype)
        assert torch.equal(val.cpu(), want), key
