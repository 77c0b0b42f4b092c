"""Parity of the CUDA path against the CPU oracle, through the C ABI.

Every test here needs a GB300 and the built library.  Sizes span several
tiles (256-column bands, 32- or 16-row stripes) with ragged tails; the five
named workloads run at full size, in the launch configuration the benchmark
times, and every output element is compared."""
import math

import numpy as np
import pytest
import torch

import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import inputs
from parity import TAG, TOL, run_and_compare

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
DT = {"f32": torch.float32, "f64": torch.float64, "i32": torch.int32}


@pytest.fixture(params=[dm.DUALMV_PATH_TMA, dm.DUALMV_PATH_DIRECT], ids=["tma", "direct"])
def path(request):
    old = dm.dualmv_set_path(request.param)
    yield request.param
    dm.dualmv_set_path(old)


def _make(dtype, M, N, lda, seed, batch=0, dist=None):
    dist = dist or {"f32": "uniform", "f64": "normal", "i32": "int8"}[dtype]
    w = inputs.Workload("t", dtype, M, N, lda, dist, seed, batch=batch)
    return inputs.generate(w, DEV)


# ------------------------------------------------------ named workloads ---

@pytest.mark.parametrize("name", list(inputs.WORKLOADS))
def test_workload_full_size(name):
    w = inputs.WORKLOADS[name]
    A, p, r = inputs.generate(w, DEV)
    err = run_and_compare(A, p, r, w.N)
    print(f"{name}: max scaled error {err:.3e}")
    del A, p, r
    torch.cuda.empty_cache()


# ------------------------------------------------------------ shape sweep --

SWEEP_M = [1, 3, 31, 32, 33, 129, 1000]
SWEEP_N = [1, 3, 4, 255, 256, 257, 1000]


@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
def test_shape_sweep(dtype, path):
    seed = 100
    for M in SWEEP_M:
        for N in SWEEP_N:
            seed += 1
            A, p, r = _make(dtype, M, N, N, seed)
            run_and_compare(A, p, r, N)


@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
@pytest.mark.parametrize("extra", [1, 3, 8, 40])
def test_padded_leading_dimension(dtype, extra, path):
    """lda > N, padding filled with NaN / INT32_MIN: never read."""
    for M, N in ((77, 300), (300, 77), (1, 513)):
        A, p, r = _make(dtype, M, N, N + extra, 7 * extra + M)
        run_and_compare(A, p, r, N)


@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
def test_misaligned_base_takes_plain_loads(dtype):
    """A starting one element past a 16-byte boundary is still correct."""
    M, N, lda = 65, 700, 704
    A, p, r = _make(dtype, M, N, lda, 55)
    flat = torch.empty(M * lda + 1, dtype=A.dtype, device=DEV)
    view = flat[1:].view(M, lda)
    view.copy_(A)
    assert view.data_ptr() % 16 != 0
    run_and_compare(view, p, r, N)


@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
def test_empty_dimensions(dtype):
    out_t = inputs.OUT_DTYPES[dtype]
    A = torch.empty(5, 1, dtype=DT[dtype], device=DEV)
    q, s = dm.dualmv(A[:, :0], torch.empty(0, dtype=DT[dtype], device=DEV),
                     torch.ones(5, dtype=DT[dtype], device=DEV))
    assert q.dtype == out_t and (q.cpu() == 0).all() and s.numel() == 0
    A = torch.empty(0, 7, dtype=DT[dtype], device=DEV)
    q, s = dm.dualmv(A, torch.ones(7, dtype=DT[dtype], device=DEV),
                     torch.empty(0, dtype=DT[dtype], device=DEV))
    assert q.numel() == 0 and (s.cpu() == 0).all()
    A = torch.empty(0, 4, 7, dtype=DT[dtype], device=DEV)
    q, s = dm.dualmv(A, torch.empty(0, 7, dtype=DT[dtype], device=DEV),
                     torch.empty(0, 4, dtype=DT[dtype], device=DEV))
    assert q.shape == (0, 4) and s.shape == (0, 7)


# ------------------------------------------------------ closed forms -------

def _identity_case(dtype, n=700):
    A = torch.eye(n, dtype=DT[dtype], device=DEV)
    g = torch.Generator(device=DEV).manual_seed(3)
    if dtype == "i32":
        p = torch.randint(-1000, 1000, (n,), generator=g, device=DEV, dtype=torch.int32)
        r = torch.randint(-1000, 1000, (n,), generator=g, device=DEV, dtype=torch.int32)
    else:
        p = torch.empty(n, dtype=DT[dtype], device=DEV).uniform_(-1, 1, generator=g)
        r = torch.empty(n, dtype=DT[dtype], device=DEV).uniform_(-1, 1, generator=g)
    return A, p, r


@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
def test_identity_is_bit_exact(dtype, path):
    """A = I: q = p and s = r bit for bit (each sum has one nonzero term),
    except fp64 on the FP32-pipe path, whose double-float split rounds the
    29 low mantissa bits to a float's 24: there the result is within 2^-47
    relative (tested against 2^-46)."""
    A, p, r = _identity_case(dtype)
    q, s = dm.dualmv(A, p, r)
    if dtype == "f64" and path == dm.DUALMV_PATH_TMA:
        for got, want in ((q, p), (s, r)):
            rel = ((got - want).abs() / want.abs()).max()
            assert float(rel) <= 2.0 ** -46
    else:
        assert torch.equal(q.cpu(), p.cpu().to(q.dtype)) and torch.equal(s.cpu(), r.cpu().to(s.dtype))


def test_identity_bit_exact_with_native_fp64():
    A, p, r = _identity_case("f64")
    old = dm.dualmv_set_path(dm.DUALMV_PATH_TMA_NATIVE_F64)
    try:
        q, s = dm.dualmv(A, p, r)
    finally:
        dm.dualmv_set_path(old)
    assert torch.equal(q, p) and torch.equal(s, r)


@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
def test_rank_one_is_bit_exact(dtype, path):
    """A = u v^T with small integers: every partial sum is an exact integer,
    so q = u (v.p) and s = v (u.r) hold bit for bit in any order."""
    M, N = 1031, 777
    g = torch.Generator(device="cpu").manual_seed(4)
    u, v = torch.randint(-8, 9, (M,), generator=g), torch.randint(-8, 9, (N,), generator=g)
    p, r = torch.randint(-8, 9, (N,), generator=g), torch.randint(-8, 9, (M,), generator=g)
    qw, sw = u * int(v @ p), v * int(u @ r)
    t = DT[dtype]
    A = torch.outer(u, v).to(t).to(DEV)
    q, s = dm.dualmv(A, p.to(t).to(DEV), r.to(t).to(DEV))
    assert torch.equal(q.cpu().to(torch.int64), qw) and torch.equal(s.cpu().to(torch.int64), sw)


@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
@pytest.mark.parametrize("M,N,pad", [(1000, 3000, 5), (4096, 2048, 0)])
def test_power_of_two_scaling_is_bit_exact(dtype, M, N, pad, path):
    """q(A, 2p, r) = 2 q and s(A, p, 4r) = 4 s bit for bit: binary scaling
    commutes with every rounding (and with the double-float split) while
    nothing overflows, and integer sums are exact.  Pins the GPU path
    without the oracle."""
    A, p, r = _make(dtype, M, N, N + pad, 21)
    A = A[:, :N]
    q, s = dm.dualmv(A, p, r)
    q2, s1 = dm.dualmv(A, p * 2, r)
    q1, s4 = dm.dualmv(A, p, r * 4)
    torch.cuda.synchronize()
    assert torch.equal(q2, q * 2) and torch.equal(s1, s)
    assert torch.equal(s4, s * 4) and torch.equal(q1, q)


@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
def test_transpose_swaps_outputs(dtype):
    """dualmv(A^T, r, p) gives (s, q): the row and column paths agree."""
    M, N = 513, 1200
    A, p, r = _make(dtype, M, N, N, 9)
    q, s = dm.dualmv(A, p, r)
    At = A.t().contiguous()
    s2, q2 = dm.dualmv(At, r, p)
    if dtype == "i32":
        assert torch.equal(q, q2) and torch.equal(s, s2)
    else:
        for a, b in ((q, q2), (s, s2)):
            den = float(torch.abs(A).double().sum())
            assert float((a.double() - b.double()).abs().max()) <= TOL[dtype] * den


def test_adjoint_identity_int_exact():
    M, N = 999, 1777
    A, p, r = _make("i32", M, N, N, 10)
    q, s = dm.dualmv(A, p, r)
    lhs = int((p.cpu().to(torch.int64) * s.cpu()).sum())
    rhs = int((r.cpu().to(torch.int64) * q.cpu()).sum())
    assert lhs == rhs


# ------------------------------------------------------------- batched -----

@pytest.mark.parametrize("dtype", ["f32", "f64", "i32"])
def test_batched_matches_single(dtype, path):
    Bn, M, N = 5, 70, 600
    A, p, r = _make(dtype, M, N, N + 4, 11, batch=Bn)
    run_and_compare(A, p, r, N)
    q, s = dm.dualmv(A[..., :N], p, r)
    for b in range(Bn):
        qb, sb = dm.dualmv(A[b, :, :N], p[b], r[b])
        if dtype == "i32":
            assert torch.equal(qb, q[b]) and torch.equal(sb, s[b])
        else:
            den = float(torch.abs(A[b, :, :N]).double().sum()) + 1.0
            assert float((qb.double() - q[b].double()).abs().max()) <= TOL[dtype] * den
            assert float((sb.double() - s[b].double()).abs().max()) <= TOL[dtype] * den


def test_batched_shared_vectors():
    """p and r given once (stride 0) apply to every problem."""
    Bn, M, N = 4, 50, 300
    A, p, r = _make("f32", M, N, N, 12, batch=Bn)
    run_and_compare(A, p[0], r[0], N)


# --------------------------------------------------- contract and guards ---

def test_outputs_stay_in_bounds():
    """Guard zones after q and s keep their sentinel (no stray writes)."""
    M, N, G = 333, 1025, 1000
    A, p, r = _make("f32", M, N, N, 13)
    qbuf = torch.full((M + G,), 7.0, device=DEV)
    sbuf = torch.full((N + G,), 7.0, device=DEV)
    dm.dualmv(A, p, r, q=qbuf[:M], s=sbuf[:N])
    torch.cuda.synchronize()
    assert (qbuf[M:] == 7.0).all() and (sbuf[N:] == 7.0).all()


def test_deterministic_bitwise():
    w = inputs.WORKLOADS["f32_16384x16384"].scaled(M=4096, N=8192, lda=8192)
    A, p, r = inputs.generate(w, DEV)
    outs = [dm.dualmv(A, p, r) for _ in range(3)]
    for q, s in outs[1:]:
        assert torch.equal(q, outs[0][0]) and torch.equal(s, outs[0][1])


def test_non_default_stream():
    M, N = 800, 900
    A, p, r = _make("f64", M, N, N, 14)
    st = torch.cuda.Stream(device=DEV)
    with torch.cuda.stream(st):
        q, s = dm.dualmv(A, p, r)
    st.synchronize()
    q2, s2 = dm.dualmv(A, p, r)
    torch.cuda.synchronize()
    assert torch.equal(q, q2) and torch.equal(s, s2)


def test_tma_and_direct_paths_agree_within_tolerance():
    M, N = 2000, 3000
    A, p, r = _make("f32", M, N, N, 15)
    old = dm.dualmv_set_path(dm.DUALMV_PATH_TMA)
    q1, s1 = dm.dualmv(A, p, r)
    dm.dualmv_set_path(dm.DUALMV_PATH_DIRECT)
    q2, s2 = dm.dualmv(A, p, r)
    dm.dualmv_set_path(old)
    den = float(torch.abs(A).sum())
    assert float((q1 - q2).abs().max()) <= 1e-5 * den
    assert float((s1 - s2).abs().max()) <= 1e-5 * den


def test_no_device_fault_recorded():
    assert dm.device_fault() == dm.DUALMV_SUCCESS


def test_tensor_api_checks_its_arguments():
    """The tensor entry point rejects what the C ABI cannot take, before
    any launch, and accepts caller-provided outputs."""
    A = torch.randn(64, 96, device="cuda:0")
    p = torch.randn(96, device="cuda:0")
    r = torch.randn(64, device="cuda:0")
    with pytest.raises(ValueError):
        dm.dualmv(A.cpu(), p.cpu(), r.cpu())                   # no CPU path
    with pytest.raises(ValueError):
        dm.dualmv(A, p.double(), r)                            # dtype mismatch
    with pytest.raises(ValueError):
        dm.dualmv(A, p, r, q=torch.empty(63, device="cuda:0"))  # q shape
    with pytest.raises(ValueError):
        dm.dualmv(A, p, r, q=torch.empty(64, device="cuda:0", dtype=torch.float64))
    with pytest.raises(ValueError):
        dm.dualmv(A.t(), r, p)                                 # not row-major
    with pytest.raises(TypeError):
        dm.dualmv(A.long(), p.long(), r.long())                # no int64 entry point
    q = torch.empty(64, device="cuda:0")
    s = torch.empty(96, device="cuda:0")
    q2, s2 = dm.dualmv(A, p, r, q=q, s=s)
    torch.cuda.synchronize()
    assert q2 is q and s2 is s
    An = A.double().cpu()
    assert torch.allclose(q.double().cpu(), An @ p.double().cpu(), rtol=1e-4, atol=1e-4)
    assert torch.allclose(s.double().cpu(), An.t() @ r.double().cpu(), rtol=1e-4, atol=1e-4)


@pytest.mark.parametrize("dtype", ["f32", "i32", "f64"])
@pytest.mark.parametrize("lda_mod4", [1, 2, 3, 0])
@pytest.mark.parametrize("base", [0, 1, 2, 3])
def test_unaligned_rows_take_phased_maps(dtype, lda_mod4, base):
    """Rows whose stride or base is not 16-byte aligned go through one pair
    of tensor maps per row phase (4-byte elements: lda odd gives 4 phases,
    lda = 2 mod 4 gives 2, a base alone 1; 8-byte elements: lda odd gives 2,
    a base alone 1).  Ragged M and N, N below one band, and fewer rows than
    phases (which fall back to plain loads) all match the oracle."""
    per16 = 2 if dtype == "f64" else 4          # elements per 16 bytes
    for M, N in ((67, 517), (130, 250), (5, 1030), (33, 256), (3, 300), (1, 70)):
        lda = N + (lda_mod4 - N) % 4
        A, p, r = _make(dtype, M, N, lda, 91 + 7 * lda_mod4 + base)
        store = torch.empty(M * lda + base + 8, dtype=A.dtype, device=DEV)
        view = store[base:base + M * lda].view(M, lda)
        view.copy_(A)
        run_and_compare(view, p, r, N)
        eff = lda if M > 1 else N                 # one row: the API passes lda = N
        nph = per16 // math.gcd(eff, per16)
        kind = dm.dualmv_last_kernel()
        if eff % per16 == 0 and base % per16 == 0:
            assert kind in (dm.DUALMV_KERNEL_STREAM, dm.DUALMV_KERNEL_WIDE,
                            dm.DUALMV_KERNEL_F64E, dm.DUALMV_KERNEL_CLUSTER), (M, N, lda, base,
                                                                               kind)
        elif M >= nph:
            assert kind == dm.DUALMV_KERNEL_PHASED, (M, N, lda, base, kind)
        else:
            assert kind == dm.DUALMV_KERNEL_PLAIN


def test_unaligned_f64_rows_keep_the_double_float_range_check():
    """fp64 rows at an odd stride take the phased double-float kernel, whose
    per-tile range check still sends tiles with huge, tiny or non-finite
    entries to native fp64: the results match the oracle and every
    non-finite value lands where it should."""
    M, N = 150, 777
    lda = N + 2                                   # odd: two row phases
    A, p, r = _make("f64", M, N, lda, 95)
    A[3, 5] = 1e60
    A[70, 600] = 3e-200
    A[100, 260] = 0.0
    store = torch.empty(M * lda + 8, dtype=A.dtype, device=DEV)
    view = store[1:1 + M * lda].view(M, lda)
    view.copy_(A)
    run_and_compare(view, p, r, N)
    assert dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_PHASED
    view[40, 300] = float("inf")
    q, s = dm.dualmv(view[:, :N], p, r)
    torch.cuda.synchronize()
    qc, sc = q.cpu(), s.cpu()
    assert math.isinf(qc[40].item()) or math.isnan(qc[40].item())
    assert torch.isfinite(torch.cat([qc[:40], qc[41:]])).all()
    assert not math.isfinite(sc[300].item())
    assert torch.isfinite(torch.cat([sc[:300], sc[301:]])).all()


@pytest.mark.parametrize("dtype,M,N,lda", [
    ("f32", 3000, 5000, 5001),      # 4 phases; many CTAs per band
    ("f32", 2500, 4098, 4098),      # 2 phases
    ("i32", 777, 20001, 20003),     # 4 phases, exact
    ("f64", 2000, 3000, 3001),      # 2 phases, double-float
])
def test_phased_many_tiles_match_oracle_and_repeat_bitwise(dtype, M, N, lda):
    """The phased kernels over many stripes and bands, where several CTAs
    share a band and their column partials meet in the combine: every
    output matches the oracle, and repeated calls give the same bits."""
    A, p, r = _make(dtype, M, N, lda, 97)
    run_and_compare(A, p, r, N)
    assert dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_PHASED
    view = A[:, :N]
    outs = [dm.dualmv(view, p, r) for _ in range(3)]
    torch.cuda.synchronize()
    for q, s in outs[1:]:
        assert torch.equal(q, outs[0][0]) and torch.equal(s, outs[0][1])


def test_last_kernel_reports_each_path():
    A, p, r = _make("f64", 96, 512, 512, 92)
    dm.dualmv(A, p, r)
    assert dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_F64E
    old = dm.dualmv_set_path(dm.DUALMV_PATH_DIRECT)
    try:
        dm.dualmv(A, p, r)
        assert dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_PLAIN
    finally:
        dm.dualmv_set_path(old)
    A, p, r = _make("f32", 96, 512, 512, 93)
    dm.dualmv(A, p, r)
    assert dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_CLUSTER
    old = dm.dualmv_set_path(dm.DUALMV_PATH_TMA)
    try:
        dm.dualmv(A, p, r)
        assert dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_STREAM
    finally:
        dm.dualmv_set_path(old)
    dm.dualmv(A[:0], p, r[:0])
    assert dm.dualmv_last_kernel() == -1
