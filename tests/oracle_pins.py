"""Pins for the CPU oracle: checks that depend only on mathematics.

Each ``pin_*`` function takes a loaded oracle library and raises
``AssertionError`` when the oracle disagrees with a value fixed
independently of it: exact rational arithmetic, a closed form, an identity,
or a published error bound.  ``tests/test_oracle_pins.py`` runs them on the
real oracle; ``tests/test_oracle_mutants.py`` runs them on copies of the
oracle with a planted mistake and expects at least one to fail.

The operations are the BICG kernel of the paper (Table 1 and Table 2):
q = A p and s = A^T r, and the GESUMMV, ATAX and GEMVER kernels of the same
tables.
The paper prints no worked example for any of them, so no printed values
can serve as golden data; everything here is derived from the definitions.
"""
from __future__ import annotations

from fractions import Fraction

import numpy as np

import oracle

U53 = Fraction(1, 2 ** 53)          # unit roundoff of binary64
MOD = 2 ** 64


def gamma(n: int) -> Fraction:
    """gamma_n = n u / (1 - n u), the classical bound of n rounded operations."""
    return n * U53 / (1 - n * U53)


def _padded(rng, M, N, extra, dtype, values):
    """M x (N + extra) storage: the matrix in the first N columns and a
    sentinel (NaN or INT32_MIN) in the padding."""
    lda = max(1, N + extra)
    A = np.empty((M, lda), dtype=dtype)
    A[:, N:] = np.nan if dtype != np.int32 else np.iinfo(np.int32).min
    A[:, :N] = values(rng, (M, N))
    return A


def _rand_float(rng, shape, dtype):
    """Values with mixed signs and exponents in [2^-20, 2^20)."""
    mant = rng.uniform(-1.0, 1.0, size=shape)
    expo = rng.integers(-20, 21, size=shape)
    return np.ldexp(mant, expo).astype(dtype)


def _exact(A, p, r, N):
    M = A.shape[0]
    F = [[Fraction(float(A[i, j])) for j in range(N)] for i in range(M)]
    P = [Fraction(float(x)) for x in p]
    R = [Fraction(float(x)) for x in r]
    q = [sum((F[i][j] * P[j] for j in range(N)), Fraction(0)) for i in range(M)]
    s = [sum((F[i][j] * R[i] for i in range(M)), Fraction(0)) for j in range(N)]
    qa = [sum((abs(F[i][j] * P[j]) for j in range(N)), Fraction(0)) for i in range(M)]
    sa = [sum((abs(F[i][j] * R[i]) for i in range(M)), Fraction(0)) for j in range(N)]
    return q, s, qa, sa


# ------------------------------------------------------------ brute force --

def pin_bruteforce_f32(lib, seed=11, cases=40):
    """f32 oracle vs exact rational sums.  Float products are exact in double,
    so only the n-1 additions round: |err| <= gamma_n * sum |a x|."""
    rng = np.random.default_rng(seed)
    for _ in range(cases):
        M, N, extra = (int(x) for x in rng.integers(0, 7, size=3))
        A = _padded(rng, M, N, extra, np.float32,
                    lambda g, sh: _rand_float(g, sh, np.float32))
        p = _rand_float(rng, N, np.float32)
        r = _rand_float(rng, M, np.float32)
        q, s = oracle.dualmv(A, p, r, N=N, lib=lib)
        eq, es, qa, sa = _exact(A, p, r, N)
        for got, want, mag, n in ((q, eq, qa, N), (s, es, sa, M)):
            for g_, w_, m_ in zip(got, want, mag):
                assert np.isfinite(g_), "padding or garbage was read"
                assert abs(Fraction(float(g_)) - w_) <= gamma(max(n, 1)) * m_, \
                    (M, N, g_, float(w_))


def pin_bruteforce_f64(lib, seed=12, cases=40):
    """f64 oracle (Dot2) vs exact rational sums, within the published bound
    |res - x.y| <= u |x.y| + gamma_n^2 sum |x||y| (Ogita, Rump, Oishi 2005)."""
    rng = np.random.default_rng(seed)
    for _ in range(cases):
        M, N, extra = (int(x) for x in rng.integers(0, 7, size=3))
        A = _padded(rng, M, N, extra, np.float64,
                    lambda g, sh: _rand_float(g, sh, np.float64))
        p = _rand_float(rng, N, np.float64)
        r = _rand_float(rng, M, np.float64)
        q, s = oracle.dualmv(A, p, r, N=N, lib=lib)
        eq, es, qa, sa = _exact(A, p, r, N)
        for got, want, mag, n in ((q, eq, qa, N), (s, es, sa, M)):
            for g_, w_, m_ in zip(got, want, mag):
                assert np.isfinite(g_)
                bound = U53 * abs(w_) + gamma(max(n, 1)) ** 2 * m_
                assert abs(Fraction(float(g_)) - w_) <= bound, (M, N)


def pin_bruteforce_i32(lib, seed=13, cases=40):
    """i32 oracle vs Python integers reduced modulo 2^64, over the full int32
    range so that products need 63 bits and sums wrap."""
    rng = np.random.default_rng(seed)
    lo, hi = np.iinfo(np.int32).min, np.iinfo(np.int32).max
    for _ in range(cases):
        M, N, extra = (int(x) for x in rng.integers(0, 7, size=3))
        A = _padded(rng, M, N, extra, np.int32,
                    lambda g, sh: g.integers(lo, hi, size=sh, endpoint=True))
        p = rng.integers(lo, hi, size=N, endpoint=True).astype(np.int32)
        r = rng.integers(lo, hi, size=M, endpoint=True).astype(np.int32)
        q, s = oracle.dualmv(A, p, r, N=N, lib=lib)
        for i in range(M):
            want = sum(int(A[i, j]) * int(p[j]) for j in range(N)) % MOD
            assert int(q[i]) % MOD == want, (M, N, i)
        for j in range(N):
            want = sum(int(A[i, j]) * int(r[i]) for i in range(M)) % MOD
            assert int(s[j]) % MOD == want, (M, N, j)


def pin_wraparound_i32(lib):
    """Sums past 2^63 wrap: 4 products of (-2^31)^2 = 2^62 sum to 2^64 = 0."""
    m = np.iinfo(np.int32).min
    A = np.full((4, 4), m, dtype=np.int32)
    p = np.full(4, m, dtype=np.int32)
    q, s = oracle.dualmv(A, p, p, lib=lib)
    assert (q == 0).all() and (s == 0).all()
    A = np.full((1, 2), m, dtype=np.int32)
    q, _ = oracle.dualmv(A, np.full(2, m, np.int32), np.ones(1, np.int32), lib=lib)
    assert int(q[0]) == -(2 ** 63)      # 2^62 + 2^62 = 2^63 wraps to -2^63


# ------------------------------------------------------ compensated sums --

def pin_dot2_cancellation(lib):
    """Ill-conditioned sums that plain double arithmetic gets wrong and Dot2
    gets exactly right, in both the row (q) and column (s) directions.

    TwoSum: 2^60 + 1 - 2^60 = 1 (plain double gives 0).
    TwoProduct: (1+2^-30)^2 - (1+2^-29) = 2^-60 (plain double gives 0)."""
    big = 2.0 ** 60
    A = np.array([[big, 1.0, -big]], dtype=np.float64)
    one3 = np.ones(3, dtype=np.float64)
    q, _ = oracle.dualmv(A, one3, np.ones(1), lib=lib)
    assert q[0] == 1.0, q
    _, s = oracle.dualmv(A.T.copy(), np.ones(1), one3, lib=lib)
    assert s[0] == 1.0, s
    a = 1.0 + 2.0 ** -30
    A = np.array([[a, 1.0 + 2.0 ** -29]], dtype=np.float64)
    q, _ = oracle.dualmv(A, np.array([a, -1.0]), np.ones(1), lib=lib)
    assert q[0] == 2.0 ** -60, q
    _, s = oracle.dualmv(A.T.copy(), np.ones(1), np.array([a, -1.0]), lib=lib)
    assert s[0] == 2.0 ** -60, s


# ----------------------------------------------------------- closed forms --

def pin_identity(lib, n=37):
    """A = I: q = p and s = r exactly, for every dtype."""
    rng = np.random.default_rng(5)
    for dt in (np.float32, np.float64):
        A = np.eye(n, dtype=dt)
        p = rng.uniform(-1, 1, n).astype(dt)
        r = rng.uniform(-1, 1, n).astype(dt)
        q, s = oracle.dualmv(A, p, r, lib=lib)
        assert (q == p.astype(np.float64)).all() and (s == r.astype(np.float64)).all()
    A = np.eye(n, dtype=np.int32)
    p = rng.integers(-1000, 1000, n).astype(np.int32)
    r = rng.integers(-1000, 1000, n).astype(np.int32)
    q, s = oracle.dualmv(A, p, r, lib=lib)
    assert (q == p).all() and (s == r).all()


def pin_rank_one(lib, M=23, N=41):
    """A = u v^T with small integers: q = u (v.p) and s = v (u.r), all values
    exact integers in every dtype."""
    rng = np.random.default_rng(6)
    u = rng.integers(-8, 9, M)
    v = rng.integers(-8, 9, N)
    p = rng.integers(-8, 9, N)
    r = rng.integers(-8, 9, M)
    qw = u * int(v @ p)
    sw = v * int(u @ r)
    for dt in (np.float32, np.float64, np.int32):
        A = np.outer(u, v).astype(dt)
        q, s = oracle.dualmv(A, p.astype(dt), r.astype(dt), lib=lib)
        assert (q == qw).all() and (s == sw).all(), dt


def pin_adjoint(lib, M=19, N=29):
    """p.s = r.q (both equal r^T A p): exact modulo 2^64 for integers, within
    rounding for floats."""
    rng = np.random.default_rng(7)
    lo, hi = np.iinfo(np.int32).min, np.iinfo(np.int32).max
    A = rng.integers(lo, hi, (M, N), endpoint=True).astype(np.int32)
    p = rng.integers(lo, hi, N, endpoint=True).astype(np.int32)
    r = rng.integers(lo, hi, M, endpoint=True).astype(np.int32)
    q, s = oracle.dualmv(A, p, r, lib=lib)
    lhs = sum(int(p[j]) * int(s[j]) for j in range(N)) % MOD
    rhs = sum(int(r[i]) * int(q[i]) for i in range(M)) % MOD
    assert lhs == rhs
    A = rng.uniform(-1, 1, (M, N))
    p = rng.uniform(-1, 1, N)
    r = rng.uniform(-1, 1, M)
    q, s = oracle.dualmv(A, p, r, lib=lib)
    scale = float(np.abs(r) @ np.abs(A) @ np.abs(p))
    assert abs(float(p @ s) - float(r @ q)) <= 1e-13 * scale


def pin_power_of_two_scaling(lib, M=17, N=33):
    """Scaling p by 2 scales q by 2 exactly; scaling r by 4 scales s by 4."""
    rng = np.random.default_rng(8)
    for dt in (np.float32, np.float64):
        A = rng.uniform(-1, 1, (M, N)).astype(dt)
        p = rng.uniform(-1, 1, N).astype(dt)
        r = rng.uniform(-1, 1, M).astype(dt)
        q, s = oracle.dualmv(A, p, r, lib=lib)
        q2, _ = oracle.dualmv(A, (2 * p).astype(dt), r, lib=lib)
        _, s4 = oracle.dualmv(A, p, (4 * r).astype(dt), lib=lib)
        assert (q2 == 2 * q).all() and (s4 == 4 * s).all()


def pin_shapes_and_empty(lib):
    """Outputs have the right lengths; empty dimensions give zeros."""
    q, s = oracle.dualmv(np.zeros((0, 5), np.float32), np.ones(5, np.float32),
                         np.ones(0, np.float32), lib=lib)
    assert q.shape == (0,) and s.shape == (5,) and (s == 0).all()
    A = np.full((4, 3), np.nan, np.float64)
    q, s = oracle.dualmv(A, np.ones(0), np.ones(4), N=0, lib=lib)
    assert q.shape == (4,) and s.shape == (0,) and (q == 0).all()


def pin_absdot(lib):
    """Denominators equal the exact magnitude sums on small integers and
    bound |q| and |s|."""
    rng = np.random.default_rng(9)
    M, N = 6, 9
    A = rng.integers(-8, 9, (M, N)).astype(np.float64)
    p = rng.integers(-8, 9, N).astype(np.float64)
    r = rng.integers(-8, 9, M).astype(np.float64)
    qa, sa = oracle.absdot(A, p, r, lib=lib)
    assert (qa == np.abs(A) @ np.abs(p)).all()
    assert (sa == np.abs(r) @ np.abs(A)).all()
    q, s = oracle.dualmv(A, p, r, lib=lib)
    assert (np.abs(q) <= qa).all() and (np.abs(s) <= sa).all()
    qa32, sa32 = oracle.absdot(A.astype(np.float32), p.astype(np.float32),
                               r.astype(np.float32), lib=lib)
    assert (qa32 == qa).all() and (sa32 == sa).all()


# --------------------------------------------------------- trimmed mean --

def pin_trimmed_mean(lib):
    """Eq. 3 with R = 30, k = 3 (the paper's setting, Section 4.1.4): the
    mean of the 24 middle values of a shuffled 1..30 is 15.5; outliers at
    both ends are dropped; R <= 2k is rejected."""
    rng = np.random.default_rng(10)
    t = rng.permutation(np.arange(1, 31)).astype(float)
    assert oracle.trimmed_mean(t, 3, lib=lib) == 15.5
    t = [5.0] * 24 + [1e9, 1e9, 1e9, -1e9, -1e9, -1e9]
    assert oracle.trimmed_mean(t, 3, lib=lib) == 5.0
    assert oracle.trimmed_mean([1.0, 2.0, 4.0], 0, lib=lib) == 7.0 / 3.0
    for bad in (([1.0, 2.0], 1), ([1.0] * 6, 3)):
        try:
            oracle.trimmed_mean(*bad, lib=lib)
        except ValueError:
            continue
        raise AssertionError("R <= 2k accepted")


# ------------------------------------------------------- GESUMMV, ATAX --

def _exact_dot_rows(A, x, N):
    M = A.shape[0]
    F = [[Fraction(float(A[i, j])) for j in range(N)] for i in range(M)]
    X = [Fraction(float(v)) for v in x]
    dots = [sum((F[i][j] * X[j] for j in range(N)), Fraction(0)) for i in range(M)]
    mags = [sum((abs(F[i][j] * X[j]) for j in range(N)), Fraction(0)) for i in range(M)]
    return F, dots, mags


def pin_gesummv_bruteforce(lib, seed=14, cases=30):
    """y = alpha A x + beta B x against exact rationals, within
    (gamma_(N+2) + 3u) (|alpha| sum|A||x| + |beta| sum|B||x|) (a
    double-accumulated or Dot2 sum, then two products and one addition)."""
    rng = np.random.default_rng(seed)
    for case in range(cases):
        dt = np.float32 if case % 2 == 0 else np.float64
        M, N = (int(v) for v in rng.integers(0, 7, size=2))
        ea, eb = (int(v) for v in rng.integers(0, 4, size=2))
        A = _padded(rng, M, N, ea, dt, lambda g, sh: _rand_float(g, sh, dt))
        B = _padded(rng, M, N, eb, dt, lambda g, sh: _rand_float(g, sh, dt))
        x = _rand_float(rng, N, dt)
        alpha, beta = 0.75, -1.5
        y = oracle.gesummv(A, B, x, alpha, beta, N=N, lib=lib)
        _, da, ma = _exact_dot_rows(A, x, N)
        _, db, mb = _exact_dot_rows(B, x, N)
        for i in range(M):
            assert np.isfinite(y[i]), "padding read"
            want = Fraction(alpha) * da[i] + Fraction(beta) * db[i]
            mag = abs(Fraction(alpha)) * ma[i] + abs(Fraction(beta)) * mb[i]
            assert abs(Fraction(float(y[i])) - want) <= (gamma(N + 2) + 3 * U53) * mag, (M, N, i)


def pin_gesummv_closed_forms(lib):
    """B = 0 gives alpha (A x) exactly (alpha a power of two); A = B with
    alpha = beta = 1 gives exactly twice A x; an ill-conditioned row that
    only compensated sums get right."""
    rng = np.random.default_rng(15)
    for dt in (np.float32, np.float64):
        A = rng.uniform(-1, 1, (9, 13)).astype(dt)
        x = rng.uniform(-1, 1, 13).astype(dt)
        ax, _ = oracle.dualmv(A, x, np.zeros(9, dt), lib=lib)
        y = oracle.gesummv(A, np.zeros_like(A), x, 4.0, 3.0, lib=lib)
        assert (y == 4.0 * ax).all()
        y = oracle.gesummv(A, A.copy(), x, 1.0, 1.0, lib=lib)
        assert (y == 2.0 * ax).all()
    big = 2.0 ** 60
    A = np.array([[big, 1.0, -big]])
    y = oracle.gesummv(A, -A, np.ones(3), 1.0, 0.5, lib=lib)
    assert y[0] == 0.5, y


def pin_atax_bruteforce(lib, seed=16, cases=30):
    """y = A^T (A x) against exact rationals.  Bound per output j, with
    D_j = sum_i |A_ij| sum_k |A_ik||x_k|: (gamma_N + gamma_M) D_j for the
    double-accumulated float oracle, (4u + 2 gamma^2) D_j for Dot2 with tmp
    rounded to double."""
    rng = np.random.default_rng(seed)
    for case in range(cases):
        dt = np.float32 if case % 2 == 0 else np.float64
        M, N, extra = (int(v) for v in rng.integers(0, 7, size=3))
        A = _padded(rng, M, N, extra, dt, lambda g, sh: _rand_float(g, sh, dt))
        x = _rand_float(rng, N, dt)
        y = oracle.atax(A, x, N=N, lib=lib)
        F, tmp, mags = _exact_dot_rows(A, x, N)
        for j in range(N):
            assert np.isfinite(y[j]), "padding read"
            want = sum((F[i][j] * tmp[i] for i in range(M)), Fraction(0))
            D = sum((abs(F[i][j]) * mags[i] for i in range(M)), Fraction(0))
            g = max(M, N, 1)
            bound = (2 * gamma(g)) * D if dt == np.float32 else (4 * U53 + 2 * gamma(g) ** 2) * D
            assert abs(Fraction(float(y[j])) - want) <= bound, (M, N, j)


def pin_atax_closed_forms(lib):
    """A a permutation: y = x exactly; A = u v^T with small integers:
    y = v (u.u)(v.x) exactly."""
    rng = np.random.default_rng(17)
    perm = rng.permutation(11)
    for dt in (np.float32, np.float64):
        P = np.zeros((11, 11), dt)
        P[np.arange(11), perm] = 1.0
        x = rng.uniform(-1, 1, 11).astype(dt)
        assert (oracle.atax(P, x, lib=lib) == x.astype(np.float64)).all()
        u = rng.integers(-8, 9, 7)
        v = rng.integers(-8, 9, 5)
        xi = rng.integers(-8, 9, 5)
        A = np.outer(u, v).astype(dt)
        want = v * int(u @ u) * int(v @ xi)
        assert (oracle.atax(A, xi.astype(dt), lib=lib) == want).all()
    # A row whose product with x cancels: tmp = 2^60 + 1 - 2^60 = 1 needs the
    # compensated sum; then y = A^T tmp is that row itself.
    big = 2.0 ** 60
    A = np.array([[big, 1.0, -big]])
    assert (oracle.atax(A, np.ones(3), lib=lib) == A[0]).all()


# -------------------------------------------------------------- GEMVER --

def pin_gemver_bruteforce(lib, seed=18, cases=24):
    """GEMVER against exact rationals: A_hat, the new x and the new w, each
    within a small multiple of the unit roundoff times the magnitude of its
    terms (the new x's error carried into w)."""
    rng = np.random.default_rng(seed)
    for case in range(cases):
        dt = np.float32 if case % 2 == 0 else np.float64
        M, N, extra = (int(v) for v in rng.integers(1, 6, size=3))
        A = _padded(rng, M, N, extra, dt, lambda g, sh: _rand_float(g, sh, dt))
        u1, u2, w, y = (_rand_float(rng, M, dt) for _ in range(4))
        v1, v2, x, z = (_rand_float(rng, N, dt) for _ in range(4))
        alpha, beta = 1.5, -0.75
        ah, wo, xo = oracle.gemver(A, u1, v1, u2, v2, w, x, y, z, alpha, beta, N=N, lib=lib)
        F = lambda v: Fraction(float(v))  # noqa: E731
        Ah = [[F(A[i, j]) + F(u1[i]) * F(v1[j]) + F(u2[i]) * F(v2[j]) for j in range(N)]
              for i in range(M)]
        Am = [[abs(F(A[i, j])) + abs(F(u1[i]) * F(v1[j])) + abs(F(u2[i]) * F(v2[j]))
               for j in range(N)] for i in range(M)]
        Xe = [F(x[j]) + Fraction(beta) * sum((Ah[i][j] * F(y[i]) for i in range(M)), Fraction(0))
              + F(z[j]) for j in range(N)]
        Xm = [abs(F(x[j])) + abs(Fraction(beta)) * sum((Am[i][j] * abs(F(y[i])) for i in range(M)),
                                                       Fraction(0)) + abs(F(z[j])) for j in range(N)]
        We = [F(w[i]) + Fraction(alpha) * sum((Ah[i][j] * Xe[j] for j in range(N)), Fraction(0))
              for i in range(M)]
        Wm = [abs(F(w[i])) + abs(Fraction(alpha)) * sum((Am[i][j] * Xm[j] for j in range(N)),
                                                        Fraction(0)) for i in range(M)]
        c = gamma(max(M, N) + 6) if dt == np.float32 else 16 * U53 + gamma(max(M, N)) ** 2
        # A_hat: three exact products summed in double (f32 inputs), or a
        # compensated sum rounded once (f64 inputs).
        for i in range(M):
            for j in range(N):
                b = (2 * U53 * Am[i][j] if dt == np.float32
                     else U53 * abs(Ah[i][j]) + 4 * U53 * U53 * Am[i][j])
                assert abs(Fraction(float(ah[i, j])) - Ah[i][j]) <= b
        for j in range(N):
            assert abs(Fraction(float(xo[j])) - Xe[j]) <= c * Xm[j], (M, N, j)
        for i in range(M):
            assert abs(Fraction(float(wo[i])) - We[i]) <= 2 * c * Wm[i], (M, N, i)


def pin_gemver_integers_exact(lib):
    """Small integers keep every GEMVER quantity an exact integer; compare
    with integer arithmetic, and check that u1 = u2 = 0 leaves A_hat = A."""
    rng = np.random.default_rng(19)
    M, N = 9, 13
    A = rng.integers(-8, 9, (M, N))
    u1, u2, w, y = (rng.integers(-4, 5, M) for _ in range(4))
    v1, v2, x, z = (rng.integers(-4, 5, N) for _ in range(4))
    Ah = A + np.outer(u1, v1) + np.outer(u2, v2)
    X = x + 2 * (Ah.T @ y) + z
    W = w + 3 * (Ah @ X)
    for dt in (np.float32, np.float64):
        ah, wo, xo = oracle.gemver(A.astype(dt), *(v.astype(dt) for v in (u1, v1, u2, v2, w, x, y, z)),
                                   3.0, 2.0, lib=lib)
        assert (ah == Ah).all() and (xo == X).all() and (wo == W).all()
        zero = np.zeros(M, dt)
        ah, _, _ = oracle.gemver(A.astype(dt), zero, v1.astype(dt), zero, v2.astype(dt),
                                 w.astype(dt), x.astype(dt), y.astype(dt), z.astype(dt),
                                 3.0, 2.0, lib=lib)
        assert (ah == A).all()
    # A cancelling update that only the compensated f64 sum gets right:
    # 2^60 + 1*1 + (-2^60)*1 = 1.
    one = np.ones(1)
    ah, _, _ = oracle.gemver(np.array([[2.0 ** 60]]), one, one, -(2.0 ** 60) * one, one,
                             one, one, one, one, 1.0, 1.0, lib=lib)
    assert ah[0, 0] == 1.0, ah


ALL_PINS = [
    pin_bruteforce_f32, pin_bruteforce_f64, pin_bruteforce_i32,
    pin_wraparound_i32, pin_dot2_cancellation, pin_identity, pin_rank_one,
    pin_adjoint, pin_power_of_two_scaling, pin_shapes_and_empty, pin_absdot,
    pin_trimmed_mean, pin_gesummv_bruteforce, pin_gesummv_closed_forms,
    pin_atax_bruteforce, pin_atax_closed_forms, pin_gemver_bruteforce,
    pin_gemver_integers_exact,
]


def failing_pins(lib):
    """Names of the pins that fail (or crash) on ``lib``."""
    bad = []
    for pin in ALL_PINS:
        try:
            pin(lib)
        except Exception:           # noqa: BLE001 - any failure counts
            bad.append(pin.__name__)
    return bad
