"""CPU oracle for the fused dual matrix-vector product (PolyBench BICG).

TEST INFRASTRUCTURE ONLY.  Only the test suite, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py`` may import this package.  The
product path (the CUDA library and its binding) never touches it, and this
package imports nothing from the product.

The arithmetic lives in ``oracle.c`` (plain C, built here with gcc).  This
module only builds that file, loads it with ctypes and marshals numpy arrays.

Definition (the BICG kernel of the paper's Table 1 and Table 2, which the
paper names without a formula; this is PolyBench's BiCG sub-kernel):

    q_i = sum_j A[i, j] * p_j        s_j = sum_i A[i, j] * r_i

with A an M x N row-major matrix of leading dimension lda >= N whose
padding columns are never read.

Returned precision: float32 inputs give float64 results (double accumulation
of exact products), float64 inputs give float64 results computed with the
compensated dot product Dot2 (Ogita, Rump and Oishi, 2005), int32 inputs give
int64 results with wrap-around modulo 2^64.

Parity is pinned against the mathematics, not against this code, in
``tests/test_oracle_pins.py``: exact rational brute force, closed forms
(identity, rank one), the adjoint identity, power-of-two scaling, padding
sentinels and an ill-conditioned dot product that only a compensated sum
gets right.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_CFLAGS = ["-std=c99", "-O2", "-fno-fast-math", "-ffp-contract=off", "-fPIC",
           "-shared"]
_lock = threading.Lock()
_lib = None
# The all-core baseline (oracle_omp.c): the same loops on every host core.
_OMP_SRC = os.path.join(_HERE, "oracle_omp.c")
_OMP_LIB_PATH = os.path.join(_HERE, "liboracle_omp.so")
_omp_lib = None


def build(src: str = _SRC, out: str = _LIB_PATH) -> str:
    """Compile ``src`` into the shared library ``out`` with gcc."""
    cmd = ["gcc", *_CFLAGS, "-o", out, src, "-lm"]
    subprocess.run(cmd, check=True)
    return out


def build_omp(src: str = _OMP_SRC, out: str = _OMP_LIB_PATH) -> str:
    """Compile the OpenMP all-core baseline ``oracle_omp.c`` with gcc."""
    cmd = ["gcc", *_CFLAGS, "-fopenmp", "-o", out, src, "-lm"]
    subprocess.run(cmd, check=True)
    return out


def load_omp():
    """Load (building first if needed) the all-core baseline library."""
    global _omp_lib
    with _lock:
        if _omp_lib is None:
            if (not os.path.exists(_OMP_LIB_PATH)
                    or os.path.getmtime(_OMP_LIB_PATH) < os.path.getmtime(_OMP_SRC)):
                build_omp()
            lib = ctypes.CDLL(_OMP_LIB_PATH)
            i64, vp = ctypes.c_int64, ctypes.c_void_p
            for t in ("f32", "f64", "i32"):
                fn = getattr(lib, f"oracle_omp_dualmv_{t}")
                fn.argtypes = [i64, i64, vp, i64, vp, vp, vp, vp]
                fn.restype = ctypes.c_int
            lib.oracle_omp_threads.argtypes, lib.oracle_omp_threads.restype = [], ctypes.c_int
            _omp_lib = lib
    return _omp_lib


def omp_threads() -> int:
    """Threads the all-core baseline runs on (OpenMP's default team size)."""
    return int(load_omp().oracle_omp_threads())


def dualmv_omp(A: np.ndarray, p: np.ndarray, r: np.ndarray, N: int | None = None):
    """``dualmv`` on every host core (OpenMP): the same outputs as
    :func:`dualmv`, bit for bit (each output summed in the same order)."""
    lib = load_omp()
    M, N, lda, p, r = _prep(A, p, r, N)
    tag, out_t = _IN[A.dtype]
    q = np.zeros(M, dtype=out_t)
    s = np.zeros(N, dtype=out_t)
    rc = getattr(lib, f"oracle_omp_dualmv_{tag}")(M, N, _ptr(A), lda, _ptr(p), _ptr(r),
                                                 _ptr(q), _ptr(s))
    if rc != 0:
        raise RuntimeError(f"oracle_omp_dualmv_{tag} returned {rc}")
    return q, s


def _stale() -> bool:
    if not os.path.exists(_LIB_PATH):
        return True
    return os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)


def load(path: str | None = None):
    """Load (building first if needed) the oracle library.

    ``path`` loads another build of ``oracle.c`` instead, which the mutation
    tests use to check that the pins catch a planted mistake.
    """
    global _lib
    if path is not None:
        return _declare(ctypes.CDLL(path))
    with _lock:
        if _lib is None:
            if _stale():
                build()
            _lib = _declare(ctypes.CDLL(_LIB_PATH))
    return _lib


def _declare(lib):
    i64 = ctypes.c_int64
    vp = ctypes.c_void_p
    for name in ("oracle_dualmv_f32", "oracle_dualmv_f64", "oracle_dualmv_i32",
                 "oracle_absdot_f32", "oracle_absdot_f64"):
        fn = getattr(lib, name)
        fn.argtypes = [i64, i64, vp, i64, vp, vp, vp, vp]
        fn.restype = ctypes.c_int
    lib.oracle_trimmed_mean.argtypes = [vp, i64, i64, vp]
    lib.oracle_trimmed_mean.restype = ctypes.c_int
    dbl = ctypes.c_double
    for name in ("oracle_gesummv_f32", "oracle_gesummv_f64"):
        fn = getattr(lib, name)
        fn.argtypes = [i64, i64, dbl, vp, i64, dbl, vp, i64, vp, vp]
        fn.restype = ctypes.c_int
    for name in ("oracle_atax_f32", "oracle_atax_f64"):
        fn = getattr(lib, name)
        fn.argtypes = [i64, i64, vp, i64, vp, vp]
        fn.restype = ctypes.c_int
    for name in ("oracle_gemver_f32", "oracle_gemver_f64"):
        fn = getattr(lib, name)
        fn.argtypes = [i64, i64, dbl, dbl, vp, i64] + [vp] * 11
        fn.restype = ctypes.c_int
    return lib


_IN = {np.dtype(np.float32): ("f32", np.float64),
       np.dtype(np.float64): ("f64", np.float64),
       np.dtype(np.int32): ("i32", np.int64)}


def _ptr(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data) if a.size else None


def _prep(A: np.ndarray, p: np.ndarray, r: np.ndarray, N: int | None):
    if A.ndim != 2:
        raise ValueError("A must be 2-D (M x lda storage)")
    M, lda = A.shape
    N = lda if N is None else int(N)
    if not A.flags.c_contiguous:
        raise ValueError("A must be a C-contiguous M x lda buffer")
    if N < 0 or N > lda:
        raise ValueError("need 0 <= N <= lda")
    if A.dtype not in _IN:
        raise TypeError(f"unsupported dtype {A.dtype}")
    p = np.ascontiguousarray(p, dtype=A.dtype)
    r = np.ascontiguousarray(r, dtype=A.dtype)
    if p.shape != (N,) or r.shape != (M,):
        raise ValueError("p must have N elements and r must have M elements")
    return M, N, max(lda, 1), p, r


def dualmv(A: np.ndarray, p: np.ndarray, r: np.ndarray, N: int | None = None,
           lib=None):
    """Return ``(q, s)`` for one matrix.

    ``A`` is the M x lda storage (C-contiguous); only its first ``N`` columns
    (default: all of them) belong to the matrix.
    """
    lib = lib or load()
    M, N, lda, p, r = _prep(A, p, r, N)
    tag, out_t = _IN[A.dtype]
    q = np.zeros(M, dtype=out_t)
    s = np.zeros(N, dtype=out_t)
    rc = getattr(lib, f"oracle_dualmv_{tag}")(M, N, _ptr(A), lda, _ptr(p),
                                             _ptr(r), _ptr(q), _ptr(s))
    if rc != 0:
        raise RuntimeError(f"oracle_dualmv_{tag} returned {rc}")
    return q, s


def absdot(A: np.ndarray, p: np.ndarray, r: np.ndarray, N: int | None = None,
           lib=None):
    """Return ``(sum_j |A_ij||p_j|, sum_i |A_ij||r_i|)`` in float64."""
    lib = lib or load()
    M, N, lda, p, r = _prep(A, p, r, N)
    tag = "f32" if A.dtype == np.float32 else "f64"
    if A.dtype == np.int32:
        A = A.astype(np.float64)
        p = p.astype(np.float64)
        r = r.astype(np.float64)
        tag = "f64"
    qa = np.zeros(M, dtype=np.float64)
    sa = np.zeros(N, dtype=np.float64)
    rc = getattr(lib, f"oracle_absdot_{tag}")(M, N, _ptr(A), lda, _ptr(p),
                                             _ptr(r), _ptr(qa), _ptr(sa))
    if rc != 0:
        raise RuntimeError(f"oracle_absdot_{tag} returned {rc}")
    return qa, sa


def dualmv_batched(A: np.ndarray, p: np.ndarray, r: np.ndarray,
                   N: int | None = None, lib=None):
    """Batched form: ``A`` is B x M x lda, ``p`` is B x N, ``r`` is B x M.

    Each problem is independent; this is a plain loop over the batch.
    """
    qs, ss = [], []
    for b in range(A.shape[0]):
        q, s = dualmv(A[b], p[b], r[b], N=N, lib=lib)
        qs.append(q)
        ss.append(s)
    out_t = _IN[A.dtype][1]
    M = A.shape[1]
    N = A.shape[2] if N is None else N
    if not qs:
        return np.zeros((0, M), out_t), np.zeros((0, N), out_t)
    return np.stack(qs), np.stack(ss)


def trimmed_mean(times, k: int, lib=None) -> float:
    """Eq. 3 of the paper: mean of the sorted timings without the k lowest
    and the k highest (requires R > 2k)."""
    lib = lib or load()
    t = np.array(times, dtype=np.float64)
    out = np.zeros(1, dtype=np.float64)
    rc = lib.oracle_trimmed_mean(_ptr(t), t.size, int(k), _ptr(out))
    if rc != 0:
        raise ValueError("trimmed mean needs R > 2k and k >= 0")
    return float(out[0])


def _float_tag(A: np.ndarray) -> str:
    if A.dtype == np.float32:
        return "f32"
    if A.dtype == np.float64:
        return "f64"
    raise TypeError(f"unsupported dtype {A.dtype}")


def gesummv(A: np.ndarray, B: np.ndarray, x: np.ndarray, alpha: float, beta: float,
            N: int | None = None, lib=None) -> np.ndarray:
    """GESUMMV (Table 1 / Table 2): y = alpha (A x) + beta (B x), in float64.

    A and B are M x lda and M x ldb C-contiguous storage; only their first
    N columns (default: all of A's) belong to the matrices."""
    lib = lib or load()
    tag = _float_tag(A)
    if B.dtype != A.dtype or A.ndim != 2 or B.ndim != 2 or A.shape[0] != B.shape[0]:
        raise ValueError("A and B must be 2-D with the same dtype and row count")
    if not (A.flags.c_contiguous and B.flags.c_contiguous):
        raise ValueError("A and B must be C-contiguous")
    M = A.shape[0]
    N = A.shape[1] if N is None else int(N)
    if N > A.shape[1] or N > B.shape[1]:
        raise ValueError("N exceeds a leading dimension")
    x = np.ascontiguousarray(x, dtype=A.dtype)
    if x.shape != (N,):
        raise ValueError("x must have N elements")
    y = np.zeros(M, dtype=np.float64)
    rc = getattr(lib, f"oracle_gesummv_{tag}")(M, N, float(alpha), _ptr(A), max(A.shape[1], 1),
                                               float(beta), _ptr(B), max(B.shape[1], 1),
                                               _ptr(x), _ptr(y))
    if rc != 0:
        raise RuntimeError(f"oracle_gesummv_{tag} returned {rc}")
    return y


def atax(A: np.ndarray, x: np.ndarray, N: int | None = None, lib=None) -> np.ndarray:
    """ATAX (Table 1): y = A^T (A x), in float64 (A is M x lda storage)."""
    lib = lib or load()
    tag = _float_tag(A)
    if A.ndim != 2 or not A.flags.c_contiguous:
        raise ValueError("A must be a C-contiguous 2-D buffer")
    M = A.shape[0]
    N = A.shape[1] if N is None else int(N)
    x = np.ascontiguousarray(x, dtype=A.dtype)
    if x.shape != (N,) or N > A.shape[1]:
        raise ValueError("x must have N elements, N <= lda")
    y = np.zeros(N, dtype=np.float64)
    rc = getattr(lib, f"oracle_atax_{tag}")(M, N, _ptr(A), max(A.shape[1], 1), _ptr(x), _ptr(y))
    if rc != 0:
        raise RuntimeError(f"oracle_atax_{tag} returned {rc}")
    return y


def gemver(A: np.ndarray, u1, v1, u2, v2, w, x, y, z, alpha: float, beta: float,
           N: int | None = None, lib=None):
    """GEMVER (Table 1 / Table 2): returns ``(A_hat, w_new, x_new)`` in
    float64 for A_hat = A + u1 v1^T + u2 v2^T, x_new = x + beta A_hat^T y
    + z, w_new = w + alpha A_hat x_new (A is M x lda storage)."""
    lib = lib or load()
    tag = _float_tag(A)
    if A.ndim != 2 or not A.flags.c_contiguous:
        raise ValueError("A must be a C-contiguous 2-D buffer")
    M = A.shape[0]
    N = A.shape[1] if N is None else int(N)
    vecs = [np.ascontiguousarray(v, dtype=A.dtype) for v in (u1, v1, u2, v2, w, x, y, z)]
    want = [M, N, M, N, M, N, M, N]
    if any(v.shape != (n,) for v, n in zip(vecs, want)):
        raise ValueError("vector lengths do not match A")
    ahat = np.zeros((M, N), dtype=np.float64)
    wo = np.zeros(M, dtype=np.float64)
    xo = np.zeros(N, dtype=np.float64)
    rc = getattr(lib, f"oracle_gemver_{tag}")(M, N, float(alpha), float(beta), _ptr(A),
                                              max(A.shape[1], 1), *[_ptr(v) for v in vecs],
                                              _ptr(ahat), _ptr(wo), _ptr(xo))
    if rc != 0:
        raise RuntimeError(f"oracle_gemver_{tag} returned {rc}")
    return ahat, wo, xo
