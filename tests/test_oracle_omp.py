"""The all-core CPU baseline (oracle/oracle_omp.c) against the oracle.

It sums every output in the oracle's order, so its results must be the
oracle's bit for bit, for every dtype, with padded rows, widths that are
not a multiple of its column block, and empty shapes."""
import numpy as np
import pytest

import oracle


def _case(dtype, M, N, lda, seed):
    rng = np.random.default_rng(seed)
    if dtype == np.int32:
        A = rng.integers(-2**31, 2**31, (M, lda), dtype=np.int64).astype(np.int32)
        p = rng.integers(-2**31, 2**31, N, dtype=np.int64).astype(np.int32)
        r = rng.integers(-2**31, 2**31, M, dtype=np.int64).astype(np.int32)
    else:
        A = (rng.standard_normal((M, lda)) * np.exp2(rng.integers(-30, 30, (M, lda)))).astype(dtype)
        p = rng.standard_normal(N).astype(dtype)
        r = rng.standard_normal(M).astype(dtype)
    A[:, N:] = np.array(-7, dtype=dtype)  # padding: never read
    return A, p, r


@pytest.mark.parametrize("dtype", [np.float32, np.float64, np.int32])
@pytest.mark.parametrize("M,N,lda", [(1, 1, 1), (97, 1000, 1003), (300, 256, 256),
                                     (5, 5000, 5000), (0, 7, 7), (7, 0, 1)])
def test_all_core_baseline_matches_oracle_bitwise(dtype, M, N, lda):
    A, p, r = _case(dtype, M, N, lda, M * 31 + N)
    q1, s1 = oracle.dualmv(A, p, r, N=N)
    q2, s2 = oracle.dualmv_omp(A, p, r, N=N)
    assert q1.tobytes() == q2.tobytes() and s1.tobytes() == s2.tobytes()


def test_all_core_baseline_reports_its_threads():
    assert oracle.omp_threads() >= 1
