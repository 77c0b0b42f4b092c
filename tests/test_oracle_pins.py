"""The CPU oracle against values fixed by mathematics (no GPU needed)."""
import numpy as np
import pytest

import oracle
import oracle_pins as P


@pytest.fixture(scope="module")
def lib():
    return oracle.load()


@pytest.mark.parametrize("pin", P.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(lib, pin):
    pin(lib)


def test_batched_is_independent_problems(lib):
    """The batched oracle solves each problem with its own p and r."""
    rng = np.random.default_rng(3)
    A = rng.uniform(-1, 1, (3, 5, 7))
    p = rng.uniform(-1, 1, (3, 7))
    r = rng.uniform(-1, 1, (3, 5))
    q, s = oracle.dualmv_batched(A, p, r, lib=lib)
    for b in range(3):
        qb, sb = oracle.dualmv(A[b], p[b], r[b], lib=lib)
        assert (q[b] == qb).all() and (s[b] == sb).all()


def test_rejects_bad_arguments(lib):
    with pytest.raises(ValueError):
        oracle.dualmv(np.zeros((2, 3)), np.zeros(4), np.zeros(2), lib=lib)
    with pytest.raises(ValueError):
        oracle.dualmv(np.zeros((2, 3)), np.zeros(3), np.zeros(3), lib=lib)
