"""Small fp32 dual products in one thread-block cluster (dualmv_small.cuh).

A call of at most 8 MiB of A with 256 <= N <= 2048 (N and lda multiples of
4, A and p 16-byte aligned) runs as one cluster of 16 CTAs: each CTA owns
whole rows, so q is finished inside it, and the CTAs' column partials meet
through distributed shared memory.  These tests check the outputs against
the oracle on shapes across that range (ragged row counts, fewer rows than
CTAs, the largest N and size), that the path is the one taken, that
everything outside the range goes to the streaming kernels, and that
repeated calls give the same bits."""
import pytest
import torch

import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import inputs
from parity import TOL, run_and_compare

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _make(M, N, lda, seed):
    return inputs.generate(inputs.Workload("small", "f32", M, N, lda, "uniform", seed), DEV)


@pytest.mark.parametrize("M,N,lda", [
    (1024, 1024, 1024),     # the 4 MiB workload
    (1, 256, 256), (7, 260, 264), (15, 512, 516), (16, 2048, 2048), (17, 2044, 2048),
    (333, 700, 712), (4096, 512, 512), (2048, 1024, 1024),   # 8 MiB exactly
    (1000, 1028, 1028),     # N just past 1024: the 16-vector form
])
def test_cluster_path_matches_oracle(M, N, lda):
    A, p, r = _make(M, N, lda, M + N)
    err = run_and_compare(A, p, r, N)
    assert dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_CLUSTER, (M, N, lda)
    assert err <= TOL["f32"]


@pytest.mark.parametrize("M,N,lda,why", [
    (64, 2052, 2052, "N above 2048"),
    (64, 252, 252, "N below 256"),
    (64, 1022, 1022, "N not a multiple of 4"),
    (64, 1024, 1027, "lda not a multiple of 4"),
    (2049, 1024, 1024, "more than 8 MiB"),
])
def test_outside_the_range_takes_the_streaming_kernels(M, N, lda, why):
    A, p, r = _make(M, N, lda, 7)
    run_and_compare(A, p, r, N)
    assert dm.dualmv_last_kernel() != dm.DUALMV_KERNEL_CLUSTER, why


def test_misaligned_p_and_forced_paths_take_the_streaming_kernels():
    M, N = 300, 1024
    A, p, r = _make(M, N + 4, N + 4, 8)
    pp = torch.empty(N + 1, dtype=torch.float32, device=DEV)
    pp[1:] = p[:N]
    run_and_compare(A, pp[1:], r, N)            # p 4 bytes off the 16-byte grid
    assert dm.dualmv_last_kernel() != dm.DUALMV_KERNEL_CLUSTER
    for path in (dm.DUALMV_PATH_TMA, dm.DUALMV_PATH_DIRECT):
        old = dm.dualmv_set_path(path)
        try:
            run_and_compare(A, p[:N], r, N)
            assert dm.dualmv_last_kernel() != dm.DUALMV_KERNEL_CLUSTER
        finally:
            dm.dualmv_set_path(old)
    old = dm.dualmv_set_variant(dm.DUALMV_DTYPE_F32, 0)   # a forced variant, even entry 0
    try:
        run_and_compare(A, p[:N], r, N)
        assert dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_STREAM
    finally:
        dm.dualmv_set_variant(dm.DUALMV_DTYPE_F32, old)


def test_cluster_path_is_deterministic_and_agrees_with_the_stream_kernel():
    M, N = 1500, 1200
    A, p, r = _make(M, N, N, 9)
    outs = [dm.dualmv(A, p, r) for _ in range(3)]
    torch.cuda.synchronize()
    assert dm.dualmv_last_kernel() == dm.DUALMV_KERNEL_CLUSTER
    for q, s in outs[1:]:
        assert torch.equal(q, outs[0][0]) and torch.equal(s, outs[0][1])
    old = dm.dualmv_set_path(dm.DUALMV_PATH_TMA)
    try:
        q2, s2 = dm.dualmv(A, p, r)
    finally:
        dm.dualmv_set_path(old)
    den_q = A.abs().double() @ p.abs().double()
    den_s = r.abs().double() @ A.abs().double()
    assert float(((outs[0][0].double() - q2.double()).abs() / den_q).max()) <= 2 * TOL["f32"]
    assert float(((outs[0][1].double() - s2.double()).abs() / den_s).max()) <= 2 * TOL["f32"]
