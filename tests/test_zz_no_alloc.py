"""dualmv_f32_noalloc: the entry point for callers that cannot allocate
device memory during the call (frameworks that own every allocation, loops
that must stay out of allocators).  It keeps its scratch in a fixed array
inside the library.  These tests check, through the C ABI:

  * two calls in a row give dualmv_f32's results and the oracle's, within
    the f32 bar, on both of its branches (TMA for aligned rows, plain loads
    for an odd row stride or a base off the 16-byte grid);
  * those calls take nothing from the library's workspace pool or from the
    device (cudaMemGetInfo) and create no torch allocation;
  * problems too large for the array are refused.

This file is collected last on purpose: a failure here comes after every
other test has run.  It also passes alone in a fresh process (the first
call of the library on the device is made before the measured calls)."""
import numpy as np
import pytest
import torch

import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import inputs
from parity import TOL, compare_problem, scaled_error

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _noalloc_into(Av, p, r, q, s):
    M, N = Av.shape
    rc = dm.dualmv_f32_noalloc(M, N, Av.data_ptr(), Av.stride(0), p.data_ptr(),
                               r.data_ptr(), q.data_ptr(), s.data_ptr(),
                               torch.cuda.current_stream().cuda_stream)
    assert rc == dm.DUALMV_SUCCESS, dm.dualmv_status_string(rc)


def _problem(M, N, lda, seed, col0=0):
    """Seeded f32 problem; the matrix is columns col0 .. col0 + N - 1 of an
    M x lda buffer (col0 = 1 puts its base 4 bytes off the 16-byte grid)."""
    w = inputs.Workload("noalloc", "f32", M, lda, lda, "uniform", seed)
    A, _, r = inputs.generate(w, DEV)
    g = torch.Generator(device=DEV).manual_seed(seed + 1000)
    p = torch.empty(N, dtype=torch.float32, device=DEV).uniform_(-1, 1, generator=g)
    return A, A[:, col0:col0 + N], p, r


# (M, N, lda, col0): aligned rows (TMA branch), an odd row stride and a
# misaligned base (plain-load branch).
CASES = [(16384, 16384, 16384, 0), (1000, 3001, 3004, 0), (77, 200, 200, 0),
         (1000, 3001, 3001, 0), (513, 2047, 2048, 1)]


@pytest.mark.parametrize("M,N,lda,col0", CASES)
def test_two_calls_in_a_row_match_dualmv_f32_and_the_oracle(M, N, lda, col0):
    dev = torch.cuda.current_device()
    probs = [_problem(M, N, lda, seed, col0) for seed in (31, 32)]
    outs = [(torch.empty(M, device=DEV), torch.empty(N, device=DEV)) for _ in probs]
    # The existing entry point's results (it takes workspace from the pool),
    # and one call of the new one, which does its once-per-device set-up.
    refs = [dm.dualmv(Av, p, r) for _, Av, p, r in probs]
    _noalloc_into(probs[0][1], probs[0][2], probs[0][3], *outs[0])
    torch.cuda.synchronize()

    # Two calls in a row, the second reusing the scratch the first left.
    _, high_before = dm.dualmv_pool_usage(dev, reset_high=True)
    free_before = torch.cuda.mem_get_info()[0]
    allocs_before = torch.cuda.memory_stats().get("allocation.all.allocated", 0)
    for (_, Av, p, r), (q, s) in zip(probs, outs):
        _noalloc_into(Av, p, r, q, s)
    torch.cuda.synchronize()
    _, high_after = dm.dualmv_pool_usage(dev)
    assert high_after == 0, f"workspace pool in use during the calls: {high_after} bytes"
    assert torch.cuda.mem_get_info()[0] == free_before
    assert torch.cuda.memory_stats().get("allocation.all.allocated", 0) == allocs_before
    assert dm.device_fault() == dm.DUALMV_SUCCESS

    for (A, Av, p, r), (q, s), (qr, sr) in zip(probs, outs, refs):
        # Against dualmv_f32, the existing entry point.
        den_q = (Av.abs().double() @ p.abs().double()).cpu().numpy()
        den_s = (r.abs().double() @ Av.abs().double()).cpu().numpy()
        err = max(scaled_error(q.cpu().numpy(), qr.double().cpu().numpy(), den_q),
                  scaled_error(s.cpu().numpy(), sr.double().cpu().numpy(), den_s))
        assert err <= TOL["f32"], err
        # Against the oracle, element by element.
        store = np.ascontiguousarray(A.cpu().numpy()[:, col0:])
        err = compare_problem("f32", q.cpu().numpy(), s.cpu().numpy(), store,
                              p.cpu().numpy(), r.cpu().numpy(), N)
        assert err <= TOL["f32"], err


def test_rejects_problems_beyond_the_scratch():
    assert dm.dualmv_f32_noalloc_scratch_bytes() == 8 << 20
    M, N = 32768, 16384
    A = torch.empty(M, N, dtype=torch.float32, device=DEV)
    p = torch.empty(N, device=DEV)
    r = torch.empty(M, device=DEV)
    q = torch.empty(M, device=DEV)
    s = torch.empty(N, device=DEV)
    rc = dm.dualmv_f32_noalloc(M, N, A.data_ptr(), N, p.data_ptr(), r.data_ptr(),
                               q.data_ptr(), s.data_ptr(), None)
    assert rc == dm.DUALMV_ERR_TOO_LARGE
    assert "scratch" in dm.dualmv_status_string(rc)
