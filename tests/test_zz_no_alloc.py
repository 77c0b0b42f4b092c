"""dualmv_f32_noalloc: the entry point for callers that cannot allocate
device memory during the call (frameworks that own every allocation, loops
that must stay out of allocators).  It keeps its scratch in a fixed array
inside the library, so these tests check that it gives the same results as
dualmv_f32, call after call, and that it refuses problems too large for the
array.  This file is collected last on purpose: a failure here comes after
every other test has run."""
import pytest
import torch

import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import inputs
from parity import TOL, scaled_error

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _noalloc(Av, p, r):
    M, N = Av.shape
    q = torch.empty(M, dtype=torch.float32, device=DEV)
    s = torch.empty(N, dtype=torch.float32, device=DEV)
    rc = dm.dualmv_f32_noalloc(M, N, Av.data_ptr(), Av.stride(0), p.data_ptr(),
                               r.data_ptr(), q.data_ptr(), s.data_ptr(),
                               torch.cuda.current_stream().cuda_stream)
    assert rc == dm.DUALMV_SUCCESS, dm.dualmv_status_string(rc)
    return q, s


def _check_against_dualmv_f32(Av, p, r, qn, sn):
    q, s = dm.dualmv(Av, p, r)
    torch.cuda.synchronize()
    den_q = (Av.abs().double() @ p.abs().double()).cpu().numpy()
    den_s = (r.abs().double() @ Av.abs().double()).cpu().numpy()
    err = max(scaled_error(qn.cpu().numpy(), q.double().cpu().numpy(), den_q),
              scaled_error(sn.cpu().numpy(), s.double().cpu().numpy(), den_s))
    assert err <= TOL["f32"], err


@pytest.mark.parametrize("M,N,lda", [(16384, 16384, 16384), (1000, 3001, 3004), (77, 200, 200)])
def test_two_calls_in_a_row_match_dualmv_f32(M, N, lda):
    for seed in (31, 32):   # the second call reuses the scratch the first one left
        w = inputs.Workload("noalloc", "f32", M, N, lda, "uniform", seed)
        A, p, r = inputs.generate(w, DEV)
        Av = A[:, :N]
        qn, sn = _noalloc(Av, p, r)
        _check_against_dualmv_f32(Av, p, r, qn, sn)
    assert dm.device_fault() == dm.DUALMV_SUCCESS


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
