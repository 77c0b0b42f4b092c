"""Failure detection on the GPU without a fault: a bounded wait that runs out.

Every wait in the library's kernels (on a TMA stage, a peer CTA's partials
or a cluster barrier) gives up after about 2 s, sets the device fault word
and lets the kernel exit, so the host sees DUALMV_ERR_TIMEOUT from
dualmv_device_fault instead of a hung GPU.  dualmv_selftest_wait_timeout
runs those same waits on an mbarrier phase that nothing completes.  These
tests check, for the CTA-scope and the cluster-scope wait:

  * the wait runs out (the kernel reports it did not complete) after about
    the 2 s bound, not at once and not much later;
  * dualmv_device_fault reports DUALMV_ERR_TIMEOUT once, then clears;
  * the context stays usable: a dual product on the same stream right after
    gives the oracle's results and leaves no fault."""
import time

import pytest
import torch

import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import inputs
from parity import TOL, compare_problem

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.mark.parametrize("cluster_scope", [0, 1], ids=["cta", "cluster"])
def test_a_bounded_wait_runs_out_and_the_context_stays_usable(cluster_scope):
    stream = torch.cuda.current_stream(DEV)
    torch.cuda.synchronize()
    assert dm.device_fault() == dm.DUALMV_SUCCESS  # nothing left from earlier tests
    waited = torch.full((1,), 7, dtype=torch.int32, device=DEV)
    t0 = time.monotonic()
    rc = dm.dualmv_selftest_wait_timeout(cluster_scope, waited.data_ptr(), stream.cuda_stream)
    assert rc == dm.DUALMV_SUCCESS, dm.dualmv_status_string(rc)
    assert dm.device_fault() == dm.DUALMV_ERR_TIMEOUT
    elapsed = time.monotonic() - t0
    assert int(waited.item()) == 0
    assert 1.5 <= elapsed <= 30.0, elapsed
    assert dm.device_fault() == dm.DUALMV_SUCCESS  # read once, then cleared

    w = inputs.Workload("after", "f32", 700, 900, 904, "uniform", 71)
    A, p, r = inputs.generate(w, DEV)
    q, s = dm.dualmv(A[:, :w.N], p, r)
    torch.cuda.synchronize()
    assert dm.device_fault() == dm.DUALMV_SUCCESS
    err = compare_problem("f32", q.cpu().numpy(), s.cpu().numpy(), A.cpu().numpy(),
                          p.cpu().numpy(), r.cpu().numpy(), w.N)
    assert err <= TOL["f32"], err


def test_a_null_result_pointer_is_refused():
    assert dm.dualmv_selftest_wait_timeout(0, None, None) == dm.DUALMV_ERR_INVALID_VALUE
