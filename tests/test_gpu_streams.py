"""Calls in flight together, and calls captured in a CUDA graph.

Every call takes its scratch from the library's stream-ordered pool, so
calls on different streams may run at once, and calls captured in a graph
replay with scratch of their own.  These tests check, for each path (the
single-cluster kernel, the fp32 and int32 streaming kernels, the
double-float fp64 kernel, a strided batch, GEMVER):

  * the same problems launched on several streams without waiting for one
    another give the bits of the same problems run one after another;
  * a graph of such calls, replayed several times, gives the bits of the
    eager calls, and those bits match the oracle;
  * GEMVER and GESUMMV, whose kernels run as programmatic dependents of one
    another (GEMVER's columns pass beside its u . y kernel, GESUMMV's pass
    over B after its pass over A): GEMVER on two streams at once, GESUMMV
    right after kernels that rewrote its inputs, and both replayed from a
    graph give the bits of the same calls run alone."""
import numpy as np
import pytest
import torch

import oracle
import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import inputs
from parity import TOL, compare_problem, scaled_error

pytestmark = pytest.mark.gpu
DEV = "cuda:0"

PROBLEMS = [
    inputs.Workload("cluster", "f32", 1024, 1024, 1024, "uniform", 41),
    inputs.Workload("stream32", "f32", 3000, 5000, 5000, "uniform", 42),
    inputs.Workload("f64e", "f64", 2000, 3000, 3000, "normal", 43),
    inputs.Workload("int32", "i32", 1000, 4100, 4104, "int8", 44),
    inputs.Workload("batch", "f32", 500, 700, 704, "uniform", 45, batch=3),
]


def _problems():
    out = []
    for w in PROBLEMS:
        A, p, r = inputs.generate(w, DEV)
        q, s = inputs.empty_outputs(w, DEV)
        out.append((w, A[..., :w.N], p, r, q, s))
    return out


def _check_oracle(w, A, p, r, q, s):
    An, pn, rn = A.cpu().numpy(), p.cpu().numpy(), r.cpu().numpy()
    qg, sg = q.cpu().numpy(), s.cpu().numpy()
    if w.batched:
        for b in range(w.batch):
            assert compare_problem(w.dtype, qg[b], sg[b], An[b], pn[b], rn[b], w.N) <= TOL[w.dtype]
    else:
        assert compare_problem(w.dtype, qg, sg, An, pn, rn, w.N) <= TOL[w.dtype]


def test_concurrent_streams_give_the_serial_bits():
    probs = _problems()
    serial = []
    for w, A, p, r, q, s in probs:
        dm.dualmv(A, p, r, q=q, s=s)
        torch.cuda.synchronize()
        serial.append((q.clone(), s.clone()))
        _check_oracle(w, A, p, r, q, s)
    streams = [torch.cuda.Stream(DEV) for _ in probs]
    for rep in range(3):
        for (w, A, p, r, q, s) in probs:
            q.zero_()
            s.zero_()
        torch.cuda.synchronize()
        # Each problem on its own stream, twice in a row, nothing in between.
        for st, (w, A, p, r, q, s) in zip(streams, probs):
            with torch.cuda.stream(st):
                dm.dualmv(A, p, r, q=q, s=s)
                dm.dualmv(A, p, r, q=q, s=s)
        torch.cuda.synchronize()
        assert dm.device_fault() == dm.DUALMV_SUCCESS
        for (w, A, p, r, q, s), (q0, s0) in zip(probs, serial):
            assert torch.equal(q, q0) and torch.equal(s, s0), (w.name, rep)


def test_graph_replays_give_the_eager_bits():
    probs = _problems()
    eager = []
    for w, A, p, r, q, s in probs:
        dm.dualmv(A, p, r, q=q, s=s)
        torch.cuda.synchronize()
        eager.append((q.clone(), s.clone()))
    side = torch.cuda.Stream(DEV)
    side.wait_stream(torch.cuda.current_stream(DEV))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        for w, A, p, r, q, s in probs:   # warm the pool on this stream first
            dm.dualmv(A, p, r, q=q, s=s)
        side.synchronize()
        with torch.cuda.graph(graph, stream=side):
            for w, A, p, r, q, s in probs:
                dm.dualmv(A, p, r, q=q, s=s)
    torch.cuda.current_stream(DEV).wait_stream(side)
    for rep in range(3):
        for (w, A, p, r, q, s) in probs:
            q.zero_()
            s.zero_()
        graph.replay()
        torch.cuda.synchronize()
        for (w, A, p, r, q, s), (q0, s0) in zip(probs, eager):
            assert torch.equal(q, q0) and torch.equal(s, s0), (w.name, rep)
    for w, A, p, r, q, s in probs:
        _check_oracle(w, A, p, r, q, s)
    del graph


def test_gemver_on_two_streams_at_once():
    """Two GEMVER problems (fp64 factorised and with update_A) on two
    streams at once give the bits of the same calls run one after another."""
    ops = [inputs.generate_gemver(inputs.Workload("g", "f64", 1500, 2000, 2000, "normal",
                                                  50 + k, op="gemver"), DEV) for k in range(2)]
    upd = [False, True]

    def run_all(concurrent):
        outs = []
        streams = [torch.cuda.Stream(DEV) for _ in ops]
        copies = [[t.clone() for t in o] for o in ops]
        torch.cuda.synchronize()
        for k, (st, c) in enumerate(zip(streams, copies)):
            A, u1, v1, u2, v2, w, x, y, z = c
            if concurrent:
                with torch.cuda.stream(st):
                    dm.gemver(A, u1, v1, u2, v2, w, x, y, z, alpha=1.5, beta=0.5,
                              update_A=upd[k])
            else:
                dm.gemver(A, u1, v1, u2, v2, w, x, y, z, alpha=1.5, beta=0.5, update_A=upd[k])
                torch.cuda.synchronize()
            outs.append((A, w, x))
        torch.cuda.synchronize()
        return outs

    serial = run_all(False)
    for _ in range(2):
        conc = run_all(True)
        for a, b in zip(serial, conc):
            for t0, t1 in zip(a, b):
                assert torch.equal(t0, t1)


@pytest.mark.parametrize("dtype", ["f64", "f32"])
def test_gesummv_back_to_back_sees_the_previous_writes(dtype):
    """GESUMMV's pass over B starts without waiting for the pass over A (it
    waits for that grid only before it exits).  Calls right after kernels
    that rewrote B and x, and a call whose x is the y the call before wrote,
    give the bits of the same calls with a synchronisation between them, and
    the oracle's values."""
    n = 1500
    dist = "normal" if dtype == "f64" else "uniform"
    A, B, x = inputs.generate_gesummv(
        inputs.Workload("g", dtype, n, n, n, dist, 60, op="gesummv"), DEV)

    def sequence(sync):
        Bc, xc = B.clone(), x.clone()
        torch.cuda.synchronize()
        y1 = dm.gesummv(A, Bc, xc, alpha=1.5, beta=0.5)
        if sync:
            torch.cuda.synchronize()
        Bc.mul_(-0.5)
        xc.add_(0.25)
        if sync:
            torch.cuda.synchronize()
        y2 = dm.gesummv(A, Bc, xc, alpha=0.5, beta=2.0)
        if sync:
            torch.cuda.synchronize()
        y3 = dm.gesummv(A, Bc, y2, alpha=1.0, beta=-1.0)
        torch.cuda.synchronize()
        return y1, y2, y3, Bc, xc

    ref = sequence(True)
    for _ in range(3):
        for t0, t1 in zip(sequence(False), ref):
            assert torch.equal(t0, t1)
    y1, y2, y3, Bc, xc = ref
    An, Bn = A.cpu().numpy(), Bc.cpu().numpy()
    want = oracle.gesummv(An, Bn, y2.cpu().numpy(), 1.0, -1.0, N=n)
    den = (np.abs(An) + np.abs(Bn)) @ np.abs(y2.cpu().numpy().astype(np.float64))
    assert scaled_error(y3.cpu().numpy(), want, den) <= TOL[dtype]


@pytest.mark.parametrize("dtype", ["f64", "f32"])
def test_gemver_and_gesummv_graph_replays_give_the_eager_bits(dtype):
    """GEMVER (its u . y kernel runs beside the columns pass, which waits for
    it only before it exits) and GESUMMV (the pass over B after the pass
    over A, the same way), captured in one CUDA graph: every replay gives the
    bits of the eager calls, and GESUMMV's y matches the oracle (GEMVER's
    parity is checked in test_gpu_ops.py)."""
    dist = "normal" if dtype == "f64" else "uniform"
    ops = inputs.generate_gemver(
        inputs.Workload("gv", dtype, 1500, 2000, 2000, dist, 80, op="gemver"), DEV)
    A, u1, v1, u2, v2, w, x, y, z = ops
    GA, GB, gx = inputs.generate_gesummv(
        inputs.Workload("gs", dtype, 1700, 1300, 1300, dist, 81, op="gesummv"), DEV)
    w0, x0 = w.clone(), x.clone()
    gy = torch.empty(1700, dtype=GA.dtype, device=DEV)

    def calls():
        dm.gemver(A, u1, v1, u2, v2, w, x, y, z, alpha=1.5, beta=0.5)
        dm.gesummv(GA, GB, gx, alpha=0.5, beta=2.0, y=gy)

    calls()
    torch.cuda.synchronize()
    eager = (w.clone(), x.clone(), gy.clone())
    side = torch.cuda.Stream(DEV)
    side.wait_stream(torch.cuda.current_stream(DEV))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        calls()                      # warm the pool on this stream first
        side.synchronize()
        with torch.cuda.graph(graph, stream=side):
            calls()
    torch.cuda.current_stream(DEV).wait_stream(side)
    for rep in range(3):
        w.copy_(w0)
        x.copy_(x0)
        gy.zero_()
        graph.replay()
        torch.cuda.synchronize()
        for t0, t1 in zip((w, x, gy), eager):
            assert torch.equal(t0, t1), rep
    assert dm.device_fault() == dm.DUALMV_SUCCESS
    An, Bn, xn = GA.cpu().numpy(), GB.cpu().numpy(), gx.cpu().numpy()
    want = oracle.gesummv(An, Bn, xn, 0.5, 2.0)
    den = 0.5 * (np.abs(An) @ np.abs(xn)) + 2.0 * (np.abs(Bn) @ np.abs(xn))
    assert scaled_error(gy.cpu().numpy(), want, den) <= TOL[dtype]
    del graph
