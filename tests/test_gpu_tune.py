"""Kernel variants and the variant tuner on the GPU.  Every compiled variant
of every dtype is held to the parity bar against the oracle on shapes that
span several tiles with ragged tails; the tuner's loop (Section 3.2) is run
on a mid-size problem per dtype and its report, its recorded choice and its
outputs are checked; a mistake planted in every candidate's outputs must be
caught by the equivalence gate (Eq. 4).  The same for strided batches and
for single-sided passes (the building blocks of GESUMMV, GEMVER and ATAX's
two-pass path): every variant with single-sided instances against the
oracle through those operations, and the pass tuner's report and choice."""
import numpy as np
import pytest
import torch

import oracle
import paper_2512_22147_gb300 as dm
from paper_2512_22147_gb300 import inputs
from parity import TOL, compare_problem, run_and_compare, scaled_error

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
CODE = {"f32": dm.DUALMV_DTYPE_F32, "f64": dm.DUALMV_DTYPE_F64, "i32": dm.DUALMV_DTYPE_I32}
DIST = {"f32": "uniform", "f64": "normal", "i32": "int8"}


def _make(dtype, M, N, lda, seed):
    return inputs.generate(inputs.Workload("t", dtype, M, N, lda, DIST[dtype], seed), DEV)


def _all_variants():
    out = []
    for tag, code in CODE.items():
        for i in range(dm.dualmv_variant_count(code)):
            out.append((tag, i))
    return out


@pytest.fixture
def forced():
    olds = {}

    def force(tag, index):
        olds.setdefault(tag, dm.dualmv_set_variant(CODE[tag], index))
        dm.dualmv_set_variant(CODE[tag], index)

    yield force
    for tag in olds:
        dm.dualmv_set_variant(CODE[tag], -1)


@pytest.mark.parametrize("tag,index", _all_variants())
@pytest.mark.parametrize("M,N,pad", [(1000, 3000, 0), (3001, 257, 4), (77, 1000, 8),
                                     (4096, 256, 0), (1, 1, 0), (513, 5000, 4),
                                     (97, 2048, 0), (130, 4100, 8)])
def test_every_variant_matches_oracle(tag, index, M, N, pad, forced):
    forced(tag, index)
    A, p, r = _make(tag, M, N, N + pad, 100 + index + M)
    run_and_compare(A, p, r, N)


@pytest.mark.parametrize("tag,index", _all_variants())
def test_every_variant_is_deterministic(tag, index, forced):
    forced(tag, index)
    A, p, r = _make(tag, 2000, 2000, 2000, 7)
    q1, s1 = dm.dualmv(A, p, r)
    q2, s2 = dm.dualmv(A, p, r)
    torch.cuda.synchronize()
    assert torch.equal(q1, q2) and torch.equal(s1, s2)


@pytest.mark.parametrize("tag,index", _all_variants())
def test_forced_variant_is_the_one_launched(tag, index, forced):
    forced(tag, index)
    A, p, r = _make(tag, 500, 700, 700, 5)
    dm.dualmv(A, p, r)
    torch.cuda.synchronize()
    assert dm.dualmv_last_variant() == index


@pytest.mark.parametrize("tag,index", [("f32", 3), ("f32", 4), ("f64", 8)])
def test_other_summation_order_changes_bits(tag, index, forced):
    """A variant with another tile shape (or fp64 arithmetic) rounds
    differently: its outputs are not bit-identical to entry 0's on random
    data, which shows the variant really ran."""
    A, p, r = _make(tag, 4096, 4096, 4096, 21)
    q0, s0 = dm.dualmv(A, p, r)
    forced(tag, index)
    q1, s1 = dm.dualmv(A, p, r)
    torch.cuda.synchronize()
    assert not (torch.equal(q0, q1) and torch.equal(s0, s1))


@pytest.mark.parametrize("N,lda,expect", [(8192, 8192, 0), (8190, 8196, 8), (1000, 1004, 8),
                                          (4096, 4128, 0)])
def test_int32_default_follows_row_alignment(N, lda, expect):
    """Untuned int32 calls take the wide tiles when rows are not 128-byte
    aligned (lda * 4 not a multiple of 128), entry 0 otherwise."""
    dm.dualmv_tune_clear()
    A, p, r = _make("i32", 300, N, lda, 4)
    run_and_compare(A, p, r, N)
    assert dm.dualmv_last_variant() == expect


def test_int32_tuner_starts_from_the_shape_default():
    M, N, lda = 1000, 8190, 8196
    A, p, r = _make("i32", M, N, lda, 13)
    dm.dualmv_tune_clear()
    rep = dm.tune(A[:, :N], p, r, repeats=7, trim=1, max_rounds=2, candidates=4,
                  min_gain=0.0, flush_l2=False)
    torch.cuda.synchronize()
    assert rep["initial"] == 8
    assert all(s["index"] != 8 for s in rep["trace"])
    w = dm.dualmv_variant_info(dm.DUALMV_DTYPE_I32, 8)
    twin = [i for i in range(dm.dualmv_variant_count(dm.DUALMV_DTYPE_I32))
            if (lambda v: v.kernel == dm.DUALMV_KERNEL_STREAM and
                (v.warps, v.rows_per_warp, v.stages) == (w.warps, w.rows_per_warp, w.stages))(
                dm.dualmv_variant_info(dm.DUALMV_DTYPE_I32, i))]
    assert len(twin) == 1   # the same tile numbers on the other kernel kind
    assert any(s["index"] == twin[0] for s in rep["trace"])
    err = compare_problem("i32", rep["q"].cpu().numpy(), rep["s"].cpu().numpy(),
                          A.cpu().numpy(), p.cpu().numpy(), r.cpu().numpy(), N)
    assert err == 0.0
    dm.dualmv_tune_clear()


def _tune(tag, M, N, **kw):
    A, p, r = _make(tag, M, N, N, 11)
    dm.dualmv_tune_clear()
    rep = dm.tune(A, p, r, **kw)
    torch.cuda.synchronize()
    return A, p, r, rep


@pytest.mark.parametrize("tag", ["f32", "f64", "i32"])
def test_tuner_report_and_choice(tag):
    M, N = 4096, 8192
    A, p, r, rep = _tune(tag, M, N, repeats=12, trim=2, max_rounds=3, candidates=4,
                         min_gain=0.0, flush_l2=True)
    n = dm.dualmv_variant_count(CODE[tag])
    assert 0 <= rep["best"] < n
    assert 1 <= rep["rounds"] <= 3
    assert rep["evaluated"] >= 1 and rep["rejected"] == 0
    assert rep["baseline_ms"] > 0 and 0 < rep["best_ms"] <= rep["baseline_ms"]
    assert rep["worst_fe"] <= TOL[tag]
    tr = rep["trace"]
    assert len(tr) == rep["evaluated"] and all(s["feasible"] for s in tr)
    assert all(0 < s["ms"] and s["fe"] <= TOL[tag] for s in tr)
    assert [s["round"] for s in tr] == sorted(s["round"] for s in tr)
    if tag != "i32":   # round 0 holds variants with another summation order
        assert max(s["fe"] for s in tr) > 0
    best_seen = min([rep["baseline_ms"]] + [s["ms"] for s in tr])
    assert rep["best_ms"] == best_seen or rep["best"] == 0
    assert dm.dualmv_tuned_variant(CODE[tag], M, N, N) == rep["best"]
    # The tuner's outputs are the chosen variant's, and they pass parity.
    err = compare_problem(tag, rep["q"].cpu().numpy(), rep["s"].cpu().numpy(),
                          A.cpu().numpy(), p.cpu().numpy(), r.cpu().numpy(), N)
    assert err <= TOL[tag]
    # Later calls of this shape run the recorded variant: same bits.
    q, s = dm.dualmv(A, p, r)
    torch.cuda.synchronize()
    assert torch.equal(q, rep["q"]) and torch.equal(s, rep["s"])
    dm.dualmv_tune_clear()
    assert dm.dualmv_tuned_variant(CODE[tag], M, N, N) == -1


@pytest.mark.parametrize("tag", ["f32", "i32"])
def test_equivalence_gate_rejects_planted_mistake(tag, monkeypatch):
    monkeypatch.setenv("DUALMV_FAULT_INJECT", "fe")
    A, p, r, rep = _tune(tag, 2048, 2048, repeats=7, trim=1, max_rounds=2, candidates=3,
                         min_gain=0.0, flush_l2=False)
    assert rep["evaluated"] >= 1
    assert rep["rejected"] == rep["evaluated"]
    assert all(not s["feasible"] and s["fe"] > TOL[tag] for s in rep["trace"])
    assert rep["best"] == 0 and rep["best_ms"] == rep["baseline_ms"]
    # The outputs left behind are the default variant's, which are correct.
    err = compare_problem(tag, rep["q"].cpu().numpy(), rep["s"].cpu().numpy(),
                          A.cpu().numpy(), p.cpu().numpy(), r.cpu().numpy(), 2048)
    assert err <= TOL[tag]
    dm.dualmv_tune_clear()


def test_tuner_off_the_tma_path_runs_default():
    A, p, r = _make("f32", 300, 301, 301, 3)   # 301 * 4 bytes: not a multiple of 16
    dm.dualmv_tune_clear()
    rep = dm.tune(A, p, r, repeats=7, trim=1)
    torch.cuda.synchronize()
    assert rep["evaluated"] == 0 and rep["best"] == 0
    err = compare_problem("f32", rep["q"].cpu().numpy(), rep["s"].cpu().numpy(),
                          A.cpu().numpy(), p.cpu().numpy(), r.cpu().numpy(), 301)
    assert err <= TOL["f32"]
    assert dm.dualmv_tuned_variant(dm.DUALMV_DTYPE_F32, 300, 301, 301) == -1


# ---- strided batches --------------------------------------------------------

def _batched_variants():
    return [(tag, i) for tag, code in CODE.items() for i in range(dm.dualmv_variant_count(code))
            if dm.dualmv_variant_info(code, i).batched]


def _make_batched(dtype, B, M, N, lda, seed):
    w = inputs.Workload("tb", dtype, M, N, lda, DIST[dtype], seed, batch=B)
    return inputs.generate(w, DEV)


# Row strides and problem strides are multiples of 16 bytes (the 3-D tensor
# map); ragged M and N, one band, many bands.
BATCHED_SHAPES = [(3, 513, 1000, 4), (5, 64, 3000, 4), (2, 1000, 257, 7), (4, 1, 300, 4)]


@pytest.mark.parametrize("tag,index", _batched_variants())
@pytest.mark.parametrize("B,M,N,pad", BATCHED_SHAPES)
def test_every_batched_variant_matches_oracle(tag, index, B, M, N, pad, forced):
    forced(tag, index)
    A, p, r = _make_batched(tag, B, M, N, N + pad, 300 + index + M)
    run_and_compare(A, p, r, N)
    assert dm.dualmv_last_variant() == index


def test_batched_calls_run_entry_zero_for_a_variant_without_batched_instance(forced):
    for tag, code in CODE.items():
        plain = [i for i in range(dm.dualmv_variant_count(code))
                 if not dm.dualmv_variant_info(code, i).batched]
        if not plain:
            continue
        forced(tag, plain[0])
        A, p, r = _make_batched(tag, 3, 300, 700, 704, 9)
        run_and_compare(A, p, r, 700)
        assert dm.dualmv_last_variant() == 0, (tag, plain[0])


@pytest.mark.parametrize("tag", ["f32", "f64", "i32"])
def test_batched_tuner_report_and_choice(tag):
    B, M, N = 16, 1024, 2048
    A, p, r = _make_batched(tag, B, M, N, N, 17)
    code = CODE[tag]
    dm.dualmv_tune_clear()
    rep = dm.tune(A, p, r, repeats=9, trim=2, max_rounds=2, candidates=3, min_gain=0.0,
                  flush_l2=True)
    torch.cuda.synchronize()
    assert rep["initial"] == 0
    assert dm.dualmv_variant_info(code, rep["best"]).batched == 1
    assert rep["evaluated"] >= 1 and rep["rejected"] == 0
    assert all(dm.dualmv_variant_info(code, st["index"]).batched for st in rep["trace"])
    assert 0 < rep["best_ms"] <= rep["baseline_ms"]
    assert rep["worst_fe"] <= TOL[tag]
    # The outputs the tuner left are the chosen variant's: against the oracle.
    An, pn, rn = A.cpu().numpy(), p.cpu().numpy(), r.cpu().numpy()
    qg, sg = rep["q"].cpu().numpy(), rep["s"].cpu().numpy()
    for b in range(B):
        assert compare_problem(tag, qg[b], sg[b], An[b], pn[b], rn[b], N) <= TOL[tag]
    # Recorded for (dtype, M, N, lda, batch) and used by later batched calls;
    # the single-problem record and other batch counts are untouched.
    assert dm.dualmv_tuned_variant_batched(code, M, N, N, B) == rep["best"]
    assert dm.dualmv_tuned_variant(code, M, N, N) == -1
    assert dm.dualmv_tuned_variant_batched(code, M, N, N, B + 1) == -1
    dm.dualmv(A, p, r)
    torch.cuda.synchronize()
    assert dm.dualmv_last_variant() == rep["best"]
    dm.dualmv_tune_clear()


def test_batched_tuner_catches_a_planted_mistake(monkeypatch):
    monkeypatch.setenv("DUALMV_FAULT_INJECT", "fe")
    A, p, r = _make_batched("f32", 8, 512, 1024, 1024, 23)
    dm.dualmv_tune_clear()
    rep = dm.tune(A, p, r, repeats=7, trim=1, max_rounds=2, candidates=3, min_gain=0.0,
                  flush_l2=False)
    torch.cuda.synchronize()
    assert rep["evaluated"] >= 1 and rep["rejected"] == rep["evaluated"]
    assert rep["best"] == 0
    dm.dualmv_tune_clear()


# ---- single-sided passes --------------------------------------------------

def _sided_variants():
    out = []
    for tag in ("f32", "f64"):
        code = CODE[tag]
        for i in range(dm.dualmv_variant_count(code)):
            if dm.dualmv_variant_info(code, i).single_sided:
                out.append((tag, i))
    return out


@pytest.fixture
def two_pass_atax():
    old = dm.dualmv_atax_set_two_pass(1)
    yield
    dm.dualmv_atax_set_two_pass(old)


@pytest.mark.parametrize("tag,index", _sided_variants())
@pytest.mark.parametrize("M,N,pad", [(1000, 3000, 0), (3001, 257, 4), (77, 2048, 8)])
def test_every_single_sided_variant_matches_oracle(tag, index, M, N, pad, forced,
                                                   two_pass_atax):
    """A forced variant with single-sided instances runs GESUMMV's two rows
    passes, ATAX's two passes (rows, then columns) and GEMVER's columns pass:
    each result against the oracle, and the variant reported launched (entry
    0 is the passes' default kernel, reported as no variant; rows off the
    16-byte grid take the plain-load path, which has no variants)."""
    from test_gpu_ops import check_atax, check_gemver, check_gesummv
    forced(tag, index)
    aligned = ((N + pad) * (4 if tag == "f32" else 8)) % 16 == 0
    launched = index if (index != 0 and aligned) else -1
    seed = 300 + index + M
    A, B, x = inputs.generate_gesummv(
        inputs.Workload("g", tag, M, N, N + pad, DIST[tag], seed, op="gesummv"), DEV)
    check_gesummv(A, B, x, N, 0.75, -1.25, tag)
    assert dm.dualmv_last_variant() == launched
    A, x = inputs.generate_atax(
        inputs.Workload("a", tag, M, N, N + pad, DIST[tag], seed + 1, op="atax"), DEV)
    check_atax(A, x, N, tag)
    assert dm.dualmv_atax_last_path() == dm.DUALMV_ATAX_TWO_PASS
    assert dm.dualmv_last_variant() == launched
    ops = inputs.generate_gemver(
        inputs.Workload("v", tag, M, N, N + pad, DIST[tag], seed + 2, op="gemver"), DEV)
    check_gemver(ops, N, 1.5, -0.75, False, tag)


def _pass_oracle(tag, A, x, rows):
    An, xn = A.cpu().numpy(), x.cpu().numpy()
    M, N = An.shape
    if rows:
        want, _ = oracle.dualmv(An, xn, np.zeros(M, An.dtype))
        den, _ = oracle.absdot(An, xn, np.zeros(M, An.dtype))
    else:
        _, want = oracle.dualmv(An, np.zeros(N, An.dtype), xn)
        _, den = oracle.absdot(An, np.zeros(N, An.dtype), xn)
    return want, den


@pytest.mark.parametrize("tag", ["f32", "f64"])
@pytest.mark.parametrize("pass_", ["rows", "cols"])
def test_pass_tuner_report_and_choice(tag, pass_, two_pass_atax):
    M, N = 4096, 8192
    A, p, r = _make(tag, M, N, N, 31)
    rows = pass_ == "rows"
    x = p if rows else r
    code = CODE[tag]
    pid = dm.DUALMV_PASS_ROWS if rows else dm.DUALMV_PASS_COLS
    other = dm.DUALMV_PASS_COLS if rows else dm.DUALMV_PASS_ROWS
    dm.dualmv_tune_clear()
    rep = dm.tune_pass(A, x, pass_, repeats=9, trim=2, max_rounds=2, candidates=3,
                       min_gain=0.0, flush_l2=True)
    torch.cuda.synchronize()
    assert rep["initial"] == (1 if tag == "f64" else 0)   # the passes' default
    assert dm.dualmv_variant_info(code, rep["best"]).single_sided == 1
    assert rep["evaluated"] >= 1 and rep["rejected"] == 0
    assert all(dm.dualmv_variant_info(code, st["index"]).single_sided for st in rep["trace"])
    assert 0 < rep["best_ms"] <= rep["baseline_ms"]
    assert rep["worst_fe"] <= TOL[tag]
    # The result the tuner left is the chosen variant's: against the oracle.
    want, den = _pass_oracle(tag, A, x, rows)
    assert scaled_error(rep["out"].cpu().numpy(), want, den) <= TOL[tag]
    # Recorded for (dtype, M, N, lda, pass) only.
    assert dm.dualmv_tuned_variant_pass(code, M, N, N, pid) == rep["best"]
    assert dm.dualmv_tuned_variant_pass(code, M, N, N, other) == -1
    assert dm.dualmv_tuned_variant(code, M, N, N) == -1
    # A later forward pass of that shape runs it: GESUMMV's passes (rows),
    # ATAX's columns pass (cols).
    launched = rep["best"] if rep["best"] != 0 else -1
    if rows:
        dm.gesummv(A, A, p)
    else:
        dm.atax(A, p)
    torch.cuda.synchronize()
    assert dm.dualmv_last_variant() == launched
    dm.dualmv_tune_clear()
    assert dm.dualmv_tuned_variant_pass(code, M, N, N, pid) == -1


def test_pass_tuner_catches_a_planted_mistake(monkeypatch):
    monkeypatch.setenv("DUALMV_FAULT_INJECT", "fe")
    A, p, r = _make("f32", 2048, 2048, 2048, 37)
    dm.dualmv_tune_clear()
    rep = dm.tune_pass(A, r, "cols", repeats=7, trim=1, max_rounds=2, candidates=3,
                       min_gain=0.0, flush_l2=False)
    torch.cuda.synchronize()
    assert rep["evaluated"] >= 1 and rep["rejected"] == rep["evaluated"]
    assert all(not s["feasible"] and s["fe"] > TOL["f32"] for s in rep["trace"])
    assert rep["best"] == 0
    want, den = _pass_oracle("f32", A, r, False)
    assert scaled_error(rep["out"].cpu().numpy(), want, den) <= TOL["f32"]
    dm.dualmv_tune_clear()
