"""The variant tables and the tuner's host-side parts, on the CPU: the
tables describe compiled kernels that fit an SM, the neighbourhood the tuner
walks (variants differing in one property) reaches every entry, the forced
and tuned selections round-trip, the library's trimmed mean (Eq. 3) agrees
with the oracle's, and bad tuner arguments are rejected before any CUDA
call."""
import math
import random

import pytest

import oracle
import paper_2512_22147_gb300 as dm

DTYPES = [dm.DUALMV_DTYPE_F32, dm.DUALMV_DTYPE_F64, dm.DUALMV_DTYPE_I32]
SMEM_LIMIT = 227 * 1024
FAKE = 0x10000  # never dereferenced


def table(dtype):
    return [dm.dualmv_variant_info(dtype, i) for i in range(dm.dualmv_variant_count(dtype))]


@pytest.mark.parametrize("dtype", DTYPES)
def test_variant_tables_are_well_formed(dtype):
    tab = table(dtype)
    assert len(tab) >= 4
    keys = set()
    for i, v in enumerate(tab):
        assert v.index == i
        assert v.kernel in (dm.DUALMV_KERNEL_STREAM, dm.DUALMV_KERNEL_F64E, dm.DUALMV_KERNEL_WIDE)
        if v.kernel == dm.DUALMV_KERNEL_WIDE:   # one 256-column sub-band per warp
            assert v.tile_rows == v.rows_per_warp and v.band_cols == 256 * v.warps
        elif v.kernel == dm.DUALMV_KERNEL_F64E:
            assert v.tile_rows == v.warps * v.rows_per_warp and v.band_cols in (128, 256)
        else:
            assert v.tile_rows == v.warps * v.rows_per_warp and v.band_cols == 256
        assert v.threads == (v.warps + v.producer_warp) * 32
        assert v.producer_warp in (0, 1)
        if v.kernel != dm.DUALMV_KERNEL_F64E:
            assert v.producer_warp == 1
        assert 0 < v.smem_bytes <= SMEM_LIMIT
        assert v.rows_per_warp in (1, 2, 4, 8, 16) and v.stages >= 2
        if v.kernel != dm.DUALMV_KERNEL_F64E:
            assert v.native_cols == 0
        if v.packed:
            assert v.kernel == dm.DUALMV_KERNEL_F64E and v.native_cols == 0
        keys.add((v.kernel, v.warps, v.rows_per_warp, v.stages, v.native_cols,
                  v.producer_warp, v.packed, v.band_cols))
    assert len(keys) == len(tab), "two entries describe the same kernel"
    kinds = {v.kernel for v in tab}
    if dtype == dm.DUALMV_DTYPE_F32:
        assert kinds == {dm.DUALMV_KERNEL_STREAM}
    elif dtype == dm.DUALMV_DTYPE_I32:
        assert kinds == {dm.DUALMV_KERNEL_STREAM, dm.DUALMV_KERNEL_WIDE}
    else:
        assert kinds == {dm.DUALMV_KERNEL_STREAM, dm.DUALMV_KERNEL_F64E}


@pytest.mark.parametrize("dtype,elem,acc", [(dm.DUALMV_DTYPE_F32, 4, 4),
                                            (dm.DUALMV_DTYPE_F64, 8, 8),
                                            (dm.DUALMV_DTYPE_I32, 4, 8)])
def test_entry_zero_is_the_default_plan(dtype, elem, acc):
    v = dm.dualmv_variant_info(dtype, 0)
    pl = dm.dualmv_plan(4096, 4096, 1, elem, acc, 152)
    assert (v.tile_rows, v.band_cols, v.threads) == (pl.tile_rows, pl.band_cols, pl.threads)
    assert v.smem_bytes == pl.smem_bytes


def _neighbours(a, b):
    return sum((a.kernel != b.kernel, a.warps != b.warps, a.rows_per_warp != b.rows_per_warp,
                a.stages != b.stages, a.native_cols != b.native_cols,
                a.producer_warp != b.producer_warp, a.packed != b.packed,
                a.kernel == b.kernel and a.band_cols != b.band_cols)) == 1


@pytest.mark.parametrize("dtype", DTYPES)
def test_neighbourhood_reaches_every_variant(dtype):
    tab = table(dtype)
    seen, todo = {0}, [0]
    while todo:
        i = todo.pop()
        for j, v in enumerate(tab):
            if j not in seen and _neighbours(tab[i], v):
                seen.add(j)
                todo.append(j)
    assert seen == set(range(len(tab)))


def test_unknown_dtype_and_index():
    assert dm.dualmv_variant_count(7) == -1
    with pytest.raises(dm.DualmvError):
        dm.dualmv_variant_info(0, dm.dualmv_variant_count(0))
    with pytest.raises(dm.DualmvError):
        dm.dualmv_variant_info(5, 0)
    with pytest.raises(ValueError):
        dm.dualmv_set_variant(0, dm.dualmv_variant_count(0))
    with pytest.raises(ValueError):
        dm.dualmv_set_variant(3, 0)


@pytest.mark.parametrize("dtype", DTYPES)
def test_forced_variant_round_trip(dtype):
    old = dm.dualmv_set_variant(dtype, 2)
    try:
        assert old == -1
        assert dm.dualmv_set_variant(dtype, 1) == 2
    finally:
        assert dm.dualmv_set_variant(dtype, -1) == 1


def test_no_tuned_variant_recorded_by_default():
    dm.dualmv_tune_clear()
    assert dm.dualmv_tuned_variant(dm.DUALMV_DTYPE_F32, 16384, 16384, 16384) == -1


def test_trimmed_mean_agrees_with_oracle():
    rng = random.Random(5)
    for _ in range(200):
        R = rng.randint(1, 40)
        k = rng.randint(0, (R - 1) // 2)
        t = [rng.lognormvariate(0, 1) for _ in range(R)]
        got = dm.dualmv_trimmed_mean(t, k)
        want = oracle.trimmed_mean(t, k)
        assert math.isclose(got, want, rel_tol=1e-15, abs_tol=0.0), (R, k, got, want)
    assert dm.dualmv_trimmed_mean(list(range(1, 31)), 3) == 15.5


def test_trimmed_mean_rejects_small_samples():
    for R, k in ((0, 0), (2, 1), (6, 3), (5, -1)):
        with pytest.raises(dm.DualmvError):
            dm.dualmv_trimmed_mean([1.0] * R, k)


def _cfg(**kw):
    base = dict(repeats=10, trim=2, max_rounds=3, candidates=4, min_gain=0.0, flush_l2=0)
    base.update(kw)
    return dm.TuneConfig(base["repeats"], base["trim"], base["max_rounds"], base["candidates"],
                         base["min_gain"], base["flush_l2"])


@pytest.mark.parametrize("tag", ["f32", "f64", "i32"])
@pytest.mark.parametrize("cfg", [
    None, _cfg(repeats=4, trim=2), _cfg(trim=-1), _cfg(max_rounds=-1), _cfg(candidates=0),
    _cfg(min_gain=-0.1), _cfg(min_gain=float("nan")),
])
def test_tune_rejects_bad_configuration(tag, cfg):
    fn = getattr(dm, f"dualmv_tune_{tag}")
    res = dm.TuneResult()
    assert fn(64, 64, FAKE, 64, FAKE, FAKE, FAKE, FAKE, cfg, res, None) == \
        dm.DUALMV_ERR_INVALID_VALUE


@pytest.mark.parametrize("tag", ["f32", "f64", "i32"])
def test_tune_rejects_bad_problem(tag):
    fn = getattr(dm, f"dualmv_tune_{tag}")
    res = dm.TuneResult()
    assert fn(64, 64, FAKE, 63, FAKE, FAKE, FAKE, FAKE, _cfg(), res, None) == \
        dm.DUALMV_ERR_INVALID_VALUE
    assert fn(64, 64, None, 64, FAKE, FAKE, FAKE, FAKE, _cfg(), res, None) == \
        dm.DUALMV_ERR_INVALID_VALUE
    assert fn(64, 64, FAKE, 64, FAKE, FAKE, FAKE, FAKE, _cfg(), None, None) == \
        dm.DUALMV_ERR_INVALID_VALUE


def test_last_variant_before_any_call():
    assert dm.dualmv_last_variant() == -1


# ---- strided batches ------------------------------------------------------

def _batched_ids(tab):
    return {i for i, v in enumerate(tab) if v.batched}


@pytest.mark.parametrize("dtype", DTYPES)
def test_batched_instances(dtype):
    """Entry 0 (what untuned batched calls run) and every streaming-kernel
    shape have a batched instance; the wide int32 tiles do not; the tuner's
    walk over the batched entries reaches each of them from entry 0."""
    tab = table(dtype)
    ids = _batched_ids(tab)
    assert 0 in ids
    for i, v in enumerate(tab):
        if v.kernel == dm.DUALMV_KERNEL_STREAM and dtype != dm.DUALMV_DTYPE_F64:
            assert v.batched == 1, i
        if v.kernel == dm.DUALMV_KERNEL_WIDE:
            assert v.batched == 0, i
        assert v.batched in (0, 1)
    assert len(ids) >= 4
    seen, todo = {0}, [0]
    while todo:
        i = todo.pop()
        for j in ids:
            if j not in seen and _neighbours(tab[i], tab[j]):
                seen.add(j)
                todo.append(j)
    assert seen == ids


def test_no_batched_tuned_variant_recorded_by_default():
    dm.dualmv_tune_clear()
    assert dm.dualmv_tuned_variant_batched(dm.DUALMV_DTYPE_F32, 2048, 2048, 2048, 256) == -1
    assert dm.dualmv_tuned_variant_batched(dm.DUALMV_DTYPE_F64, 64, 64, 64, 1) == -1


@pytest.mark.parametrize("tag", ["f32", "f64", "i32"])
def test_batched_tune_rejects_bad_arguments(tag):
    fn = getattr(dm, f"dualmv_tune_{tag}_strided_batched")
    res = dm.TuneResult()
    good = (64, 64, FAKE, 64, 4096, FAKE, 64, FAKE, 64, FAKE, 64, FAKE, 64, 3)

    def call(args, cfg=_cfg(), r=res):
        return fn(*args, cfg, r, None)
    assert call(good, cfg=_cfg(repeats=4, trim=2)) == dm.DUALMV_ERR_INVALID_VALUE
    assert call(good, cfg=None) == dm.DUALMV_ERR_INVALID_VALUE
    assert call(good, r=None) == dm.DUALMV_ERR_INVALID_VALUE
    bad_lda = good[:3] + (63,) + good[4:]
    assert call(bad_lda) == dm.DUALMV_ERR_INVALID_VALUE
    bad_stride_q = good[:10] + (63,) + good[11:]          # q rows overlap
    assert call(bad_stride_q) == dm.DUALMV_ERR_INVALID_VALUE
    neg_batch = good[:13] + (-1,)
    assert call(neg_batch) == dm.DUALMV_ERR_INVALID_VALUE
    null_a = good[:2] + (None,) + good[3:]
    assert call(null_a) == dm.DUALMV_ERR_INVALID_VALUE


# ---- single-sided passes --------------------------------------------------

def _sided_ids(tab):
    return {i for i, v in enumerate(tab) if v.single_sided}


@pytest.mark.parametrize("dtype", DTYPES)
def test_single_sided_instances(dtype):
    """fp32: every shape has single-sided instances (the passes of GESUMMV,
    GEMVER and ATAX's fallback); fp64: the packed self-loading 256-column
    shapes, entry 0 among them; int32 (no single-sided calls): none.  The
    tuner's walk over those entries reaches each of them from entry 0."""
    tab = table(dtype)
    ids = _sided_ids(tab)
    for v in tab:
        assert v.single_sided in (0, 1) and v.pad_ == 0
    if dtype == dm.DUALMV_DTYPE_I32:
        assert ids == set()
        return
    assert 0 in ids
    if dtype == dm.DUALMV_DTYPE_F32:
        assert ids == set(range(len(tab)))
    else:
        for i in ids:
            v = tab[i]
            assert v.kernel == dm.DUALMV_KERNEL_F64E and v.packed == 1 and \
                v.producer_warp == 0 and v.band_cols == 256, i
        assert len(ids) >= 4
    seen, todo = {0}, [0]
    while todo:
        i = todo.pop()
        for j in ids:
            if j not in seen and _neighbours(tab[i], tab[j]):
                seen.add(j)
                todo.append(j)
    assert seen == ids


def test_no_pass_tuned_variant_recorded_by_default():
    dm.dualmv_tune_clear()
    for pass_ in (dm.DUALMV_PASS_ROWS, dm.DUALMV_PASS_COLS):
        assert dm.dualmv_tuned_variant_pass(dm.DUALMV_DTYPE_F32, 4096, 4096, 4096, pass_) == -1
    assert dm.dualmv_tuned_variant_pass(dm.DUALMV_DTYPE_F32, 4096, 4096, 4096, 3) == -1


@pytest.mark.parametrize("tag", ["f32", "f64"])
def test_pass_tune_rejects_bad_arguments(tag):
    fn = getattr(dm, f"dualmv_tune_pass_{tag}")
    res = dm.TuneResult()
    rows, cols = dm.DUALMV_PASS_ROWS, dm.DUALMV_PASS_COLS
    assert fn(64, 64, FAKE, 64, 0, FAKE, FAKE, _cfg(), res, None) == dm.DUALMV_ERR_INVALID_VALUE
    assert fn(64, 64, FAKE, 64, 3, FAKE, FAKE, _cfg(), res, None) == dm.DUALMV_ERR_INVALID_VALUE
    for p in (rows, cols):
        assert fn(64, 64, FAKE, 64, p, FAKE, FAKE, None, res, None) == \
            dm.DUALMV_ERR_INVALID_VALUE
        assert fn(64, 64, FAKE, 64, p, FAKE, FAKE, _cfg(repeats=4, trim=2), res, None) == \
            dm.DUALMV_ERR_INVALID_VALUE
        assert fn(64, 64, FAKE, 64, p, FAKE, FAKE, _cfg(), None, None) == \
            dm.DUALMV_ERR_INVALID_VALUE
        assert fn(64, 64, FAKE, 63, p, FAKE, FAKE, _cfg(), res, None) == \
            dm.DUALMV_ERR_INVALID_VALUE
        assert fn(64, 64, None, 64, p, FAKE, FAKE, _cfg(), res, None) == \
            dm.DUALMV_ERR_INVALID_VALUE
        assert fn(64, 64, FAKE, 64, p, None, FAKE, _cfg(), res, None) == \
            dm.DUALMV_ERR_INVALID_VALUE
        assert fn(64, 64, FAKE, 64, p, FAKE, None, _cfg(), res, None) == \
            dm.DUALMV_ERR_INVALID_VALUE
        assert fn(-1, 64, FAKE, 64, p, FAKE, FAKE, _cfg(), res, None) == \
            dm.DUALMV_ERR_INVALID_VALUE


def test_tune_pass_api_rejects_bad_arguments():
    """api.tune_pass checks its tensors before any library call."""
    torch = pytest.importorskip("torch")
    A = torch.zeros(4, 6, dtype=torch.float32)
    with pytest.raises(ValueError):
        dm.tune_pass(A, torch.zeros(6), "diagonal")
    with pytest.raises(ValueError):
        dm.tune_pass(A.to(torch.int32), torch.zeros(6, dtype=torch.int32), "rows")
    with pytest.raises(ValueError):
        dm.tune_pass(A[None], torch.zeros(6), "rows")
    with pytest.raises(ValueError):            # rows: x has N = 6 elements
        dm.tune_pass(A, torch.zeros(4), "rows")
    with pytest.raises(ValueError):            # cols: x has M = 4 elements
        dm.tune_pass(A, torch.zeros(6), "cols")
    with pytest.raises(ValueError):            # out of the wrong length
        dm.tune_pass(A, torch.zeros(6), "rows", out=torch.zeros(6))
    with pytest.raises(ValueError):            # x of another dtype
        dm.tune_pass(A, torch.zeros(6, dtype=torch.float64), "rows")
