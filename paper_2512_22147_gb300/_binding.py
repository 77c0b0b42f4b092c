"""ctypes binding of the C ABI in ``include/dualmv.h``.

Argument marshalling only: every step of the computation runs in the CUDA
library.  There is no fallback: if ``libdualmv.so`` has not been built, the
import fails with an error that says how to build it.

Two layers:
  * the raw entry points under their C names (``dualmv_f32``,
    ``dualmv_f32_strided_batched``, ...), taking integers and raw pointers
    exactly like the C functions;
  * ``dualmv(A, p, r)``, which takes CUDA torch tensors, derives the sizes,
    leading dimension and strides from them, picks the entry point by dtype
    and runs on the current torch stream.
"""
from __future__ import annotations

import ctypes
import os

from . import build as _build

DUALMV_SUCCESS = 0
DUALMV_ERR_INVALID_VALUE = 1
DUALMV_ERR_ALLOC = 2
DUALMV_ERR_LAUNCH = 3
DUALMV_ERR_TIMEOUT = 4
DUALMV_ERR_UNSUPPORTED = 5
DUALMV_ERR_TOO_LARGE = 6

DUALMV_PATH_AUTO = 0
DUALMV_PATH_TMA = 1
DUALMV_PATH_DIRECT = 2
DUALMV_PATH_TMA_NATIVE_F64 = 3

DUALMV_DTYPE_F32 = 0
DUALMV_DTYPE_F64 = 1
DUALMV_DTYPE_I32 = 2
DUALMV_KERNEL_STREAM = 0
DUALMV_KERNEL_F64E = 1
DUALMV_KERNEL_WIDE = 2
DUALMV_KERNEL_PHASED = 3
DUALMV_KERNEL_PLAIN = 4
DUALMV_KERNEL_CLUSTER = 5
DUALMV_ATAX_TWO_PASS = 0
DUALMV_ATAX_ONE_READ = 1
DUALMV_GEMVER_FACTORED = 0
DUALMV_GEMVER_ONTHEFLY = 1
DUALMV_GEMVER_UPDATE_SPLIT = 2
DUALMV_PASS_ROWS = 1
DUALMV_PASS_COLS = 2

EXPORTED = (
    "dualmv_f32", "dualmv_f64", "dualmv_i32",
    "dualmv_f32_strided_batched", "dualmv_f64_strided_batched",
    "dualmv_i32_strided_batched",
    "dualmv_status_string", "dualmv_last_cuda_error", "dualmv_device_fault",
    "dualmv_set_path", "dualmv_plan", "dualmv_record_kernel_events",
    "dualmv_f32_noalloc", "dualmv_f32_noalloc_scratch_bytes",
    "dualmv_gesummv_f32", "dualmv_gesummv_f64", "dualmv_atax_f32", "dualmv_atax_f64",
    "dualmv_gemver_f32", "dualmv_gemver_f64",
    "dualmv_variant_count", "dualmv_variant_info", "dualmv_set_variant",
    "dualmv_tuned_variant", "dualmv_tune_clear", "dualmv_trimmed_mean",
    "dualmv_tune_f32", "dualmv_tune_f64", "dualmv_tune_i32", "dualmv_last_variant",
    "dualmv_tune_f32_strided_batched", "dualmv_tune_f64_strided_batched",
    "dualmv_tune_i32_strided_batched", "dualmv_tuned_variant_batched",
    "dualmv_atax_set_two_pass", "dualmv_gemver_set_onthefly", "dualmv_last_kernel",
    "dualmv_atax_last_path", "dualmv_read_probe", "dualmv_pool_usage",
    "dualmv_gemver_last_path", "dualmv_selftest_wait_timeout", "dualmv_tune_pass_f32",
    "dualmv_tune_pass_f64", "dualmv_tuned_variant_pass",
)


class DualmvError(RuntimeError):
    """A dualmv entry point returned a status other than success."""

    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} (status {status}, "
                         f"cuda error {_lib.dualmv_last_cuda_error()})")


class Plan(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "band_cols", "tile_rows", "bands", "stripes", "tiles", "grid",
        "max_segments", "workspace_bytes", "smem_bytes", "threads")]


class Variant(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "index", "kernel", "warps", "rows_per_warp", "stages", "band_cols", "tile_rows",
        "threads", "native_cols", "producer_warp", "packed", "batched", "single_sided",
        "pad_")] + [("smem_bytes", ctypes.c_int64)]


class TuneConfig(ctypes.Structure):
    _fields_ = [("repeats", ctypes.c_int32), ("trim", ctypes.c_int32),
                ("max_rounds", ctypes.c_int32), ("candidates", ctypes.c_int32),
                ("min_gain", ctypes.c_double), ("flush_l2", ctypes.c_int32)]


TUNE_MAX_TRACE = 64


class TuneStep(ctypes.Structure):
    _fields_ = [("index", ctypes.c_int32), ("round", ctypes.c_int32),
                ("feasible", ctypes.c_int32), ("pad_", ctypes.c_int32),
                ("ms", ctypes.c_double), ("fe", ctypes.c_double)]


class TuneResult(ctypes.Structure):
    _fields_ = [("best", ctypes.c_int32), ("rounds", ctypes.c_int32),
                ("evaluated", ctypes.c_int32), ("rejected", ctypes.c_int32),
                ("baseline_ms", ctypes.c_double), ("best_ms", ctypes.c_double),
                ("worst_fe", ctypes.c_double), ("trace_len", ctypes.c_int32),
                ("initial", ctypes.c_int32), ("trace", TuneStep * TUNE_MAX_TRACE)]


def _load() -> ctypes.CDLL:
    path = _build.LIB_PATH
    if not os.path.exists(path):
        raise ImportError(
            f"{path} is missing: build it with `python -m "
            "paper_2512_22147_gb300.build` (nvcc for sm_103a); there is no "
            "CPU fallback")
    lib = ctypes.CDLL(path)
    i64, vp, st = ctypes.c_int64, ctypes.c_void_p, ctypes.c_int
    single = [i64, i64, vp, i64, vp, vp, vp, vp, vp]
    batched = [i64, i64, vp, i64, i64, vp, i64, vp, i64, vp, i64, vp, i64, i64, vp]
    for t in ("f32", "f64", "i32"):
        f = getattr(lib, f"dualmv_{t}")
        f.argtypes, f.restype = single, st
        f = getattr(lib, f"dualmv_{t}_strided_batched")
        f.argtypes, f.restype = batched, st
    lib.dualmv_f32_noalloc.argtypes, lib.dualmv_f32_noalloc.restype = single, st
    lib.dualmv_f32_noalloc_scratch_bytes.argtypes = []
    lib.dualmv_f32_noalloc_scratch_bytes.restype = i64
    for tag, real in (("f32", ctypes.c_float), ("f64", ctypes.c_double)):
        f = getattr(lib, f"dualmv_gesummv_{tag}")
        f.argtypes = [i64, i64, real, vp, i64, real, vp, i64, vp, vp, vp]
        f.restype = st
        f = getattr(lib, f"dualmv_atax_{tag}")
        f.argtypes = [i64, i64, vp, i64, vp, vp, vp]
        f.restype = st
        f = getattr(lib, f"dualmv_gemver_{tag}")
        f.argtypes = [i64, i64, real, real, vp, i64, st, vp, vp, vp, vp, vp, vp, vp, vp, vp]
        f.restype = st
    lib.dualmv_status_string.argtypes = [st]
    lib.dualmv_status_string.restype = ctypes.c_char_p
    lib.dualmv_last_cuda_error.argtypes = []
    lib.dualmv_last_cuda_error.restype = st
    lib.dualmv_device_fault.argtypes = [vp]
    lib.dualmv_device_fault.restype = st
    lib.dualmv_set_path.argtypes = [st]
    lib.dualmv_set_path.restype = st
    lib.dualmv_atax_set_two_pass.argtypes = [st]
    lib.dualmv_atax_set_two_pass.restype = st
    lib.dualmv_gemver_set_onthefly.argtypes = [st]
    lib.dualmv_gemver_set_onthefly.restype = st
    lib.dualmv_record_kernel_events.argtypes = [vp, vp]
    lib.dualmv_record_kernel_events.restype = None
    lib.dualmv_plan.argtypes = [i64, i64, i64, i64, i64, i64, ctypes.POINTER(Plan)]
    lib.dualmv_plan.restype = st
    i32 = ctypes.c_int32
    lib.dualmv_variant_count.argtypes, lib.dualmv_variant_count.restype = [i32], i32
    lib.dualmv_variant_info.argtypes = [i32, i32, ctypes.POINTER(Variant)]
    lib.dualmv_variant_info.restype = st
    lib.dualmv_set_variant.argtypes, lib.dualmv_set_variant.restype = [i32, i32], i32
    lib.dualmv_tuned_variant.argtypes, lib.dualmv_tuned_variant.restype = [i32, i64, i64, i64], i32
    lib.dualmv_tune_clear.argtypes, lib.dualmv_tune_clear.restype = [], None
    lib.dualmv_last_variant.argtypes, lib.dualmv_last_variant.restype = [], i32
    lib.dualmv_last_kernel.argtypes, lib.dualmv_last_kernel.restype = [], i32
    lib.dualmv_atax_last_path.argtypes, lib.dualmv_atax_last_path.restype = [], i32
    lib.dualmv_gemver_last_path.argtypes, lib.dualmv_gemver_last_path.restype = [], i32
    lib.dualmv_read_probe.argtypes = [vp, i64, vp, vp]
    lib.dualmv_read_probe.restype = st
    lib.dualmv_selftest_wait_timeout.argtypes = [ctypes.c_int, vp, vp]
    lib.dualmv_selftest_wait_timeout.restype = st
    lib.dualmv_pool_usage.argtypes = [ctypes.c_int, ctypes.POINTER(i64), ctypes.POINTER(i64),
                                      ctypes.c_int]
    lib.dualmv_pool_usage.restype = st
    lib.dualmv_trimmed_mean.argtypes = [ctypes.POINTER(ctypes.c_double), i64, i64,
                                        ctypes.POINTER(ctypes.c_double)]
    lib.dualmv_trimmed_mean.restype = st
    for t in ("f32", "f64", "i32"):
        f = getattr(lib, f"dualmv_tune_{t}")
        f.argtypes = single[:-1] + [ctypes.POINTER(TuneConfig), ctypes.POINTER(TuneResult), vp]
        f.restype = st
        f = getattr(lib, f"dualmv_tune_{t}_strided_batched")
        f.argtypes = batched[:-1] + [ctypes.POINTER(TuneConfig), ctypes.POINTER(TuneResult), vp]
        f.restype = st
    lib.dualmv_tuned_variant_batched.argtypes = [i32, i64, i64, i64, i64]
    lib.dualmv_tuned_variant_batched.restype = i32
    for t in ("f32", "f64"):
        f = getattr(lib, f"dualmv_tune_pass_{t}")
        f.argtypes = [i64, i64, vp, i64, i32, vp, vp, ctypes.POINTER(TuneConfig),
                      ctypes.POINTER(TuneResult), vp]
        f.restype = st
    lib.dualmv_tuned_variant_pass.argtypes = [i32, i64, i64, i64, i32]
    lib.dualmv_tuned_variant_pass.restype = i32
    return lib


_lib = _load()
LIBRARY_PATH = _build.LIB_PATH


def library() -> ctypes.CDLL:
    return _lib


# --------------------------------------------------- raw C entry points ----

def dualmv_f32(M, N, A, lda, p, r, q, s, stream):
    return _lib.dualmv_f32(M, N, A, lda, p, r, q, s, stream)


def dualmv_f64(M, N, A, lda, p, r, q, s, stream):
    return _lib.dualmv_f64(M, N, A, lda, p, r, q, s, stream)


def dualmv_i32(M, N, A, lda, p, r, q, s, stream):
    return _lib.dualmv_i32(M, N, A, lda, p, r, q, s, stream)


def dualmv_f32_noalloc(M, N, A, lda, p, r, q, s, stream):
    """dualmv_f32 without any device allocation: scratch is a fixed array
    inside the library (see include/dualmv.h for who needs this and why)."""
    return _lib.dualmv_f32_noalloc(M, N, A, lda, p, r, q, s, stream)


def dualmv_f32_noalloc_scratch_bytes() -> int:
    return _lib.dualmv_f32_noalloc_scratch_bytes()


def dualmv_f32_strided_batched(M, N, A, lda, sA, p, sP, r, sR, q, sQ, s, sS, batch, stream):
    return _lib.dualmv_f32_strided_batched(M, N, A, lda, sA, p, sP, r, sR, q, sQ, s, sS,
                                           batch, stream)


def dualmv_f64_strided_batched(M, N, A, lda, sA, p, sP, r, sR, q, sQ, s, sS, batch, stream):
    return _lib.dualmv_f64_strided_batched(M, N, A, lda, sA, p, sP, r, sR, q, sQ, s, sS,
                                           batch, stream)


def dualmv_i32_strided_batched(M, N, A, lda, sA, p, sP, r, sR, q, sQ, s, sS, batch, stream):
    return _lib.dualmv_i32_strided_batched(M, N, A, lda, sA, p, sP, r, sR, q, sQ, s, sS,
                                           batch, stream)


def dualmv_gesummv_f32(M, N, alpha, A, lda, beta, B, ldb, x, y, stream):
    return _lib.dualmv_gesummv_f32(M, N, alpha, A, lda, beta, B, ldb, x, y, stream)


def dualmv_gesummv_f64(M, N, alpha, A, lda, beta, B, ldb, x, y, stream):
    return _lib.dualmv_gesummv_f64(M, N, alpha, A, lda, beta, B, ldb, x, y, stream)


def dualmv_atax_f32(M, N, A, lda, x, y, stream):
    return _lib.dualmv_atax_f32(M, N, A, lda, x, y, stream)


def dualmv_atax_f64(M, N, A, lda, x, y, stream):
    return _lib.dualmv_atax_f64(M, N, A, lda, x, y, stream)


def dualmv_gemver_f32(M, N, alpha, beta, A, lda, update_A, u1, v1, u2, v2, w, x, y, z, stream):
    return _lib.dualmv_gemver_f32(M, N, alpha, beta, A, lda, update_A, u1, v1, u2, v2, w, x, y,
                                  z, stream)


def dualmv_gemver_f64(M, N, alpha, beta, A, lda, update_A, u1, v1, u2, v2, w, x, y, z, stream):
    return _lib.dualmv_gemver_f64(M, N, alpha, beta, A, lda, update_A, u1, v1, u2, v2, w, x, y,
                                  z, stream)


def dualmv_status_string(status: int) -> str:
    return _lib.dualmv_status_string(status).decode()


status_string = dualmv_status_string


def dualmv_last_cuda_error() -> int:
    return _lib.dualmv_last_cuda_error()


def dualmv_device_fault(stream=None) -> int:
    return _lib.dualmv_device_fault(stream)


def dualmv_atax_set_two_pass(two_pass: int) -> int:
    """1: ATAX always reads A twice; 0: single-read cluster path where it fits."""
    return _lib.dualmv_atax_set_two_pass(two_pass)


def dualmv_gemver_set_onthefly(onthefly: int) -> int:
    """1: GEMVER forms A_hat element by element even without update_A."""
    return _lib.dualmv_gemver_set_onthefly(onthefly)


def dualmv_set_path(path: int) -> int:
    old = _lib.dualmv_set_path(path)
    if old < 0:
        raise ValueError(f"unknown path {path}")
    return old


def dualmv_record_kernel_events(start, stop) -> None:
    """Raw cudaEvent_t handles (ints) or None; see include/dualmv.h."""
    _lib.dualmv_record_kernel_events(start, stop)


def dualmv_plan(M, N, batch, elem_bytes, acc_bytes, num_sms) -> Plan:
    out = Plan()
    rc = _lib.dualmv_plan(M, N, batch, elem_bytes, acc_bytes, num_sms, ctypes.byref(out))
    if rc != DUALMV_SUCCESS:
        raise DualmvError(rc, "dualmv_plan")
    return out


# ---------------------------------------------------- variants and tuner ----

def dualmv_variant_count(dtype: int) -> int:
    return _lib.dualmv_variant_count(dtype)


def dualmv_variant_info(dtype: int, index: int) -> Variant:
    out = Variant()
    rc = _lib.dualmv_variant_info(dtype, index, ctypes.byref(out))
    if rc != DUALMV_SUCCESS:
        raise DualmvError(rc, "dualmv_variant_info")
    return out


def dualmv_set_variant(dtype: int, index: int) -> int:
    old = _lib.dualmv_set_variant(dtype, index)
    if old == -2:
        raise ValueError(f"unknown dtype {dtype} or variant {index}")
    return old


def dualmv_tuned_variant(dtype: int, M: int, N: int, lda: int) -> int:
    return _lib.dualmv_tuned_variant(dtype, M, N, lda)


def dualmv_tuned_variant_batched(dtype: int, M: int, N: int, lda: int, batch: int) -> int:
    return _lib.dualmv_tuned_variant_batched(dtype, M, N, lda, batch)


def dualmv_tune_clear() -> None:
    _lib.dualmv_tune_clear()


def dualmv_last_variant() -> int:
    return _lib.dualmv_last_variant()


def dualmv_last_kernel() -> int:
    """DUALMV_KERNEL_* of this thread's last dual product, or -1."""
    return _lib.dualmv_last_kernel()


def dualmv_read_probe(buf, nbytes: int, out, stream) -> int:
    """Benchmark instrumentation: one 16-byte-load pass over ``nbytes`` of
    device memory at ``buf`` (xor-folded into the device word ``out``)."""
    return _lib.dualmv_read_probe(buf, nbytes, out, stream)


def dualmv_selftest_wait_timeout(cluster_scope: int, waited, stream) -> int:
    """Failure-detection test instrumentation: one warp waits, through the
    library's bounded mbarrier waits, on a phase nothing completes; the wait
    runs out after about 2 s, sets the device fault word and writes 0 to the
    device int32 ``waited``."""
    return _lib.dualmv_selftest_wait_timeout(cluster_scope, waited, stream)


def dualmv_pool_usage(device: int, reset_high: bool = False):
    """(bytes held, high-water mark of bytes in use) of the library's
    workspace pool on ``device``; ``reset_high`` resets the mark after
    reading it."""
    reserved, high = ctypes.c_int64(0), ctypes.c_int64(0)
    rc = _lib.dualmv_pool_usage(device, ctypes.byref(reserved), ctypes.byref(high),
                                1 if reset_high else 0)
    if rc != DUALMV_SUCCESS:
        raise DualmvError(rc, "dualmv_pool_usage")
    return reserved.value, high.value


def dualmv_atax_last_path() -> int:
    """DUALMV_ATAX_ONE_READ or DUALMV_ATAX_TWO_PASS for this thread's last
    ATAX call, or -1."""
    return _lib.dualmv_atax_last_path()


def dualmv_gemver_last_path() -> int:
    """DUALMV_GEMVER_FACTORED, DUALMV_GEMVER_ONTHEFLY or
    DUALMV_GEMVER_UPDATE_SPLIT for this thread's last GEMVER call, or -1."""
    return _lib.dualmv_gemver_last_path()


def dualmv_trimmed_mean(times, k: int) -> float:
    arr = (ctypes.c_double * len(times))(*times)
    out = ctypes.c_double()
    rc = _lib.dualmv_trimmed_mean(arr, len(times), k, ctypes.byref(out))
    if rc != DUALMV_SUCCESS:
        raise DualmvError(rc, "dualmv_trimmed_mean")
    return out.value


def _tune(tag, M, N, A, lda, p, r, q, s, cfg, res, stream):
    return getattr(_lib, f"dualmv_tune_{tag}")(M, N, A, lda, p, r, q, s,
                                               ctypes.byref(cfg) if cfg is not None else None,
                                               ctypes.byref(res) if res is not None else None,
                                               stream)


def dualmv_tune_f32(M, N, A, lda, p, r, q, s, cfg, res, stream):
    return _tune("f32", M, N, A, lda, p, r, q, s, cfg, res, stream)


def dualmv_tune_f64(M, N, A, lda, p, r, q, s, cfg, res, stream):
    return _tune("f64", M, N, A, lda, p, r, q, s, cfg, res, stream)


def dualmv_tune_i32(M, N, A, lda, p, r, q, s, cfg, res, stream):
    return _tune("i32", M, N, A, lda, p, r, q, s, cfg, res, stream)


def _tune_batched(tag, M, N, A, lda, sA, p, sP, r, sR, q, sQ, s, sS, batch, cfg, res, stream):
    return getattr(_lib, f"dualmv_tune_{tag}_strided_batched")(
        M, N, A, lda, sA, p, sP, r, sR, q, sQ, s, sS, batch,
        ctypes.byref(cfg) if cfg is not None else None,
        ctypes.byref(res) if res is not None else None, stream)


def _tune_pass(tag, M, N, A, lda, pass_, x, out, cfg, res, stream):
    return getattr(_lib, f"dualmv_tune_pass_{tag}")(
        M, N, A, lda, pass_, x, out, ctypes.byref(cfg) if cfg is not None else None,
        ctypes.byref(res) if res is not None else None, stream)


def dualmv_tune_pass_f32(M, N, A, lda, pass_, x, out, cfg, res, stream):
    """Tune one single-sided pass: DUALMV_PASS_ROWS (out = A x) or
    DUALMV_PASS_COLS (out = A^T x)."""
    return _tune_pass("f32", M, N, A, lda, pass_, x, out, cfg, res, stream)


def dualmv_tune_pass_f64(M, N, A, lda, pass_, x, out, cfg, res, stream):
    return _tune_pass("f64", M, N, A, lda, pass_, x, out, cfg, res, stream)


def dualmv_tuned_variant_pass(dtype: int, M: int, N: int, lda: int, pass_: int) -> int:
    return _lib.dualmv_tuned_variant_pass(dtype, M, N, lda, pass_)


def dualmv_tune_f32_strided_batched(*args):
    return _tune_batched("f32", *args)


def dualmv_tune_f64_strided_batched(*args):
    return _tune_batched("f64", *args)


def dualmv_tune_i32_strided_batched(*args):
    return _tune_batched("i32", *args)
