"""GB300-native fused dual matrix-vector product (BICG: q = A p, s = A^T r).

The computation is the BICG kernel that the paper tunes (Table 1 and
Table 2).  It runs in hand-written CUDA for sm_103a behind the C ABI of
``include/dualmv.h``; this package holds the in-tree build script, the
ctypes binding (``_binding``), a tensor-level wrapper (``api.dualmv``) and
the seeded workload generator (``inputs``).

The CUDA library is loaded on first use of any binding name (for example
``paper_2512_22147_gb300.dualmv``); if ``libdualmv.so`` has not been built
that first use raises ImportError.  There is no CPU fallback.
"""
import importlib

_BINDING_NAMES = {
    "DUALMV_ERR_ALLOC", "DUALMV_ERR_INVALID_VALUE", "DUALMV_ERR_LAUNCH",
    "DUALMV_ERR_TIMEOUT", "DUALMV_ERR_UNSUPPORTED", "DUALMV_ERR_TOO_LARGE", "DUALMV_PATH_AUTO",
    "DUALMV_PATH_DIRECT", "DUALMV_PATH_TMA", "DUALMV_PATH_TMA_NATIVE_F64", "DUALMV_SUCCESS", "EXPORTED",
    "LIBRARY_PATH", "DualmvError", "Plan", "dualmv_device_fault", "dualmv_f32",
    "dualmv_f32_strided_batched", "dualmv_f64", "dualmv_f64_strided_batched",
    "dualmv_i32", "dualmv_i32_strided_batched", "dualmv_last_cuda_error",
    "dualmv_plan", "dualmv_record_kernel_events", "dualmv_set_path",
    "dualmv_status_string", "library", "dualmv_f32_noalloc",
    "dualmv_f32_noalloc_scratch_bytes", "dualmv_gesummv_f32", "dualmv_gesummv_f64",
    "dualmv_atax_f32", "dualmv_atax_f64", "dualmv_gemver_f32", "dualmv_gemver_f64",
    "DUALMV_DTYPE_F32", "DUALMV_DTYPE_F64", "DUALMV_DTYPE_I32", "DUALMV_KERNEL_STREAM",
    "DUALMV_KERNEL_F64E", "DUALMV_KERNEL_WIDE", "Variant", "TuneConfig", "TuneResult", "dualmv_variant_count",
    "dualmv_variant_info", "dualmv_set_variant", "dualmv_tuned_variant", "dualmv_tune_clear",
    "dualmv_trimmed_mean", "dualmv_tune_f32", "dualmv_tune_f64", "dualmv_tune_i32",
    "dualmv_last_variant", "TuneStep", "dualmv_atax_set_two_pass",
    "dualmv_gemver_set_onthefly", "dualmv_last_kernel", "DUALMV_KERNEL_PHASED",
    "DUALMV_KERNEL_PLAIN", "dualmv_atax_last_path", "DUALMV_ATAX_ONE_READ",
    "DUALMV_ATAX_TWO_PASS", "dualmv_read_probe", "dualmv_pool_usage",
    "dualmv_selftest_wait_timeout", "DUALMV_KERNEL_CLUSTER",
    "dualmv_gemver_last_path", "DUALMV_GEMVER_FACTORED", "DUALMV_GEMVER_ONTHEFLY",
    "DUALMV_GEMVER_UPDATE_SPLIT", "dualmv_tune_f32_strided_batched",
    "dualmv_tune_f64_strided_batched", "dualmv_tune_i32_strided_batched",
    "dualmv_tuned_variant_batched", "dualmv_tune_pass_f32", "dualmv_tune_pass_f64",
    "dualmv_tuned_variant_pass", "DUALMV_PASS_ROWS", "DUALMV_PASS_COLS",
}
_API_NAMES = {"dualmv", "device_fault", "gesummv", "atax", "gemver", "tune", "tune_pass",
              "variants"}


def __getattr__(name):
    if name in _BINDING_NAMES:
        return getattr(importlib.import_module("._binding", __name__), name)
    if name in _API_NAMES:
        return getattr(importlib.import_module(".api", __name__), name)
    raise AttributeError(f"module {__name__!r} has no attribute {name!r}")


def __dir__():
    return sorted(set(globals()) | _BINDING_NAMES | _API_NAMES)
