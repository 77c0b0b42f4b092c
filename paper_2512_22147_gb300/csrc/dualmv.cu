// Host side of the dualmv library: argument checks, the work planner, TMA
// descriptors, the stream-ordered workspace and the C ABI declared in
// include/dualmv.h.  The operation is the BICG kernel of the paper (Table 1
// and Table 2): q = A p and s = A^T r from a single pass over A.
#include "dualmv.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <tuple>
#include <type_traits>
#include <vector>

#include "dualmv_kernels.cuh"
#include "dualmv_f64e.cuh"
#include "dualmv_tune.cuh"
#include "dualmv_wide.cuh"
#include "dualmv_atax.cuh"
#include "dualmv_atax_f64.cuh"
#include "dualmv_ops.cuh"
#include "dualmv_probe.cuh"
#include "dualmv_small.cuh"
#include "dualmv_gemver_update.cuh"

namespace {

using dmv::kBandCols;
using dmv::Params;

// Tile shape per element width: W consumer warps x RPW rows per warp, and
// the ring depth.  Every tile of the generic kernel is 32 KiB of A.  Four
// stages: with the consumers releasing each stage as soon as they have
// read it, 3, 4, 5 and 6 stages gave 1.022, 1.025, 1.017 and 0.998 of the
// measured copy bandwidth on the f32 16384^2 workload (two stages 0.96).
constexpr int kWarps = 8;
constexpr int kRpw4 = 4;   // 4-byte elements: 32 rows x 1 KiB
constexpr int kRpw8 = 2;   // 8-byte elements: 16 rows x 2 KiB
constexpr int kStages = 4;
constexpr int kDirectCtasPerSm = 4;
// fp64 on the FP32 pipes (dualmv_f64e.cuh).
#ifndef DUALMV_F64E_WARPS
#define DUALMV_F64E_WARPS 12
#endif
#ifndef DUALMV_F64E_RPW
#define DUALMV_F64E_RPW 4
#endif
#ifndef DUALMV_F64E_STAGES
#define DUALMV_F64E_STAGES 2
#endif
#ifndef DUALMV_F64E_BAND
#define DUALMV_F64E_BAND 256
#endif
constexpr int kF64eWarps = DUALMV_F64E_WARPS;
constexpr int kF64eRpw = DUALMV_F64E_RPW;
constexpr int kF64eStages = DUALMV_F64E_STAGES;
constexpr int kF64eBand = DUALMV_F64E_BAND;
// No producer warp: each consumer warp loads its own boxes.  The kernel is
// latency-bound (dependent chains of error-free FP32 transformations), so it
// turns warps into throughput: 12 warps (three per SM sub-partition, 163
// registers each) with two 8 KiB stages apiece, as many as shared memory
// holds.  A producer warp would take a warp slot and registers from them.
constexpr bool kF64eSelf = true;
// The double-float arithmetic of each lane's column pairs runs as packed
// FP32x2 instructions, with no native fp64 columns: the kernel is bound by
// instruction issue, and the pairs halve the FP32 instructions.
constexpr bool kF64ePack = true;
constexpr int kF64eNativeCols = 0;

// Which stream kernel a call uses.
enum class Kind { kTma, kDirect, kF64e };

thread_local int g_last_cuda_error = 0;
thread_local cudaEvent_t g_kernel_ev_start = nullptr;
thread_local cudaEvent_t g_kernel_ev_stop = nullptr;
thread_local int32_t g_last_variant = -1;
thread_local int32_t g_last_kernel = -1;
thread_local int32_t g_last_atax_path = -1;
int g_path = DUALMV_PATH_AUTO;
int g_atax_two_pass = 0;  // 1: ATAX always takes the two-pass path
int g_gemver_onthefly = 0;  // 1: GEMVER applies the update element by element
thread_local int32_t g_last_gemver_path = -1;

dualmv_status cuda_fail(cudaError_t e) {
    g_last_cuda_error = static_cast<int>(e);
    return DUALMV_ERR_LAUNCH;
}

// ------------------------------------------------------- per-device state --

constexpr int kMaxDevices = 64;

struct DeviceState {
    std::once_flag once;
    cudaError_t init_error = cudaSuccess;
    int sms = 0;
    cudaMemPool_t pool = nullptr;
};
DeviceState g_dev[kMaxDevices];

cudaError_t device_state(int dev, DeviceState **out) {
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    DeviceState &st = g_dev[dev];
    std::call_once(st.once, [&]() {
        cudaError_t e = cudaDeviceGetAttribute(&st.sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) { st.init_error = e; return; }
        cudaMemPoolProps props;
        std::memset(&props, 0, sizeof props);
        props.allocType = cudaMemAllocationTypePinned;
        props.handleTypes = cudaMemHandleTypeNone;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = dev;
        e = cudaMemPoolCreate(&st.pool, &props);
        if (e != cudaSuccess) { st.init_error = e; return; }
        // Keep freed workspace cached in the pool between calls.
        uint64_t keep = UINT64_MAX;
        e = cudaMemPoolSetAttribute(st.pool, cudaMemPoolAttrReleaseThreshold, &keep);
        if (e != cudaSuccess) { st.init_error = e; return; }
    });
    *out = &st;
    return st.init_error;
}

// ------------------------------------------------------------ TMA encode --

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t,
                                   void *, const cuuint64_t *, const cuuint64_t *,
                                   const cuuint32_t *, const cuuint32_t *,
                                   CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = []() -> EncodeTiledFn {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return nullptr;
        return reinterpret_cast<EncodeTiledFn>(p);
    }();
    return fn;
}

template <typename T> CUtensorMapDataType tma_dtype();
template <> CUtensorMapDataType tma_dtype<float>() { return CU_TENSOR_MAP_DATA_TYPE_FLOAT32; }
template <> CUtensorMapDataType tma_dtype<double>() { return CU_TENSOR_MAP_DATA_TYPE_FLOAT64; }
template <> CUtensorMapDataType tma_dtype<int32_t>() { return CU_TENSOR_MAP_DATA_TYPE_INT32; }

// L2 promotion for the TMA loads of A: the largest of 256, 128 and 64 bytes
// that divides the base address and every row (and problem) stride, else
// none.  Each box row starts a whole number of bands (1 or 2 KiB) into its
// matrix row, so with this choice no promoted chunk reaches into a
// neighbouring band; a larger promotion on misaligned rows would make both
// bands fetch the shared chunk, and the second fetch comes long after the
// first has left L2.
CUtensorMapL2promotion l2_promotion(uintptr_t base, int64_t row_bytes, int64_t batch_bytes,
                                    bool three_d) {
    const int64_t sizes[3] = {256, 128, 64};
    const CUtensorMapL2promotion kinds[3] = {CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                             CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                                             CU_TENSOR_MAP_L2_PROMOTION_L2_64B};
    for (int i = 0; i < 3; ++i) {
        const int64_t s = sizes[i];
        if (base % (uintptr_t)s == 0 && row_bytes % s == 0 && (!three_d || batch_bytes % s == 0))
            return kinds[i];
    }
    return CU_TENSOR_MAP_L2_PROMOTION_NONE;
}

// Encodes A as a 2-D (N, M) or 3-D (N, M, batch) tiled tensor with a box of
// kBandCols x tile_rows (x 1).  Columns >= N and rows >= M read as zero.
// The last tensor map this thread encoded, reused when a call repeats the
// matrix (same address, shape, strides, box and element type).
struct MapMemo {
    bool valid = false;
    int64_t key[10];
    CUtensorMap map;
};
thread_local MapMemo g_map_memo;

template <typename T>
bool encode_a_uncached(CUtensorMap *map, const T *A, int64_t M, int64_t N, int64_t lda,
                       int64_t strideA, int64_t batch, int box_cols, int tile_rows,
                       bool three_d);

template <typename T>
bool encode_a(CUtensorMap *map, const T *A, int64_t M, int64_t N, int64_t lda,
              int64_t strideA, int64_t batch, int box_cols, int tile_rows, bool three_d) {
    const int64_t key[10] = {(int64_t)reinterpret_cast<uintptr_t>(A), M, N, lda,
                             three_d ? strideA : 0, three_d ? batch : 1, box_cols, tile_rows,
                             three_d ? 1 : 0, (int64_t)tma_dtype<T>()};
    if (g_map_memo.valid && std::memcmp(key, g_map_memo.key, sizeof key) == 0) {
        *map = g_map_memo.map;
        return true;
    }
    if (!encode_a_uncached<T>(map, A, M, N, lda, strideA, batch, box_cols, tile_rows, three_d))
        return false;
    std::memcpy(g_map_memo.key, key, sizeof key);
    g_map_memo.map = *map;
    g_map_memo.valid = true;
    return true;
}

template <typename T>
bool encode_a_uncached(CUtensorMap *map, const T *A, int64_t M, int64_t N, int64_t lda,
                       int64_t strideA, int64_t batch, int box_cols, int tile_rows,
                       bool three_d) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const int64_t es = sizeof(T);
    const CUtensorMapL2promotion promo =
        l2_promotion(reinterpret_cast<uintptr_t>(A), lda * es, strideA * es, three_d);
    cuuint64_t dims[3] = {(cuuint64_t)N, (cuuint64_t)M, (cuuint64_t)batch};
    cuuint64_t strides[2] = {(cuuint64_t)(lda * es), (cuuint64_t)(strideA * es)};
    cuuint32_t box[3] = {(cuuint32_t)box_cols, (cuuint32_t)tile_rows, 1u};
    cuuint32_t estr[3] = {1u, 1u, 1u};
    CUresult rc = fn(map, tma_dtype<T>(), three_d ? 3u : 2u, const_cast<T *>(A), dims,
                     strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_NONE, promo,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return rc == CUDA_SUCCESS;
}

// Phased tensor maps for one problem whose row stride or base TMA cannot
// take: NPH = 16 / gcd(lda * size, 16) phases (rows ph, ph + NPH, ...), each
// a 2-D tensor of N + ph_off columns from its first row's start rounded down
// to 16 bytes (ph_off elements before it), with row stride NPH * lda * size.
// A band's box starts at the band's column (16-byte aligned in the tensor)
// and so holds the row's columns shifted by ph_off; the small box after it
// holds the ph_off columns pushed past it.  Columns past N + ph_off are out
// of the tensor: no copy reads past a row's last element.  Returns the phase
// count, or 0 when the shape does not fit this path.
// L2 fills of the phased maps: a box row starts only 16-byte aligned, so a
// 256-byte promotion fetches a segment shared with the next band, often
// evicted before that band reads it.  f32 16384 x 16383: 81.3% of HBM with
// 256-byte fills, 82.8% with none, 83.6% with 64-byte fills.
#ifndef DUALMV_PHASED_PROMO
#define DUALMV_PHASED_PROMO CU_TENSOR_MAP_L2_PROMOTION_L2_64B
#endif
template <typename T>
int encode_phased(dmv::TmapSet *maps, Params *prm, const T *A, int64_t M, int64_t N,
                  int64_t lda, int tile_rows) {
    constexpr int64_t es = sizeof(T);
    const int64_t row_bytes = lda * es;
    const int nph = row_bytes % 16 == 0 ? 1 : row_bytes % 8 == 0 ? 2 : 4;
    if (reinterpret_cast<uintptr_t>(A) % es != 0 || (int64_t)nph * row_bytes % 16 != 0 ||
        M < nph || N < 1 || M >= INT32_MAX || N >= INT32_MAX - 16 || tile_rows % nph != 0)
        return 0;
    EncodeTiledFn fn = encode_fn();
    if (!fn) return 0;
    for (int ph = 0; ph < nph; ++ph) {
        const uintptr_t addr = reinterpret_cast<uintptr_t>(A + ph * lda);
        const uintptr_t base = addr & ~(uintptr_t)15;
        const int64_t off = (int64_t)(addr - base) / es;
        const int64_t rows = (M - ph + nph - 1) / nph;
        cuuint64_t dims[2] = {(cuuint64_t)(N + off), (cuuint64_t)rows};
        cuuint64_t strides[1] = {(cuuint64_t)(nph * row_bytes)};
        cuuint32_t estr[2] = {1u, 1u};
        for (int k = 0; k < 2; ++k) {
            cuuint32_t box[2] = {(cuuint32_t)(k == 0 ? kBandCols : 16 / es),
                                 (cuuint32_t)(tile_rows / nph)};
            CUresult rc = fn(&maps->m[2 * ph + k], tma_dtype<T>(), 2u,
                             reinterpret_cast<void *>(base), dims, strides, box, estr,
                             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                             DUALMV_PHASED_PROMO, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
            if (rc != CUDA_SUCCESS) return 0;
        }
        prm->ph_off[ph] = (int32_t)off;
    }
    prm->ph_n = nph;
    return nph;
}

// ------------------------------------------------------------------ plan --

// Warps, rows per warp and shared memory of each stream kernel.
struct Geometry {
    int64_t band_cols;  // columns per band (tile width)
    int64_t tile_rows;  // rows per tile (stripe height)
    int64_t box_cols;   // columns per TMA box
    int64_t box_rows;   // rows per TMA box
    int64_t smem;
    int64_t threads;
};

template <typename T>
constexpr int default_rpw() { return sizeof(T) == 4 ? kRpw4 : kRpw8; }

template <typename T, int W, int RPW, int S>
Geometry stream_geometry(bool tma) {
    Geometry g;
    g.band_cols = kBandCols;
    g.tile_rows = W * RPW;
    g.box_cols = kBandCols;
    g.box_rows = g.tile_rows;
    g.smem = tma ? dmv::SmemLayout<T, W, RPW, S, true>::kTotal
                 : dmv::SmemLayout<T, W, RPW, S, false>::kTotal;
    g.threads = (W + (tma ? 1 : 0)) * 32;
    return g;
}

template <int W, int RPW, int S, bool kSelf = kF64eSelf, int BAND = kF64eBand>
Geometry f64e_geometry() {
    Geometry g;
    g.band_cols = BAND;
    g.tile_rows = W * RPW;
    g.box_cols = BAND;
    g.box_rows = RPW;  // one box per consumer warp
    g.smem = dmv::F64eLayout<W, RPW, S, BAND>::kTotal;
    g.threads = (W + (kSelf ? 0 : 1)) * 32;
    return g;
}

// Wide int32 tiles: RPW rows by W * 256 columns, one 256-column box per
// consumer warp.
template <int W, int RPW, int S>
Geometry wide_geometry() {
    Geometry g;
    g.band_cols = (int64_t)W * kBandCols;
    g.tile_rows = RPW;
    g.box_cols = kBandCols;
    g.box_rows = RPW;
    g.smem = dmv::WideLayout<W, RPW, S>::kTotal;
    g.threads = (W + 1) * 32;
    return g;
}

template <typename T>
Geometry generic_geometry(bool tma) {
    return stream_geometry<T, kWarps, default_rpw<T>(), kStages>(tma);
}

Geometry geometry(int64_t elem_bytes, int64_t acc_bytes, Kind kind) {
    if (kind == Kind::kF64e) return f64e_geometry<kF64eWarps, kF64eRpw, kF64eStages>();
    const bool tma = kind == Kind::kTma;
    if (elem_bytes == 8) return generic_geometry<double>(tma);
    return acc_bytes == 8 ? generic_geometry<int32_t>(tma) : generic_geometry<float>(tma);
}

// The last plan this thread made, reused when a call repeats the shape (the
// segment count below loops over every CTA, a few microseconds per call).
struct PlanMemo {
    bool valid = false;
    int64_t key[9];
    dualmv_plan_t plan;
};
thread_local PlanMemo g_plan_memo;

dualmv_status make_plan_geo(int64_t M, int64_t N, int64_t batch, int64_t elem_bytes,
                            int64_t acc_bytes, int64_t ctas, const Geometry &geo,
                            dualmv_plan_t *pl) {
    if (M <= 0 || N <= 0 || batch <= 0 || ctas <= 0 || pl == nullptr)
        return DUALMV_ERR_INVALID_VALUE;
    if ((elem_bytes != 4 && elem_bytes != 8) || (acc_bytes != 4 && acc_bytes != 8) ||
        acc_bytes < elem_bytes)
        return DUALMV_ERR_INVALID_VALUE;
    const int64_t key[9] = {M, N, batch, elem_bytes, acc_bytes, ctas, geo.band_cols,
                            geo.tile_rows, geo.smem * 4096 + geo.threads};
    if (g_plan_memo.valid && std::memcmp(key, g_plan_memo.key, sizeof key) == 0) {
        *pl = g_plan_memo.plan;
        return DUALMV_SUCCESS;
    }
    const int64_t bm = geo.tile_rows;
    dualmv_plan_t p;
    std::memset(&p, 0, sizeof p);
    p.band_cols = geo.band_cols;
    p.tile_rows = bm;
    p.bands = (N + p.band_cols - 1) / p.band_cols;
    p.stripes = (M + bm - 1) / bm;
    if (p.bands > INT64_MAX / p.stripes / batch) return DUALMV_ERR_INVALID_VALUE;
    p.tiles = batch * p.bands * p.stripes;
    p.grid = p.tiles < ctas ? p.tiles : ctas;
    // Most segments (bands touched) of any CTA.
    int64_t most = 0;
    for (int64_t c = 0; c < p.grid; ++c) {
        const int64_t t0 = dmv::cta_first_tile(c, p.tiles, p.grid);
        const int64_t t1 = dmv::cta_first_tile(c + 1, p.tiles, p.grid);
        const int64_t nseg = (t1 - 1) / p.stripes - t0 / p.stripes + 1;
        if (nseg > most) most = nseg;
    }
    p.max_segments = most;
    const int64_t q_ws = p.bands > 1 ? batch * p.bands * M * acc_bytes : 0;
    const int64_t s_ws = p.grid * p.max_segments * p.band_cols * acc_bytes;
    // int32 inputs (4-byte elements, 8-byte sums) accumulate atomically into
    // q and s and take no workspace.
    const bool atomic_out = elem_bytes == 4 && acc_bytes == 8;
    p.workspace_bytes = atomic_out ? 0 : ((q_ws + 255) / 256) * 256 + s_ws;
    p.smem_bytes = geo.smem;
    p.threads = geo.threads;
    *pl = p;
    std::memcpy(g_plan_memo.key, key, sizeof key);
    g_plan_memo.plan = p;
    g_plan_memo.valid = true;
    return DUALMV_SUCCESS;
}

dualmv_status make_plan(int64_t M, int64_t N, int64_t batch, int64_t elem_bytes,
                        int64_t acc_bytes, int64_t ctas, Kind kind, dualmv_plan_t *pl) {
    if (kind == Kind::kF64e && elem_bytes != 8) return DUALMV_ERR_INVALID_VALUE;
    if ((elem_bytes != 4 && elem_bytes != 8) || (acc_bytes != 4 && acc_bytes != 8))
        return DUALMV_ERR_INVALID_VALUE;
    return make_plan_geo(M, N, batch, elem_bytes, acc_bytes, ctas,
                         geometry(elem_bytes, acc_bytes, kind), pl);
}

// ------------------------------------------------------------ validation --

dualmv_status validate(int64_t M, int64_t N, const void *A, int64_t lda, int64_t strideA,
                       const void *p, int64_t strideP, const void *r, int64_t strideR,
                       const void *q, int64_t strideQ, const void *s, int64_t strideS,
                       int64_t batch, uint32_t outputs = dmv::kOutBoth) {
    const bool want_q = (outputs & dmv::kOutQ) != 0, want_s = (outputs & dmv::kOutS) != 0;
    if (M < 0 || N < 0 || batch < 0) return DUALMV_ERR_INVALID_VALUE;
    if (lda < (N > 1 ? N : 1)) return DUALMV_ERR_INVALID_VALUE;
    if (strideA < 0 || strideP < 0 || strideR < 0 || strideQ < 0 || strideS < 0)
        return DUALMV_ERR_INVALID_VALUE;
    if (batch == 0) return DUALMV_SUCCESS;
    if (M > 0 && N > 0 &&
        (A == nullptr || (want_q && p == nullptr) || (want_s && r == nullptr)))
        return DUALMV_ERR_INVALID_VALUE;
    if (want_q && M > 0 && q == nullptr) return DUALMV_ERR_INVALID_VALUE;
    if (want_s && N > 0 && s == nullptr) return DUALMV_ERR_INVALID_VALUE;
    if (batch > 1 && ((want_q && strideQ < M) || (want_s && strideS < N)))
        return DUALMV_ERR_INVALID_VALUE;
    // Index arithmetic stays in int64: the last element of A must be addressable.
    if (M > 0 && N > 0) {
        const int64_t lim = INT64_MAX / 4;
        if (M > lim / lda) return DUALMV_ERR_INVALID_VALUE;
        if (batch > 1 && strideA > 0 && batch - 1 > (lim - M * lda) / strideA)
            return DUALMV_ERR_INVALID_VALUE;
    }
    return DUALMV_SUCCESS;
}

bool fault_injected(const char *what) {
    const char *v = std::getenv("DUALMV_FAULT_INJECT");
    return v != nullptr && std::strcmp(v, what) == 0;
}

bool fault_injected_alloc() { return fault_injected("alloc"); }

// ------------------------------------------------------------- launching --

// Raises kernel K's dynamic shared-memory limit to `bytes` the first time K
// is launched on device `dev` (the attribute is per device and per kernel).
template <auto K>
cudaError_t smem_opt_in(int64_t bytes, int dev) {
    static std::atomic<uint64_t> done{0};
    const uint64_t bit = 1ull << (dev & 63);
    if (done.load(std::memory_order_acquire) & bit) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(K, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)bytes);
    if (e == cudaSuccess) done.fetch_or(bit, std::memory_order_acq_rel);
    return e;
}

// Launches `kern` as a programmatic dependent of the kernel enqueued just
// before it on `stream`: it may start early and waits (griddepcontrol.wait)
// before using that kernel's results.
template <typename Kern, typename... Args>
cudaError_t launch_dependent(Kern kern, dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                             Args... args) {
    cudaLaunchConfig_t cfg;
    std::memset(&cfg, 0, sizeof cfg);
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

template <typename T, bool kTma, bool k3d, int kOut = dmv::kOutBoth, bool kRank2 = false,
          int W = kWarps, int RPW = default_rpw<T>(), int S = kStages, bool kRev = false>
cudaError_t launch_stream(const CUtensorMap &map, const Params &prm, const dualmv_plan_t &pl,
                          int dev, cudaStream_t stream) {
    constexpr auto kern =
        dmv::dualmv_stream_kernel<T, W, RPW, S, kTma, k3d, kOut, kRank2, kRev>;
    cudaError_t e = smem_opt_in<kern>(pl.smem_bytes, dev);
    if (e != cudaSuccess) return e;
    // After the zeroing kernel, or a late-wait pass (Params::pdl_late).
    if (std::is_same<T, int32_t>::value || prm.pdl_late)
        return launch_dependent(kern, dim3((unsigned)pl.grid), dim3((unsigned)pl.threads),
                                (size_t)pl.smem_bytes, stream, map, prm);
    kern<<<(unsigned)pl.grid, (unsigned)pl.threads, (size_t)pl.smem_bytes, stream>>>(map, prm);
    return cudaGetLastError();
}

template <int NPH>
Geometry f64e_phased_geometry_n() {
    // The phased fp64 kernel: self-loading warps on 256-column bands.
    Geometry g = f64e_geometry<kF64eWarps, kF64eRpw, kF64eStages, true, kBandCols>();
    g.smem = dmv::F64eLayout<kF64eWarps, kF64eRpw, kF64eStages, kBandCols, NPH>::kTotal;
    return g;
}

template <int NPH>
cudaError_t launch_f64e_phased_n(const dmv::TmapSet &maps, const Params &prm,
                                 const dualmv_plan_t &pl, int dev, cudaStream_t stream) {
    constexpr auto kern =
        dmv::dualmv_stream_f64e_phased_kernel<kF64eWarps, kF64eRpw, kF64eStages, NPH>;
    cudaError_t e = smem_opt_in<kern>(pl.smem_bytes, dev);
    if (e != cudaSuccess) return e;
    return launch_dependent(kern, dim3((unsigned)pl.grid), dim3((unsigned)pl.threads),
                            (size_t)pl.smem_bytes, stream, maps, prm);
}

// The 4-byte phased kernel's tile: W consumer warps x 4 rows, ring depth.
// Its realignment makes it latency bound where the aligned kernel is not.
// Measured (% of HBM, whole call; f32 16384 x 16383 / int32 4001 x 100003,
// both at lda = N):
//   warps x stages   8 x 6   10 x 5   12 x 4   15 x 3
//   f32              83.5    90.6     88.5     87.2
//   int32            66.7    72.8     85.7     94.4
// f32 wants ring depth, int32 (64-bit sums) warps.  16 x 3 leaves f32 at
// 96 registers and does not fit int32's 8-byte scratch.
#ifndef DUALMV_PHASED_WARPS_F32
#define DUALMV_PHASED_WARPS_F32 10
#endif
#ifndef DUALMV_PHASED_STAGES_F32
#define DUALMV_PHASED_STAGES_F32 5
#endif
#ifndef DUALMV_PHASED_WARPS_I32
#define DUALMV_PHASED_WARPS_I32 15
#endif
#ifndef DUALMV_PHASED_STAGES_I32
#define DUALMV_PHASED_STAGES_I32 3
#endif
template <typename T>
constexpr int phased_warps() {
    return std::is_same<T, int32_t>::value ? DUALMV_PHASED_WARPS_I32 : DUALMV_PHASED_WARPS_F32;
}
template <typename T>
constexpr int phased_stages() {
    return std::is_same<T, int32_t>::value ? DUALMV_PHASED_STAGES_I32 : DUALMV_PHASED_STAGES_F32;
}

// Dynamic shared memory a CTA may opt into on sm_100-class parts.
constexpr int kMaxDynSmem = 227 * 1024;
template <typename T>
constexpr bool phased_layouts_fit() {
    constexpr int W = phased_warps<T>(), R = default_rpw<T>(), S = phased_stages<T>();
    return dmv::SmemLayout<T, W, R, S, true, 1>::kTotal <= kMaxDynSmem &&
           dmv::SmemLayout<T, W, R, S, true, 2>::kTotal <= kMaxDynSmem &&
           dmv::SmemLayout<T, W, R, S, true, 4>::kTotal <= kMaxDynSmem;
}
static_assert(phased_layouts_fit<float>() && phased_layouts_fit<int32_t>(),
              "a phased tile shape exceeds the shared memory of a CTA");
static_assert(dmv::F64eLayout<kF64eWarps, kF64eRpw, kF64eStages, kBandCols, 1>::kTotal <=
                      kMaxDynSmem &&
                  dmv::F64eLayout<kF64eWarps, kF64eRpw, kF64eStages, kBandCols, 2>::kTotal <=
                      kMaxDynSmem,
              "a phased fp64 layout exceeds the shared memory of a CTA");

template <typename T, int NPH>
Geometry phased_geometry_n() {
    constexpr int W = phased_warps<T>(), S = phased_stages<T>();
    Geometry g = stream_geometry<T, W, default_rpw<T>(), S>(true);
    g.smem = dmv::SmemLayout<T, W, default_rpw<T>(), S, true, NPH>::kTotal;
    return g;
}
template <typename T>
Geometry phased_geometry(int nph) {
    if constexpr (sizeof(T) == 8)  // the double-float kernel's layout
        return nph == 1 ? f64e_phased_geometry_n<1>() : f64e_phased_geometry_n<2>();
    return nph == 1 ? phased_geometry_n<T, 1>()
                    : nph == 2 ? phased_geometry_n<T, 2>() : phased_geometry_n<T, 4>();
}

template <typename T, int NPH>
cudaError_t launch_phased_n(const dmv::TmapSet &maps, const Params &prm, const dualmv_plan_t &pl,
                            int dev, cudaStream_t stream) {
    constexpr auto kern =
        dmv::dualmv_stream_phased_kernel<T, phased_warps<T>(), default_rpw<T>(), phased_stages<T>(),
                                         NPH>;
    cudaError_t e = smem_opt_in<kern>(pl.smem_bytes, dev);
    if (e != cudaSuccess) return e;
    if constexpr (std::is_same<T, int32_t>::value)  // after the zeroing kernel
        return launch_dependent(kern, dim3((unsigned)pl.grid), dim3((unsigned)pl.threads),
                                (size_t)pl.smem_bytes, stream, maps, prm);
    kern<<<(unsigned)pl.grid, (unsigned)pl.threads, (size_t)pl.smem_bytes, stream>>>(maps, prm);
    return cudaGetLastError();
}
template <typename T>
cudaError_t launch_phased(int nph, const dmv::TmapSet &maps, const Params &prm,
                          const dualmv_plan_t &pl, int dev, cudaStream_t stream) {
    if constexpr (sizeof(T) == 4) {  // 4-byte elements: 4 rows a warp, up to 4 phases
        switch (nph) {
        case 1: return launch_phased_n<T, 1>(maps, prm, pl, dev, stream);
        case 2: return launch_phased_n<T, 2>(maps, prm, pl, dev, stream);
        case 4: return launch_phased_n<T, 4>(maps, prm, pl, dev, stream);
        }
    } else {  // fp64: the double-float kernel, up to 2 phases
        switch (nph) {
        case 1: return launch_f64e_phased_n<1>(maps, prm, pl, dev, stream);
        case 2: return launch_f64e_phased_n<2>(maps, prm, pl, dev, stream);
        }
    }
    return cudaErrorInvalidValue;
}

template <int W, int RPW, int S>
cudaError_t launch_wide(const CUtensorMap &map, const Params &prm, const dualmv_plan_t &pl,
                        int dev, cudaStream_t stream) {
    constexpr auto kern = dmv::dualmv_wide_i32_kernel<W, RPW, S>;
    cudaError_t e = smem_opt_in<kern>(pl.smem_bytes, dev);
    if (e != cudaSuccess) return e;
    return launch_dependent(kern, dim3((unsigned)pl.grid), dim3((unsigned)pl.threads),
                            (size_t)pl.smem_bytes, stream, map, prm);  // after the zeroing
}

// Chunks per q output in the combine kernel: the smallest power of two
// giving at most about 8 band partials per thread, at most 32.
int combine_chunks(int64_t bands) {
    int c = 1;
    while (c < 32 && (int64_t)c * 8 < bands) c *= 2;
    return c;
}

template <bool k3d, int kOut = dmv::kOutBoth, int W = kF64eWarps, int RPW = kF64eRpw,
          int S = kF64eStages, int NC = kF64eNativeCols, bool kSelf = kF64eSelf,
          bool kPack = kF64ePack, int BAND = kF64eBand, bool kRev = false>
cudaError_t launch_f64e(const CUtensorMap &map, const Params &prm, const dualmv_plan_t &pl,
                        int dev, cudaStream_t stream) {
    constexpr auto kern =
        dmv::dualmv_stream_f64e_kernel<W, RPW, S, BAND, k3d, kOut, NC, kSelf, kPack, kRev>;
    cudaError_t e = smem_opt_in<kern>(pl.smem_bytes, dev);
    if (e != cudaSuccess) return e;
    // A programmatic dependent of the kernel before it (on repeated calls, the
    // previous combine kernel): its launch and prologue overlap that kernel,
    // and it waits for that grid's completion before touching memory.  fp64
    // 65536 x 4096: 0.379 -> 0.373 ms per call.  The f32 kernel, launched the
    // same way, lost 1%, so it keeps an ordinary launch.
    return launch_dependent(kern, dim3((unsigned)pl.grid), dim3((unsigned)pl.threads),
                            (size_t)pl.smem_bytes, stream, map, prm);
}

template <typename Acc>
cudaError_t launch_combine(const Params &prm, cudaStream_t stream) {
    const int chunks = combine_chunks(prm.bands);
    const int64_t rows_per_block = 256 / chunks;
    const bool want_q = (prm.outputs & dmv::kOutQ) != 0;
    const bool want_s = (prm.outputs & dmv::kOutS) != 0;
    const int64_t q_blocks = (want_q && prm.bands > 1)
                                 ? (prm.batch * prm.M + rows_per_block - 1) / rows_per_block
                                 : 0;
    const int64_t s_blocks = (want_s && prm.grid > 1) ? prm.batch * prm.bands : 0;
    const int64_t blocks = q_blocks + s_blocks;
    if (blocks == 0) return cudaSuccess;
    if (blocks > INT32_MAX) return cudaErrorInvalidConfiguration;
    // After the streaming kernel, whose workspace it reads.
    return launch_dependent(dmv::dualmv_combine_kernel<Acc>, dim3((unsigned)blocks), dim3(256),
                            0, stream, prm, q_blocks, chunks);
}

template <typename Acc>
cudaError_t zero_fill(Acc *out, int64_t len, int64_t stride, int64_t batch,
                      cudaStream_t stream) {
    if (len <= 0 || batch <= 0) return cudaSuccess;
    const int64_t total = len * batch;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    dmv::dualmv_zero_kernel<Acc><<<(unsigned)blocks, 256, 0, stream>>>(out, len, stride, batch);
    return cudaGetLastError();
}

// -------------------------------------------------------------- variants --
//
// Compiled variants of the streaming kernel for one unbatched dual product
// on the TMA path: the search space of the tuner.  Entry 0 of each table is
// the kernel untuned calls use, so selecting it changes nothing.

using LaunchFn = cudaError_t (*)(const CUtensorMap &, const Params &, const dualmv_plan_t &,
                                 int, cudaStream_t);

struct Variant {
    dualmv_variant_t info;
    Kind kind;
    Geometry geo;
    LaunchFn launch;
    LaunchFn launch3d;  // strided batches (3-D tensor map), or nullptr
    // Single-sided passes (q only, s only: GESUMMV, GEMVER's forward passes,
    // ATAX's two-pass fallback), or nullptr.
    LaunchFn launch_q = nullptr, launch_s = nullptr;
    // A rows pass walking its tiles backwards (GEMVER's, after its columns
    // pass), or nullptr: only the fp64 passes' default shape has one.
    LaunchFn launch_q_rev = nullptr;
};

template <typename T, int W, int RPW, int S, bool k3d = false>
cudaError_t launch_stream_variant(const CUtensorMap &m, const Params &p,
                                  const dualmv_plan_t &pl, int dev, cudaStream_t st) {
    return launch_stream<T, true, k3d, dmv::kOutBoth, false, W, RPW, S>(m, p, pl, dev, st);
}

template <int W, int RPW, int S, int NC, bool kSelf, bool kPack, int BAND, bool k3d = false>
cudaError_t launch_f64e_variant(const CUtensorMap &m, const Params &p, const dualmv_plan_t &pl,
                                int dev, cudaStream_t st) {
    return launch_f64e<k3d, dmv::kOutBoth, W, RPW, S, NC, kSelf, kPack, BAND>(m, p, pl, dev,
                                                                             st);
}

// Single-sided instances (kOut = kOutQ or kOutS) of the same shapes.
template <typename T, int W, int RPW, int S, int kOut>
cudaError_t launch_stream_side(const CUtensorMap &m, const Params &p, const dualmv_plan_t &pl,
                               int dev, cudaStream_t st) {
    return launch_stream<T, true, false, kOut, false, W, RPW, S>(m, p, pl, dev, st);
}

template <int W, int RPW, int S, int NC, bool kSelf, bool kPack, int BAND, int kOut,
          bool kRev = false>
cudaError_t launch_f64e_side(const CUtensorMap &m, const Params &p, const dualmv_plan_t &pl,
                             int dev, cudaStream_t st) {
    return launch_f64e<false, kOut, W, RPW, S, NC, kSelf, kPack, BAND, kRev>(m, p, pl, dev, st);
}

Variant make_variant(int32_t index, int32_t kernel, int W, int RPW, int S, Kind kind,
                     const Geometry &g, LaunchFn fn, int NC = 0, bool self_load = false,
                     LaunchFn fn3d = nullptr, LaunchFn fn_q = nullptr,
                     LaunchFn fn_s = nullptr) {
    Variant v;
    v.info.index = index;
    v.info.kernel = kernel;
    v.info.warps = W;
    v.info.rows_per_warp = RPW;
    v.info.stages = S;
    v.info.native_cols = NC;
    v.info.producer_warp = self_load ? 0 : 1;
    v.info.packed = 0;
    v.info.batched = fn3d != nullptr ? 1 : 0;
    v.info.single_sided = (fn_q != nullptr && fn_s != nullptr) ? 1 : 0;
    v.info.pad_ = 0;
    v.info.band_cols = (int32_t)g.band_cols;
    v.info.tile_rows = (int32_t)g.tile_rows;
    v.info.threads = (int32_t)g.threads;
    v.info.smem_bytes = g.smem;
    v.kind = kind;
    v.geo = g;
    v.launch = fn;
    v.launch3d = fn3d;
    v.launch_q = fn_q;
    v.launch_s = fn_s;
    return v;
}

// kBatched: the variant also has a strided-batched instance (every shape of
// the 4-byte tables; not the native fp64 entry, which no batched entry
// neighbours).  fp32 shapes also have single-sided instances.
template <typename T, int W, int RPW, int S, bool kBatched = true>
Variant stream_variant(int32_t index) {
    LaunchFn fn3d = nullptr, fn_q = nullptr, fn_s = nullptr;
    if constexpr (kBatched) fn3d = &launch_stream_variant<T, W, RPW, S, true>;
    if constexpr (std::is_same<T, float>::value) {
        fn_q = &launch_stream_side<T, W, RPW, S, dmv::kOutQ>;
        fn_s = &launch_stream_side<T, W, RPW, S, dmv::kOutS>;
    }
    return make_variant(index, DUALMV_KERNEL_STREAM, W, RPW, S, Kind::kTma,
                        stream_geometry<T, W, RPW, S>(true),
                        &launch_stream_variant<T, W, RPW, S>, 0, false, fn3d, fn_q, fn_s);
}

// kBatched: the variant also has a strided-batched instance, and
// single-sided instances (the packed self-loading 256-column shapes);
// kRevQ: a backward rows pass too (the passes' default shape).
template <int W, int RPW, int S, int NC = kF64eNativeCols, bool kSelf = kF64eSelf,
          bool kPack = kF64ePack, int BAND = kF64eBand, bool kBatched = false,
          bool kRevQ = false>
Variant f64e_variant(int32_t index) {
    LaunchFn fn3d = nullptr, fn_q = nullptr, fn_s = nullptr;
    if constexpr (kBatched) {
        fn3d = &launch_f64e_variant<W, RPW, S, NC, kSelf, kPack, BAND, true>;
        fn_q = &launch_f64e_side<W, RPW, S, NC, kSelf, kPack, BAND, dmv::kOutQ>;
        fn_s = &launch_f64e_side<W, RPW, S, NC, kSelf, kPack, BAND, dmv::kOutS>;
    }
    Variant v = make_variant(index, DUALMV_KERNEL_F64E, W, RPW, S, Kind::kF64e,
                             f64e_geometry<W, RPW, S, kSelf, BAND>(),
                             &launch_f64e_variant<W, RPW, S, NC, kSelf, kPack, BAND>, NC, kSelf,
                             fn3d, fn_q, fn_s);
    v.info.packed = kPack ? 1 : 0;
    if constexpr (kRevQ)
        v.launch_q_rev = &launch_f64e_side<W, RPW, S, NC, kSelf, kPack, BAND, dmv::kOutQ, true>;
    return v;
}

template <int W, int RPW, int S>
Variant wide_variant(int32_t index) {
    return make_variant(index, DUALMV_KERNEL_WIDE, W, RPW, S, Kind::kTma,
                        wide_geometry<W, RPW, S>(), &launch_wide<W, RPW, S>);
}

// Tile shapes of the 4-byte types: entry 0 is the default (8 x 4 rows, 6
// stages); the others each differ from one of the earlier ones in one
// property, so the neighbourhood graph the tuner walks is connected.
template <typename T>
std::vector<Variant> stream4_entries() {
    return {
        stream_variant<T, 8, 4, 4>(0), stream_variant<T, 8, 4, 6>(1),
        stream_variant<T, 8, 4, 3>(2), stream_variant<T, 8, 2, 6>(3),
        stream_variant<T, 4, 4, 6>(4), stream_variant<T, 8, 8, 3>(5),
        stream_variant<T, 4, 8, 6>(6), stream_variant<T, 8, 2, 12>(7),
    };
}

const std::vector<Variant> &f32_table() {
    static const std::vector<Variant> tab = stream4_entries<float>();
    return tab;
}

// int32 adds the wide tiles (dualmv_wide.cuh); entry kI32Wide is the one
// untuned calls use when rows are not 128-byte aligned.  Its boxes are 8
// rows by 1 KiB: with 4-row (4 KiB) boxes the TMA unit, issuing eight boxes
// per 32 KiB tile, held the kernel near 91% of HBM however few bytes it
// moved.
constexpr int32_t kI32Wide = 8;
const std::vector<Variant> &i32_table() {
    static const std::vector<Variant> tab = [] {
        std::vector<Variant> v = stream4_entries<int32_t>();
        v.push_back(wide_variant<8, 8, 3>(kI32Wide));  // 8 KiB boxes
        v.push_back(wide_variant<8, 4, 6>(kI32Wide + 1));
        v.push_back(wide_variant<4, 8, 6>(kI32Wide + 2));
        return v;
    }();
    return tab;
}

// fp64: the double-float kernel in several shapes (entry 0: 12 self-loading
// warps x 4 rows, 2 stages, packed pairs), the scalar forms with and without
// native fp64 columns, the earlier layout with a producer warp and 7
// consumers, and native fp64 FMA.
const std::vector<Variant> &f64_table() {
    static const std::vector<Variant> tab = {
        f64e_variant<12, 4, 2, 0, true, true, kF64eBand, true>(0),
        f64e_variant<8, 4, 2, 0, true, true, kF64eBand, true, true>(1),  // fp64 passes' default
        f64e_variant<8, 4, 3, 0, true, false>(2),    // scalar FP32 instructions
        f64e_variant<8, 4, 3, 2, true, false>(3),
        f64e_variant<8, 4, 3, 3, true, false>(4),
        f64e_variant<7, 4, 3, 2, true, false>(5),
        f64e_variant<7, 4, 3, 2, false, false>(6),   // a producer warp feeds 7 consumers
        f64e_variant<7, 4, 3, 0, false, false>(7),
        stream_variant<double, 7, 4, 3, false>(8),   // native fp64 FMA
        f64e_variant<6, 4, 3, 2, false, false>(9),
        f64e_variant<7, 4, 2, 2, false, false>(10),
        // 128-column bands: 4 columns per lane (fewer registers, twice the
        // share of the row reduction per element).
        f64e_variant<8, 4, 3, 0, true, true, 128>(11),
        f64e_variant<12, 4, 3, 0, true, true, 128>(12),
        f64e_variant<12, 4, 2, 0, true, true, 128>(13),
        f64e_variant<8, 8, 3, 0, true, true, 128>(14),
        f64e_variant<8, 4, 3, 0, true, true, kF64eBand, true>(15),  // two warps per sub-partition
        // Fewer warps or rows than entry 0.
        f64e_variant<10, 4, 2, 0, true, true, kF64eBand, true>(16),
        f64e_variant<12, 2, 2, 0, true, true, kF64eBand, true>(17),
        // Four warps per sub-partition on 128-column bands (128 registers).
        f64e_variant<16, 4, 3, 0, true, true, 128>(18),
    };
    return tab;
}

const std::vector<Variant> *variant_table(int32_t dtype) {
    switch (dtype) {
    case DUALMV_DTYPE_F32: return &f32_table();
    case DUALMV_DTYPE_F64: return &f64_table();
    case DUALMV_DTYPE_I32: return &i32_table();
    }
    return nullptr;
}

template <typename T> constexpr int32_t dtype_code();
template <> constexpr int32_t dtype_code<float>() { return DUALMV_DTYPE_F32; }
template <> constexpr int32_t dtype_code<double>() { return DUALMV_DTYPE_F64; }
template <> constexpr int32_t dtype_code<int32_t>() { return DUALMV_DTYPE_I32; }

// Variants differ in one property: kernel, warps, rows per warp, stages,
// band width, or (double-float kernel) native columns, loading scheme or
// packing.
bool neighbours(const dualmv_variant_t &a, const dualmv_variant_t &b) {
    const int diff = (a.kernel != b.kernel) + (a.warps != b.warps) +
                     (a.rows_per_warp != b.rows_per_warp) + (a.stages != b.stages) +
                     (a.native_cols != b.native_cols) + (a.producer_warp != b.producer_warp) +
                     (a.packed != b.packed) +
                     // the wide kernel's band width follows from its kind
                     (a.kernel == b.kernel && a.band_cols != b.band_cols);
    return diff == 1;
}

std::atomic<int32_t> g_forced_variant[3] = {{-1}, {-1}, {-1}};
std::mutex g_tuned_mu;
// Tuned choices by (dtype, M, N, lda, batch, outputs); batch 1 for single
// problems, outputs kOutBoth for dual products, kOutQ / kOutS for
// single-sided passes.
std::map<std::tuple<int32_t, int64_t, int64_t, int64_t, int64_t, uint32_t>, int32_t> g_tuned;
std::atomic<int> g_tuned_count{0};

int32_t tuned_lookup(int32_t dtype, int64_t M, int64_t N, int64_t lda, int64_t batch = 1,
                     uint32_t outputs = dmv::kOutBoth) {
    if (g_tuned_count.load(std::memory_order_acquire) == 0) return -1;
    std::lock_guard<std::mutex> lk(g_tuned_mu);
    auto it = g_tuned.find(std::make_tuple(dtype, M, N, lda, batch, outputs));
    return it == g_tuned.end() ? -1 : it->second;
}

// The variant an untuned call of this shape uses: entry 0, except int32
// rows that are not 128-byte aligned, which take the wide tiles (their 1 KiB
// box rows would otherwise straddle a line shared with the next band).
int32_t default_variant(int32_t dtype, const void *A, int64_t lda_bytes) {
    if (dtype == DUALMV_DTYPE_I32 &&
        (reinterpret_cast<uintptr_t>(A) % 128 != 0 || lda_bytes % 128 != 0))
        return kI32Wide;
    return 0;
}

// The default of a single-sided pass: fp64 entry 1 (8 warps x 4 rows, 2
// stages), whose passes, with half the dual product's arithmetic, ran
// 6-8% faster than entry 0's 12 warps on 8192^2 (the pass tuner's choice
// for rows and columns); fp32 entry 0.
constexpr int32_t kF64SidedDefault = 1;
int32_t sided_default_variant(int32_t dtype) {
    return dtype == DUALMV_DTYPE_F64 ? kF64SidedDefault : 0;
}

// The variant a call runs: `index` if the caller (the tuner) names one, else
// the process-wide forced one, else the tuned one for this shape, else the
// default for the shape.  nullptr means entry 0, which the ordinary launch
// code covers.  A strided batch (batch > 1) runs a variant only if it has a
// batched instance, a single-sided pass (outputs kOutQ or kOutS) only if it
// has single-sided instances; otherwise entry 0.
const Variant *pick_variant(int32_t dtype, int64_t M, int64_t N, const void *A, int64_t lda,
                            int64_t es, int32_t index, int64_t batch = 1,
                            uint32_t outputs = dmv::kOutBoth) {
    const std::vector<Variant> *tab = variant_table(dtype);
    if (tab == nullptr) return nullptr;
    const bool sided = outputs != dmv::kOutBoth;
    if (index < 0) index = g_forced_variant[dtype].load(std::memory_order_relaxed);
    if (index < 0) index = tuned_lookup(dtype, M, N, lda, batch, outputs);
    if (index < 0)
        index = batch > 1 ? 0
                : sided   ? sided_default_variant(dtype)
                          : default_variant(dtype, A, lda * es);
    if (index <= 0 || index >= (int32_t)tab->size()) return nullptr;
    if (batch > 1 && (*tab)[index].launch3d == nullptr) return nullptr;
    if (sided && (*tab)[index].launch_q == nullptr) return nullptr;
    return &(*tab)[index];
}

// True when the call names a variant, or one is forced or tuned for this
// shape (even entry 0): such calls run the streaming kernels as chosen.
bool explicit_variant(int32_t dtype, int64_t M, int64_t N, int64_t lda, int32_t index) {
    if (index >= 0) return true;
    if (variant_table(dtype) == nullptr) return false;
    if (g_forced_variant[dtype].load(std::memory_order_relaxed) >= 0) return true;
    return tuned_lookup(dtype, M, N, lda) >= 0;
}

// ---- small fp32 problems: one thread-block cluster (dualmv_small.cuh) ----
// A call of at most kSmallMaxBytes of A, 256 <= N <= 2048, runs as one
// cluster of 16 CTAs with no workspace and no combine kernel: on the 1024^2
// workload the streaming kernel and its combine take 6.7 us hot in a graph,
// the cluster kernel 5.4 us.
constexpr int64_t kSmallMaxBytes = 8ll << 20;

struct SmallClusterCache {
    std::mutex mu;
    int ok[2][kMaxDevices] = {};  // 0 unknown, 1 placeable, -1 not
};
SmallClusterCache g_small_cache;

template <int VPL, int D>
cudaError_t launch_small_cluster(const Params &prm, int dev, cudaStream_t stream, bool *done) {
    *done = false;
    constexpr auto kern = dmv::dualmv_small_cluster_kernel<VPL, D>;
    constexpr int smem = dmv::SmallLayout<VPL>::kTotal;
    cudaLaunchConfig_t cfg;
    std::memset(&cfg, 0, sizeof cfg);
    cfg.gridDim = dim3(dmv::kSmallCluster);
    cfg.blockDim = dim3(dmv::kSmallWarps * 32);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = dmv::kSmallCluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;  // the occupancy query takes the cluster shape alone
    const int slot = VPL == 8 ? 0 : 1;
    {
        std::lock_guard<std::mutex> lk(g_small_cache.mu);
        if (g_small_cache.ok[slot][dev] == 0) {
            int clusters = 0;
            cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 smem);
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
            if (e == cudaSuccess) e = cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg);
            if (e != cudaSuccess) {  // no such cluster here: the streaming kernels
                (void)cudaGetLastError();
                clusters = 0;
            }
            g_small_cache.ok[slot][dev] = clusters > 0 ? 1 : -1;
        }
        if (g_small_cache.ok[slot][dev] < 0) return cudaSuccess;
    }
    *done = true;
    cfg.numAttrs = 2;  // and a programmatic dependent of the kernel before it
    return cudaLaunchKernelEx(&cfg, kern, prm);
}

// GEMVER's rank-2 update, applied on the fly by a single-sided pass.
// A pass whose combine a later kernel takes over: run() leaves its partial
// sums in the workspace, launches no combine kernel and does not free the
// workspace; the caller launches the kernel that adds them and then frees
// `ws` on the same stream.  used = false: the pass took no workspace (an
// empty problem, its outputs zero-filled).
struct Deferred {
    bool used = false;
    Params prm;
    void *ws = nullptr;
    int chunks = 1;
};

struct Rank2 {
    const void *u1, *v1, *u2, *v2;
    void *a_out;  // write A_hat here (may be A itself), or nullptr
    int64_t lda_out;
};

// One dual (or single-sided) matrix-vector product.  `outputs` selects q,
// s or both; single-sided calls (the building blocks of ATAX, GESUMMV and
// GEMVER) are single problems of float or double; `rank2` adds GEMVER's
// on-the-fly update to a single-sided call (native arithmetic for double).
template <typename T, typename Out>
dualmv_status run(int64_t M, int64_t N, const T *A, int64_t lda, int64_t strideA,
                  const T *p, int64_t strideP, const T *r, int64_t strideR, Out *q,
                  int64_t strideQ, Out *s, int64_t strideS, int64_t batch,
                  cudaStream_t stream, uint32_t outputs = dmv::kOutBoth,
                  const Rank2 *rank2 = nullptr, int32_t variant = -1,
                  Deferred *defer = nullptr, bool reverse = false, bool late_wait = false) {
    using Acc = typename dmv::Traits<T>::Acc;
    static_assert(sizeof(Acc) == sizeof(Out), "accumulator and output widths differ");
    constexpr bool kIntPath = std::is_same<T, int32_t>::value;
    if (outputs != dmv::kOutBoth && (kIntPath || batch > 1)) return DUALMV_ERR_UNSUPPORTED;
    if (rank2 != nullptr && outputs == dmv::kOutBoth) return DUALMV_ERR_UNSUPPORTED;
    const bool want_q = (outputs & dmv::kOutQ) != 0, want_s = (outputs & dmv::kOutS) != 0;
    g_last_variant = -1;
    g_last_kernel = -1;
    if (defer != nullptr) defer->used = false;
    dualmv_status st = validate(M, N, A, lda, strideA, p, strideP, r, strideR, q, strideQ,
                                s, strideS, batch, outputs);
    if (st != DUALMV_SUCCESS || batch == 0) return st;
    if (batch == 1) {  // strides are irrelevant for one problem
        strideA = M * lda; strideP = N; strideR = M; strideQ = M; strideS = N;
    }

    if (M == 0 || N == 0) {
        cudaError_t e = cudaSuccess;
        if (want_q) e = zero_fill(reinterpret_cast<Acc *>(q), M, strideQ, batch, stream);
        if (e == cudaSuccess && want_s)
            e = zero_fill(reinterpret_cast<Acc *>(s), N, strideS, batch, stream);
        return e == cudaSuccess ? DUALMV_SUCCESS : cuda_fail(e);
    }
    if (fault_injected_alloc()) return DUALMV_ERR_ALLOC;

    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e);
    DeviceState *ds = nullptr;
    e = device_state(dev, &ds);
    if (e != cudaSuccess) return cuda_fail(e);

    // Small fp32 dual products: one thread-block cluster, no workspace.
    if constexpr (std::is_same<T, float>::value) {
        if (batch == 1 && outputs == dmv::kOutBoth && rank2 == nullptr &&
            g_path == DUALMV_PATH_AUTO && N >= 256 && N <= 2048 && N % 4 == 0 &&
            lda % 4 == 0 && M * N * (int64_t)sizeof(T) <= kSmallMaxBytes &&
            (M + dmv::kSmallCluster - 1) / dmv::kSmallCluster <= dmv::kSmallMaxRows &&
            reinterpret_cast<uintptr_t>(A) % 16 == 0 && reinterpret_cast<uintptr_t>(p) % 16 == 0 &&
            !explicit_variant(DUALMV_DTYPE_F32, M, N, lda, variant)) {
            Params sp;
            std::memset(&sp, 0, sizeof sp);
            sp.A = A; sp.lda = lda; sp.p = p; sp.r = r; sp.q = q; sp.s = s;
            sp.M = M; sp.N = N; sp.batch = 1; sp.outputs = dmv::kOutBoth; sp.ph_n = 1;
            cudaEvent_t ev0 = g_kernel_ev_start, ev1 = g_kernel_ev_stop;
            bool done = false;
            e = ev0 ? cudaEventRecord(ev0, stream) : cudaSuccess;
            if (e == cudaSuccess)
                e = N <= 1024 ? launch_small_cluster<8, 3>(sp, dev, stream, &done)
                              : launch_small_cluster<16, 1>(sp, dev, stream, &done);
            if (e != cudaSuccess) return cuda_fail(e);
            if (done) {
                g_kernel_ev_start = g_kernel_ev_stop = nullptr;
                if (ev1) e = cudaEventRecord(ev1, stream);
                if (e != cudaSuccess) return cuda_fail(e);
                g_last_kernel = DUALMV_KERNEL_CLUSTER;
                return DUALMV_SUCCESS;
            }
        }
    }

    // Path choice: TMA needs a 16-byte aligned base, 16-byte multiple
    // strides and 32-bit coordinates.
    const int64_t es = sizeof(T);
    const bool three_d = batch > 1;
    bool tma = g_path != DUALMV_PATH_DIRECT &&
               (reinterpret_cast<uintptr_t>(A) % 16 == 0) && ((lda * es) % 16 == 0) &&
               M < INT32_MAX && N < INT32_MAX && batch < INT32_MAX &&
               (!three_d || (strideA > 0 && (strideA * es) % 16 == 0));
    // fp64 runs on the FP32 pipes unless native fp64 FMA is requested.
    Kind kind = Kind::kDirect;
    if (tma)
        kind = (es == 8 && g_path != DUALMV_PATH_TMA_NATIVE_F64 && rank2 == nullptr)
                   ? Kind::kF64e
                   : Kind::kTma;
    // A compiled variant other than the default (forced, tuned or named by
    // the tuner) for a dual product (one problem or a strided batch) or a
    // single-sided pass of one problem walking its tiles forwards, on the
    // TMA path.
    const Variant *var = nullptr;
    if (tma && rank2 == nullptr && g_path != DUALMV_PATH_TMA_NATIVE_F64 &&
        (outputs == dmv::kOutBoth || (!kIntPath && batch == 1))) {
        if (outputs == dmv::kOutQ && reverse) {
            // A rows pass walking backwards: the passes' default shape, if it
            // has a backward instance (fp64 entry 1); else the default kernel.
            const std::vector<Variant> &tab = *variant_table(dtype_code<T>());
            const int32_t d = sided_default_variant(dtype_code<T>());
            if (d > 0 && tab[d].launch_q_rev != nullptr) var = &tab[d];
        } else if (!reverse) {
            var = pick_variant(dtype_code<T>(), M, N, A, lda, es, variant, batch, outputs);
        }
    }
    if (var != nullptr) kind = var->kind;
    if (kind == Kind::kF64e) {
        // The double-float kernel counts tiles in 32 bits; a launch of 2^31
        // tiles or more (a huge batch of tiny problems) takes native fp64.
        const Geometry g = var ? var->geo : geometry(es, sizeof(Acc), kind);
        const int64_t per_problem = ((N + g.band_cols - 1) / g.band_cols) *
                                    ((M + g.tile_rows - 1) / g.tile_rows);
        if (per_problem > (INT32_MAX - 1) / batch) {
            kind = Kind::kTma;
            var = nullptr;
        }
    }
    CUtensorMap map;
    std::memset(&map, 0, sizeof map);
    if (tma) {
        const Geometry geo = var ? var->geo : geometry(es, sizeof(Acc), kind);
        tma = encode_a<T>(&map, A, M, N, lda, strideA, batch, (int)geo.box_cols,
                          (int)geo.box_rows, three_d);
        if (!tma) {
            kind = Kind::kDirect;
            var = nullptr;
        }
    }

    // Rows the TMA unit cannot take as one tensor (row stride or base not
    // 16-byte aligned): phased tensor maps, for one dual product (fp64 in the
    // double-float kernel).
    dmv::TmapSet pmaps;
    Params pinfo;
    std::memset(&pinfo, 0, sizeof pinfo);
    pinfo.ph_n = 1;
    int nph = 0;
    // The fp64 phased kernel streams 256-column bands of self-loading warps
    // whatever band width the aligned fp64 kernel is built with
    // (f64e_phased_geometry_n), so every fp64 band width may take it.
    if (kind == Kind::kDirect && g_path != DUALMV_PATH_DIRECT && !three_d &&
        rank2 == nullptr && outputs == dmv::kOutBoth &&
        (es == 4 || g_path != DUALMV_PATH_TMA_NATIVE_F64)) {
        std::memset(&pmaps, 0, sizeof pmaps);
        // Box rows: a tile's rows of one phase (4-byte kernel), or a warp's
        // (the self-loading fp64 kernel).
        const int box_rows = es == 8 ? kF64eRpw : phased_warps<T>() * default_rpw<T>();
        nph = encode_phased<T>(&pmaps, &pinfo, A, M, N, lda, box_rows);
    }

    dualmv_plan_t pl;
    st = var ? make_plan_geo(M, N, batch, es, sizeof(Acc), ds->sms, var->geo, &pl)
         : nph > 0
             ? make_plan_geo(M, N, batch, es, sizeof(Acc), ds->sms, phased_geometry<T>(nph), &pl)
             : make_plan(M, N, batch, es, sizeof(Acc),
                         (int64_t)ds->sms * (tma ? 1 : kDirectCtasPerSm), kind, &pl);
    if (st != DUALMV_SUCCESS) return st;

    // The int32 path accumulates into q and s atomically (exact, so still
    // deterministic) and needs no workspace.
    constexpr bool kAtomicOut = std::is_same<T, int32_t>::value;
    void *ws = nullptr;
    if (!kAtomicOut) {
        e = cudaMallocFromPoolAsync(&ws, (size_t)pl.workspace_bytes, ds->pool, stream);
        if (e != cudaSuccess) {
            g_last_cuda_error = static_cast<int>(e);
            return DUALMV_ERR_ALLOC;
        }
    }
    Params prm;
    std::memset(&prm, 0, sizeof prm);
    prm.ph_n = pinfo.ph_n;
    for (int ph = 0; ph < dmv::kMaxPhases; ++ph) prm.ph_off[ph] = pinfo.ph_off[ph];
    prm.A = A; prm.lda = lda; prm.strideA = strideA;
    prm.p = p; prm.strideP = strideP;
    prm.r = r; prm.strideR = strideR;
    prm.q = q; prm.strideQ = strideQ;
    prm.s = s; prm.strideS = strideS;
    prm.M = M; prm.N = N; prm.batch = batch;
    prm.outputs = outputs;
    prm.u1 = rank2 ? rank2->u1 : nullptr;
    prm.v1 = rank2 ? rank2->v1 : nullptr;
    prm.u2 = rank2 ? rank2->u2 : nullptr;
    prm.v2 = rank2 ? rank2->v2 : nullptr;
    prm.a_out = rank2 ? rank2->a_out : nullptr;
    prm.lda_out = rank2 ? rank2->lda_out : 0;
    prm.band_cols = pl.band_cols;
    prm.bands = pl.bands; prm.stripes = pl.stripes; prm.tiles = pl.tiles;
    prm.grid = pl.grid; prm.max_seg = pl.max_segments;
    // Late wait (Params::pdl_late) for the single-sided kernels below; the
    // caller's kernel before this call triggers its dependents after its wait.
    prm.pdl_late =
        (late_wait && !kIntPath && outputs != dmv::kOutBoth && rank2 == nullptr) ? 1 : 0;
    const int64_t q_ws_bytes = pl.bands > 1 ? batch * pl.bands * M * (int64_t)sizeof(Acc) : 0;
    prm.q_ws = (pl.bands > 1 && ws) ? ws : nullptr;
    prm.s_ws = ws ? static_cast<unsigned char *>(ws) + ((q_ws_bytes + 255) / 256) * 256 : nullptr;

    if (kAtomicOut) {
        const int64_t total = (M + N) * batch;
        int64_t blocks = (total + 255) / 256;
        if (blocks > (int64_t)ds->sms * 4) blocks = (int64_t)ds->sms * 4;
        dmv::dualmv_zero_outputs_kernel<Acc><<<(unsigned)blocks, 256, 0, stream>>>(
            reinterpret_cast<Acc *>(q), M, strideQ, reinterpret_cast<Acc *>(s), N, strideS,
            batch);
        e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_fail(e);
    }

    cudaEvent_t ev_start = g_kernel_ev_start, ev_stop = g_kernel_ev_stop;
    g_kernel_ev_start = g_kernel_ev_stop = nullptr;
    e = ev_start ? cudaEventRecord(ev_start, stream) : cudaSuccess;
    // The kind of streaming kernel this call launches (dualmv_last_kernel).
    const int32_t kernel_kind = var != nullptr         ? var->info.kernel
                                : nph > 0              ? (int32_t)DUALMV_KERNEL_PHASED
                                : kind == Kind::kF64e  ? (int32_t)DUALMV_KERNEL_F64E
                                : kind == Kind::kTma   ? (int32_t)DUALMV_KERNEL_STREAM
                                                       : (int32_t)DUALMV_KERNEL_PLAIN;
    if (e == cudaSuccess) {
        if (var != nullptr) {
            if (outputs == dmv::kOutQ)
                e = reverse ? var->launch_q_rev(map, prm, pl, dev, stream)
                            : var->launch_q(map, prm, pl, dev, stream);
            else if (outputs == dmv::kOutS)
                e = var->launch_s(map, prm, pl, dev, stream);
            else
                e = three_d ? var->launch3d(map, prm, pl, dev, stream)
                            : var->launch(map, prm, pl, dev, stream);
            if (e == cudaSuccess) g_last_variant = var->info.index;
        } else if (rank2 != nullptr) {
            if constexpr (!kIntPath) {
                const bool only_q = outputs == dmv::kOutQ;
                if (kind == Kind::kTma)
                    e = only_q ? launch_stream<T, true, false, dmv::kOutQ, true>(map, prm, pl, dev, stream)
                               : launch_stream<T, true, false, dmv::kOutS, true>(map, prm, pl, dev, stream);
                else
                    e = only_q ? launch_stream<T, false, false, dmv::kOutQ, true>(map, prm, pl, dev, stream)
                               : launch_stream<T, false, false, dmv::kOutS, true>(map, prm, pl, dev, stream);
            }
        } else if (outputs != dmv::kOutBoth) {
            if constexpr (!kIntPath) {
                // Single-sided products (one problem, float or double).
                const bool only_q = outputs == dmv::kOutQ;
                // reverse: a rows-only pass that follows a pass over the same
                // A walks each CTA's tiles backwards (see Deferred).
                const bool rev = reverse && only_q;
                if (kind == Kind::kF64e) {
                    // Entry 0's shape: untuned fp64 passes run entry 1 as a
                    // variant (above); this serves a forced or tuned entry 0.
                    if constexpr (std::is_same<T, double>::value)
                        e = rev ? launch_f64e<false, dmv::kOutQ, kF64eWarps, kF64eRpw, kF64eStages,
                                              kF64eNativeCols, kF64eSelf, kF64ePack, kF64eBand,
                                              true>(map, prm, pl, dev, stream)
                            : only_q ? launch_f64e<false, dmv::kOutQ>(map, prm, pl, dev, stream)
                                     : launch_f64e<false, dmv::kOutS>(map, prm, pl, dev, stream);
                } else if (kind == Kind::kTma) {
                    e = rev ? launch_stream<T, true, false, dmv::kOutQ, false, kWarps,
                                            default_rpw<T>(), kStages, true>(map, prm, pl, dev,
                                                                              stream)
                        : only_q ? launch_stream<T, true, false, dmv::kOutQ>(map, prm, pl, dev, stream)
                                 : launch_stream<T, true, false, dmv::kOutS>(map, prm, pl, dev, stream);
                } else {
                    e = only_q ? launch_stream<T, false, false, dmv::kOutQ>(map, prm, pl, dev, stream)
                               : launch_stream<T, false, false, dmv::kOutS>(map, prm, pl, dev, stream);
                }
            }
        } else if (kind == Kind::kF64e) {
            e = three_d ? launch_f64e<true>(map, prm, pl, dev, stream)
                        : launch_f64e<false>(map, prm, pl, dev, stream);
            if (e == cudaSuccess) g_last_variant = 0;
        } else if (kind == Kind::kTma) {
            e = three_d ? launch_stream<T, true, true>(map, prm, pl, dev, stream)
                        : launch_stream<T, true, false>(map, prm, pl, dev, stream);
            // Entry 0 of the f64 table is the double-float kernel: the
            // native fp64 default kernel is no entry of it.
            if (e == cudaSuccess && !std::is_same<T, double>::value) g_last_variant = 0;
        } else if (nph > 0) {
            e = launch_phased<T>(nph, pmaps, prm, pl, dev, stream);
        } else {
            e = launch_stream<T, false, false>(map, prm, pl, dev, stream);
        }
    }
    if (e == cudaSuccess) g_last_kernel = kernel_kind;
    if (e == cudaSuccess && ev_stop) e = cudaEventRecord(ev_stop, stream);
    if (e == cudaSuccess && defer != nullptr && !kAtomicOut) {
        defer->used = true;
        defer->prm = prm;
        defer->ws = ws;
        defer->chunks = combine_chunks(prm.bands);
        return DUALMV_SUCCESS;
    }
    if (e == cudaSuccess && !kAtomicOut) e = launch_combine<Acc>(prm, stream);
    cudaError_t ef = ws ? cudaFreeAsync(ws, stream) : cudaSuccess;
    if (e != cudaSuccess) return cuda_fail(e);
    if (ef != cudaSuccess) return cuda_fail(ef);
    return DUALMV_SUCCESS;
}

// --------------------------------------------- operations built on dualmv --

// Stream-ordered scratch of n elements from the device's pool.
template <typename T>
dualmv_status pool_alloc(T **out, int64_t n, cudaStream_t stream) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e);
    DeviceState *ds = nullptr;
    e = device_state(dev, &ds);
    if (e != cudaSuccess) return cuda_fail(e);
    void *p = nullptr;
    e = cudaMallocFromPoolAsync(&p, (size_t)(n > 0 ? n : 1) * sizeof(T), ds->pool, stream);
    if (e != cudaSuccess) {
        g_last_cuda_error = static_cast<int>(e);
        return DUALMV_ERR_ALLOC;
    }
    *out = static_cast<T *>(p);
    return DUALMV_SUCCESS;
}

// GESUMMV (Table 1 / Table 2): tmp = A x, y = B x, y = alpha tmp + beta y.
// Each matrix is streamed once by a rows-only pass; a small kernel forms y.
template <typename T>
dualmv_status gesummv_run(int64_t M, int64_t N, T alpha, const T *A, int64_t lda, T beta,
                          const T *B, int64_t ldb, const T *x, T *y, cudaStream_t stream) {
    if (M < 0 || N < 0 || lda < (N > 1 ? N : 1) || ldb < (N > 1 ? N : 1))
        return DUALMV_ERR_INVALID_VALUE;
    if (M == 0) return DUALMV_SUCCESS;
    if (y == nullptr || (N > 0 && (A == nullptr || B == nullptr || x == nullptr)))
        return DUALMV_ERR_INVALID_VALUE;
    if (N == 0) {
        cudaError_t e = zero_fill(y, M, M, 1, stream);
        return e == cudaSuccess ? DUALMV_SUCCESS : cuda_fail(e);
    }
    if (fault_injected_alloc()) return DUALMV_ERR_ALLOC;
    // Both rows-only passes leave their band partials (no combine kernels);
    // gesummv_final_kernel adds them in the combine's order and forms y.
    // The pass over B shares no buffer with the pass over A, which lets its
    // dependents launch only once every grid before it has completed: B's
    // pass runs in late-wait mode (Params::pdl_late), its CTAs taking the
    // SMs that A's leave, and the final kernel's wait for it covers both.
    T *tmp = nullptr;
    dualmv_status st = pool_alloc(&tmp, M, stream);
    if (st != DUALMV_SUCCESS) return st;
    Deferred da, db;
    st = run<T, T>(M, N, A, lda, 0, x, 0, nullptr, 0, tmp, 0, nullptr, 0, 1, stream,
                   dmv::kOutQ, nullptr, -1, &da);
    if (st == DUALMV_SUCCESS)
        st = run<T, T>(M, N, B, ldb, 0, x, 0, nullptr, 0, y, 0, nullptr, 0, 1, stream,
                       dmv::kOutQ, nullptr, -1, &db, false, true);
    cudaError_t e = cudaSuccess;
    if (st == DUALMV_SUCCESS) {
        if (!da.used) da.prm.q = tmp;
        if (!db.used) db.prm.q = y;
        const int a_direct = (!da.used || da.prm.bands == 1) ? 1 : 0;
        const int b_direct = (!db.used || db.prm.bands == 1) ? 1 : 0;
        const int chunks = da.used ? da.chunks : db.used ? db.chunks : 1;
        const int64_t rows = 256 / chunks;
        const int64_t blocks = (M + rows - 1) / rows;
        if (blocks > INT32_MAX) {
            st = DUALMV_ERR_UNSUPPORTED;
        } else {
            e = launch_dependent(dmv::gesummv_final_kernel<T>, dim3((unsigned)blocks), dim3(256),
                                 0, stream, da.prm, a_direct, db.prm, b_direct, chunks, y, M,
                                 alpha, beta);
            if (e != cudaSuccess) st = cuda_fail(e);
        }
    }
    void *bufs[3] = {da.ws, db.ws, tmp};
    for (void *bp : bufs) {
        if (bp == nullptr) continue;
        cudaError_t ef = cudaFreeAsync(bp, stream);
        if (st == DUALMV_SUCCESS && ef != cudaSuccess) st = cuda_fail(ef);
    }
    return st;
}

// ATAX with one read of A: clusters of C CTAs, each warp a 256-column
// sub-band of R-row stripes (fp32: dualmv_atax.cuh, 16 warps x 4 rows;
// fp64: dualmv_atax_f64.cuh, 8 warps x 4 rows in double-float arithmetic).
// Returns with *used = false, having enqueued nothing, when the problem does
// not fit the cluster path (alignment, width, no cluster of that size can be
// placed), so that the caller takes the two-pass path.
#ifndef DUALMV_ATAX_ROWS
#define DUALMV_ATAX_ROWS 4
#endif
#ifndef DUALMV_ATAX_STAGES
#define DUALMV_ATAX_STAGES 3
#endif
// fp32: 16 warps x 4-row stripes, so that a CTA covers 4096 columns and
// 16384 columns take clusters of 4 (36 fit at once: 144 SMs) instead of 8
// (15: 120 SMs).  89.2% -> 96.9% of HBM on 16384 x 16384.
#ifndef DUALMV_ATAX_WARPS
#define DUALMV_ATAX_WARPS 16
#endif
constexpr int kAtaxWarps = DUALMV_ATAX_WARPS, kAtaxRows = DUALMV_ATAX_ROWS,
              kAtaxStages = DUALMV_ATAX_STAGES;

template <typename T>
struct AtaxCfg;
template <>
struct AtaxCfg<float> {
    static constexpr int W = kAtaxWarps, R = kAtaxRows, S = kAtaxStages, kBand = kBandCols;
    static constexpr int kThreads = W * 32;
    using L = dmv::AtaxLayout<W, R, S>;
    using Params = dmv::AtaxParams;
    static constexpr auto kern = dmv::atax_cluster_kernel<W, R, S>;
    static void fill(Params &p, const float *, int64_t) {}
};
#ifndef DUALMV_ATAX64_WARPS
#define DUALMV_ATAX64_WARPS 8
#endif
#ifndef DUALMV_ATAX64_ROWS
#define DUALMV_ATAX64_ROWS 4
#endif
#ifndef DUALMV_ATAX64_STAGES
#define DUALMV_ATAX64_STAGES 3
#endif
#ifndef DUALMV_ATAX64_BAND
#define DUALMV_ATAX64_BAND 256
#endif
#ifndef DUALMV_ATAX64_NATIVE_VECS
#define DUALMV_ATAX64_NATIVE_VECS 0
#endif
#ifndef DUALMV_ATAX64_SPLIT_WARPS
#define DUALMV_ATAX64_SPLIT_WARPS 1
#endif
template <>
struct AtaxCfg<double> {
    // Three 8 KiB stages per sub-band (the column phase of a stripe runs
    // after its row phase) leave room for 8 sub-bands.  With split warps
    // each sub-band has a row warp and a column warp.
    static constexpr int W = DUALMV_ATAX64_WARPS, R = DUALMV_ATAX64_ROWS,
                         S = DUALMV_ATAX64_STAGES, kBand = DUALMV_ATAX64_BAND;
#if DUALMV_ATAX64_SPLIT_WARPS
    static constexpr int kThreads = (2 * W + 1) * 32;  // and a control warp
    using L = dmv::AtaxLayout64WS<W, R, S, kBand>;
    static constexpr auto kern =
        dmv::atax_cluster_f64_ws_kernel<W, R, S, kBand, DUALMV_ATAX64_NATIVE_VECS>;
#else
    static constexpr int kThreads = (W + 1) * 32;  // and a control warp
    using L = dmv::AtaxLayout64<W, R, S, kBand>;
    static constexpr auto kern = dmv::atax_cluster_f64_kernel<W, R, S, kBand>;
#endif
    using Params = dmv::AtaxParams64;
    static void fill(Params &p, const double *A, int64_t lda) {
        p.A = A;
        p.lda = lda;
    }
};

struct AtaxClusterCache {
    std::mutex mu;
    int max_clusters[2][kMaxDevices][dmv::kAtaxMaxCluster + 1] = {};
    bool known[2][kMaxDevices][dmv::kAtaxMaxCluster + 1] = {};
};
AtaxClusterCache g_atax_cache;

template <typename T>
dualmv_status atax_cluster_run(int64_t M, int64_t N, const T *A, int64_t lda, const T *x, T *y,
                               cudaStream_t stream, bool *used) {
    *used = false;
    using Cfg = AtaxCfg<T>;
    using L = typename Cfg::L;
    constexpr int kT = sizeof(T) == 8 ? 1 : 0;
    const int64_t es = sizeof(T);
    const int64_t bands = (N + Cfg::kBand - 1) / Cfg::kBand;
    const int64_t C = (bands + Cfg::W - 1) / Cfg::W;
    if (g_path == DUALMV_PATH_DIRECT || C > dmv::kAtaxMaxCluster ||
        reinterpret_cast<uintptr_t>(A) % 16 != 0 || (lda * es) % 16 != 0 || M >= INT32_MAX ||
        N >= INT32_MAX)
        return DUALMV_SUCCESS;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e);
    if (dev < 0 || dev >= kMaxDevices) return DUALMV_SUCCESS;
    auto kern = Cfg::kern;
    cudaLaunchConfig_t cfg;
    std::memset(&cfg, 0, sizeof cfg);
    cfg.blockDim = dim3(Cfg::kThreads);
    cfg.dynamicSmemBytes = (size_t)L::kTotal;
    cfg.stream = stream;
    // Clusters of C CTAs; a programmatic dependent of the kernel before it.
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;  // the occupancy query takes the cluster shape alone
    int max_clusters = 0;
    {
        std::lock_guard<std::mutex> lk(g_atax_cache.mu);
        if (!g_atax_cache.known[kT][dev][C]) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)L::kTotal);
            if (e == cudaSuccess && C > 8)
                e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
            if (e == cudaSuccess) {
                cfg.gridDim = dim3((unsigned)C);
                e = cudaOccupancyMaxActiveClusters(&max_clusters, kern, &cfg);
            }
            if (e != cudaSuccess) {  // no such cluster here: use two passes
                (void)cudaGetLastError();
                max_clusters = 0;
            }
            g_atax_cache.max_clusters[kT][dev][C] = max_clusters;
            g_atax_cache.known[kT][dev][C] = true;
        }
        max_clusters = g_atax_cache.max_clusters[kT][dev][C];
    }
    if (max_clusters <= 0) return DUALMV_SUCCESS;
    CUtensorMap map;
    std::memset(&map, 0, sizeof map);
    if (!encode_a<T>(&map, A, M, N, lda, M * lda, 1, Cfg::kBand, Cfg::R, false))
        return DUALMV_SUCCESS;
    const int64_t stripes = (M + Cfg::R - 1) / Cfg::R;
    const int64_t clusters = stripes < max_clusters ? stripes : max_clusters;
    T *ws = nullptr;
    dualmv_status st = pool_alloc(&ws, clusters * N, stream);
    if (st != DUALMV_SUCCESS) return st;
    *used = true;
    typename Cfg::Params prm;
    std::memset(&prm, 0, sizeof prm);
    Cfg::fill(prm, A, lda);
    prm.x = x;
    prm.y_ws = ws;
    prm.M = M;
    prm.N = N;
    prm.stripes = stripes;
    prm.clusters = clusters;
    prm.bands = bands;
    cfg.gridDim = dim3((unsigned)(clusters * C));
    cfg.numAttrs = 2;
    e = cudaLaunchKernelEx(&cfg, kern, map, prm);
    if (e == cudaSuccess) {
        int64_t blocks = (N + 255) / 256;
        if (blocks > 4096) blocks = 4096;
        e = launch_dependent(dmv::atax_sum_kernel<T>, dim3((unsigned)blocks), dim3(256), 0,
                             stream, (const T *)ws, y, N, clusters);
    }
    cudaError_t ef = cudaFreeAsync(ws, stream);
    if (e != cudaSuccess) return cuda_fail(e);
    if (ef != cudaSuccess) return cuda_fail(ef);
    return DUALMV_SUCCESS;
}

// ATAX (Table 1): y = A^T (A x).  The single-read cluster path when it fits;
// otherwise tmp = A x by a rows-only pass and y = A^T tmp by a columns-only
// pass over the same A.
template <typename T>
dualmv_status atax_run(int64_t M, int64_t N, const T *A, int64_t lda, const T *x, T *y,
                       cudaStream_t stream) {
    g_last_atax_path = -1;
    if (M < 0 || N < 0 || lda < (N > 1 ? N : 1)) return DUALMV_ERR_INVALID_VALUE;
    if (N == 0) return DUALMV_SUCCESS;
    if (y == nullptr || (M > 0 && (A == nullptr || x == nullptr)))
        return DUALMV_ERR_INVALID_VALUE;
    if (M == 0) {
        cudaError_t e = zero_fill(y, N, N, 1, stream);
        return e == cudaSuccess ? DUALMV_SUCCESS : cuda_fail(e);
    }
    if (fault_injected_alloc()) return DUALMV_ERR_ALLOC;
    if (g_atax_two_pass == 0) {
        bool used = false;
        dualmv_status sc = atax_cluster_run<T>(M, N, A, lda, x, y, stream, &used);
        if (sc == DUALMV_SUCCESS && used) g_last_atax_path = DUALMV_ATAX_ONE_READ;
        if (sc != DUALMV_SUCCESS || used) return sc;
    }
    T *tmp = nullptr;
    dualmv_status st = pool_alloc(&tmp, M, stream);
    if (st != DUALMV_SUCCESS) return st;
    st = run<T, T>(M, N, A, lda, 0, x, 0, nullptr, 0, tmp, 0, nullptr, 0, 1, stream,
                   dmv::kOutQ);
    if (st == DUALMV_SUCCESS)
        st = run<T, T>(M, N, A, lda, 0, nullptr, 0, tmp, 0, nullptr, 0, y, 0, 1, stream,
                       dmv::kOutS);
    cudaError_t ef = cudaFreeAsync(tmp, stream);
    if (st == DUALMV_SUCCESS && ef != cudaSuccess) st = cuda_fail(ef);
    if (st == DUALMV_SUCCESS) g_last_atax_path = DUALMV_ATAX_TWO_PASS;
    return st;
}

// GEMVER without writing A_hat: the rank-2 update factorises,
//   A_hat^T y = A^T y + v1 (u1 . y) + v2 (u2 . y),
//   A_hat x   = A x   + u1 (v1 . x) + u2 (v2 . x),
// so a columns-only and a rows-only pass of the plain kernels (double-float
// for fp64) and four dot products give x and w without any per-element
// update.  Each term's error stays within the bar of A_hat's magnitudes.
// The general shape (M, N > 0): five kernels.  The u . y dot products; the
// columns-only pass, which leaves its partials for gemver_x3_kernel, which
// adds them and updates x; the rows-only pass, which leaves its partials for
// gemver_w3_kernel, which adds them and updates w.  (Seven before: each pass
// had its own combine kernel.  Forming u . y inside the x kernel, every
// block for itself, put 130 thousand fp64 operations on each SM's narrow
// FP64 pipe and doubled the call.)
template <typename T>
dualmv_status gemver_factored_fused(int64_t M, int64_t N, T alpha, T beta, const T *A,
                                    int64_t lda, const T *u1, const T *v1, const T *u2,
                                    const T *v2, T *w, T *x, const T *y, const T *z,
                                    cudaStream_t stream) {
    T *s = nullptr, *t = nullptr;
    // [side][2 products][kDotChunks] chunk sums: u . y, then v . x
    double *part = nullptr;
    dualmv_status st = pool_alloc(&s, N, stream);
    if (st == DUALMV_SUCCESS) st = pool_alloc(&t, M, stream);
    if (st == DUALMV_SUCCESS) st = pool_alloc(&part, 2 * 2 * dmv::kDotChunks, stream);
    double *part_u = part, *part_v = part ? part + 2 * dmv::kDotChunks : nullptr;
    cudaError_t e = cudaSuccess;
    Deferred ds, dq;
    if (st == DUALMV_SUCCESS)
        e = launch_dependent(dmv::dots2_partial_kernel<T>, dim3(2 * dmv::kDotChunks),
                             dim3(dmv::kDotThreads), 0, stream, u1, u2, y, M, part_u);
    // s = A^T y, left as partials.  The pass runs beside the dots kernel
    // (late wait, Params::pdl_late): neither touches the other's memory.
    if (st == DUALMV_SUCCESS && e == cudaSuccess)
        st = run<T, T>(M, N, A, lda, 0, nullptr, 0, y, 0, nullptr, 0, s, 0, 1, stream,
                       dmv::kOutS, nullptr, -1, &ds, false, true);
    if (st == DUALMV_SUCCESS && e == cudaSuccess) {
        if (!ds.used) ds.prm.s = s;
        e = launch_dependent(dmv::gemver_x3_kernel<T>, dim3(dmv::kDotChunks), dim3(256), 0,
                             stream, ds.prm, ds.used ? 0 : 1, (const double *)part_u, x, v1,
                             v2, z, N, beta, part_v);
    }
    if (ds.ws != nullptr) {
        cudaError_t ef = cudaFreeAsync(ds.ws, stream);
        if (e == cudaSuccess) e = ef;
    }
    // t = A x, left as partials; each CTA walks its tiles backwards, so it
    // starts on those the columns-only pass read last (still in L2).
    if (st == DUALMV_SUCCESS && e == cudaSuccess)
        st = run<T, T>(M, N, A, lda, 0, x, 0, nullptr, 0, t, 0, nullptr, 0, 1, stream,
                       dmv::kOutQ, nullptr, -1, &dq, true);
    if (st == DUALMV_SUCCESS && e == cudaSuccess) {
        if (!dq.used) dq.prm.q = t;
        const int direct = (!dq.used || dq.prm.bands == 1) ? 1 : 0;
        const int64_t rows = 256 / dq.chunks;
        const int64_t bw = (M + rows - 1) / rows;
        if (bw > INT32_MAX) e = cudaErrorInvalidConfiguration;
        else
            e = launch_dependent(dmv::gemver_w3_kernel<T>, dim3((unsigned)bw), dim3(256), 0,
                                 stream, dq.prm, direct, dq.chunks, w, u1, u2,
                                 (const double *)part_v, M, alpha);
    }
    if (dq.ws != nullptr) {
        cudaError_t ef = cudaFreeAsync(dq.ws, stream);
        if (e == cudaSuccess) e = ef;
    }
    if (st == DUALMV_SUCCESS && e != cudaSuccess) st = cuda_fail(e);
    void *bufs[3] = {s, t, part};
    for (void *bp : bufs) {
        if (bp == nullptr) continue;
        cudaError_t ef = cudaFreeAsync(bp, stream);
        if (st == DUALMV_SUCCESS && ef != cudaSuccess) st = cuda_fail(ef);
    }
    return st;
}

template <typename T>
dualmv_status gemver_factored(int64_t M, int64_t N, T alpha, T beta, const T *A, int64_t lda,
                              const T *u1, const T *v1, const T *u2, const T *v2, T *w, T *x,
                              const T *y, const T *z, cudaStream_t stream) {
    if (M > 0 && N > 0)
        return gemver_factored_fused<T>(M, N, alpha, beta, A, lda, u1, v1, u2, v2, w, x, y, z,
                                        stream);
    // An empty dimension: the vector kernels alone (each pass zero-fills).
    T *s = nullptr, *t = nullptr;
    // [side][2 products][kDotChunks] chunk sums: u . y, then v . x
    double *part = nullptr;
    dualmv_status st = pool_alloc(&s, N, stream);
    if (st == DUALMV_SUCCESS) st = pool_alloc(&t, M, stream);
    if (st == DUALMV_SUCCESS) st = pool_alloc(&part, 2 * 2 * dmv::kDotChunks, stream);
    double *part_u = part, *part_v = part ? part + 2 * dmv::kDotChunks : nullptr;
    cudaError_t e = cudaSuccess;
    // The vector kernels are programmatic dependents of the kernel before
    // them (each waits for it before reading): their launches overlap it.
    if (st == DUALMV_SUCCESS && N > 0) {  // s = A^T y (zero when M == 0)
        e = launch_dependent(dmv::dots2_partial_kernel<T>, dim3(2 * dmv::kDotChunks),
                             dim3(dmv::kDotThreads), 0, stream, u1, u2, y, M, part_u);
        if (e == cudaSuccess)
            st = run<T, T>(M, N, A, lda, 0, nullptr, 0, y, 0, nullptr, 0, s, 0, 1, stream,
                           dmv::kOutS);
        // x, and the chunk sums of v1 . x and v2 . x for the new x.
        if (e == cudaSuccess && st == DUALMV_SUCCESS)
            e = launch_dependent(dmv::gemver_x2_kernel<T>, dim3(dmv::kDotChunks), dim3(256), 0,
                                 stream, x, (const T *)s, v1, v2, (const double *)part_u, z, N,
                                 beta, part_v);
    } else if (st == DUALMV_SUCCESS && M > 0) {  // N == 0: v . x is zero
        e = launch_dependent(dmv::dots2_partial_kernel<T>, dim3(2 * dmv::kDotChunks),
                             dim3(dmv::kDotThreads), 0, stream, v1, v2, x, N, part_v);
    }
    if (st == DUALMV_SUCCESS && e == cudaSuccess && M > 0) {  // t = A x (zero when N == 0)
        st = run<T, T>(M, N, A, lda, 0, x, 0, nullptr, 0, t, 0, nullptr, 0, 1, stream,
                       dmv::kOutQ);
        if (st == DUALMV_SUCCESS) {
            const int64_t bw = (M + 255) / 256;
            e = launch_dependent(dmv::gemver_w2_kernel<T>, dim3((unsigned)(bw > 4096 ? 4096 : bw)),
                                 dim3(256), 0, stream, w, (const T *)t, u1, u2,
                                 (const double *)part_v, M, alpha);
        }
    }
    if (st == DUALMV_SUCCESS && e != cudaSuccess) st = cuda_fail(e);
    void *bufs[3] = {s, t, part};
    for (void *bp : bufs) {
        if (bp == nullptr) continue;
        cudaError_t ef = cudaFreeAsync(bp, stream);
        if (st == DUALMV_SUCCESS && ef != cudaSuccess) st = cuda_fail(ef);
    }
    return st;
}

// GEMVER (Table 1 / Table 2): A_hat = A + u1 v1^T + u2 v2^T;
// GEMVER with update_A: the factorised columns pass and x update of
// gemver_factored_fused, then gemver_rows_update_{f64,f32}_kernel, which
// writes A_hat over A and leaves the band partials of A x (original A), and
// the w update, which adds them.  A read twice and written once.  fp64: two
// DFMAs per element (A_hat) where the on-the-fly kernel takes three.
// Needs A 16-byte aligned and a row stride that is a multiple of 16 bytes.
template <typename T>
dualmv_status gemver_update(int64_t M, int64_t N, T alpha, T beta, T *A, int64_t lda,
                            const T *u1, const T *v1, const T *u2, const T *v2, T *w, T *x,
                            const T *y, const T *z, cudaStream_t stream) {
    constexpr bool kF64 = std::is_same<T, double>::value;
    constexpr int64_t kBand = kF64 ? dmv::kGvBand : dmv::kGvBand32;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e);
    DeviceState *dst = nullptr;
    e = device_state(dev, &dst);
    if (e != cudaSuccess) return cuda_fail(e);
    const int64_t bands = (N + kBand - 1) / kBand;
    int64_t row_chunks = (2 * (int64_t)dst->sms + bands - 1) / bands;
    if (row_chunks > M) row_chunks = M;
    if (row_chunks < 1) row_chunks = 1;
    if (bands > 65535 || row_chunks > INT32_MAX) return DUALMV_ERR_UNSUPPORTED;
    T *s = nullptr, *qws = nullptr;
    double *part = nullptr;  // [side][2 products][kDotChunks] chunk sums
    dualmv_status st = pool_alloc(&s, N, stream);
    if (st == DUALMV_SUCCESS) st = pool_alloc(&part, 2 * 2 * dmv::kDotChunks, stream);
    if (st == DUALMV_SUCCESS) st = pool_alloc(&qws, bands * M, stream);
    double *part_u = part, *part_v = part ? part + 2 * dmv::kDotChunks : nullptr;
    Deferred ds;
    if (st == DUALMV_SUCCESS)
        e = launch_dependent(dmv::dots2_partial_kernel<T>, dim3(2 * dmv::kDotChunks),
                             dim3(dmv::kDotThreads), 0, stream, u1, u2, y, M, part_u);
    // s = A^T y, left as partials.  The pass runs beside the dots kernel
    // (late wait, Params::pdl_late): neither touches the other's memory.
    if (st == DUALMV_SUCCESS && e == cudaSuccess)
        st = run<T, T>(M, N, A, lda, 0, nullptr, 0, y, 0, nullptr, 0, s, 0, 1, stream,
                       dmv::kOutS, nullptr, -1, &ds, false, true);
    if (st == DUALMV_SUCCESS && e == cudaSuccess) {
        if (!ds.used) ds.prm.s = s;
        e = launch_dependent(dmv::gemver_x3_kernel<T>, dim3(dmv::kDotChunks), dim3(256), 0,
                             stream, ds.prm, ds.used ? 0 : 1, (const double *)part_u, x, v1,
                             v2, z, N, beta, part_v);
    }
    if (ds.ws != nullptr) {
        cudaError_t ef = cudaFreeAsync(ds.ws, stream);
        if (e == cudaSuccess) e = ef;
    }
    if (st == DUALMV_SUCCESS && e == cudaSuccess) {
        dmv::GvParams<T> gp;
        std::memset(&gp, 0, sizeof gp);
        gp.A = A;
        gp.lda = lda;
        gp.u1 = u1;
        gp.u2 = u2;
        gp.v1 = v1;
        gp.v2 = v2;
        gp.x = x;
        gp.q_ws = qws;
        gp.M = M;
        gp.N = N;
        gp.bands = bands;
        gp.row_chunks = row_chunks;
        const dim3 grid((unsigned)row_chunks, (unsigned)bands);
        if constexpr (kF64)
            e = launch_dependent(dmv::gemver_rows_update_f64_kernel, grid,
                                 dim3(dmv::kGvWarps * 32), 0, stream, gp);
        else
            e = launch_dependent(dmv::gemver_rows_update_f32_kernel, grid,
                                 dim3(dmv::kGvWarps * 32), 0, stream, gp);
    }
    if (st == DUALMV_SUCCESS && e == cudaSuccess) {
        Params pq;
        std::memset(&pq, 0, sizeof pq);
        pq.q_ws = qws;
        pq.bands = bands;
        pq.M = M;
        pq.batch = 1;
        const int chunks = combine_chunks(bands);
        const int64_t rows = 256 / chunks;
        const int64_t bw = (M + rows - 1) / rows;
        if (bw > INT32_MAX) e = cudaErrorInvalidConfiguration;
        else
            e = launch_dependent(dmv::gemver_w3_kernel<T>, dim3((unsigned)bw), dim3(256), 0,
                                 stream, pq, 0, chunks, w, u1, u2, (const double *)part_v, M,
                                 alpha);
    }
    if (st == DUALMV_SUCCESS && e != cudaSuccess) st = cuda_fail(e);
    void *bufs[3] = {s, part, qws};
    for (void *bp : bufs) {
        if (bp == nullptr) continue;
        cudaError_t ef = cudaFreeAsync(bp, stream);
        if (st == DUALMV_SUCCESS && ef != cudaSuccess) st = cuda_fail(ef);
    }
    return st;
}

// x = x + beta A_hat^T y + z;  w = w + alpha A_hat x.  Without update_A the
// factorised form above runs.  With it, two passes apply the rank-2 update
// as they stream A: a columns-only pass (A_hat^T y) and, after the x
// update, a rows-only pass (A_hat x) that also writes A_hat over A.  A is
// read twice and written once.
template <typename T>
dualmv_status gemver_run(int64_t M, int64_t N, T alpha, T beta, T *A, int64_t lda,
                         int update_A, const T *u1, const T *v1, const T *u2, const T *v2,
                         T *w, T *x, const T *y, const T *z, cudaStream_t stream) {
    g_last_gemver_path = -1;
    if (M < 0 || N < 0 || lda < (N > 1 ? N : 1)) return DUALMV_ERR_INVALID_VALUE;
    if (N > 0 && (x == nullptr || z == nullptr || v1 == nullptr || v2 == nullptr))
        return DUALMV_ERR_INVALID_VALUE;
    if (M > 0 && (w == nullptr || y == nullptr || u1 == nullptr || u2 == nullptr))
        return DUALMV_ERR_INVALID_VALUE;
    if (M > 0 && N > 0 && A == nullptr) return DUALMV_ERR_INVALID_VALUE;
    if (M == 0 && N == 0) return DUALMV_SUCCESS;
    if (fault_injected_alloc()) return DUALMV_ERR_ALLOC;
    if (!update_A && g_gemver_onthefly == 0) {
        g_last_gemver_path = DUALMV_GEMVER_FACTORED;
        return gemver_factored<T>(M, N, alpha, beta, A, lda, u1, v1, u2, v2, w, x, y, z,
                                  stream);
    }
    if (g_gemver_onthefly == 0 && M > 0 && N > 0 && (lda * (int64_t)sizeof(T)) % 16 == 0 &&
        reinterpret_cast<uintptr_t>(A) % 16 == 0) {
        g_last_gemver_path = DUALMV_GEMVER_UPDATE_SPLIT;
        return gemver_update<T>(M, N, alpha, beta, A, lda, u1, v1, u2, v2, w, x, y, z, stream);
    }
    g_last_gemver_path = DUALMV_GEMVER_ONTHEFLY;
    T *s = nullptr, *t = nullptr;
    dualmv_status st = pool_alloc(&s, N, stream);
    if (st != DUALMV_SUCCESS) return st;
    st = pool_alloc(&t, M, stream);
    if (st != DUALMV_SUCCESS) {
        cudaFreeAsync(s, stream);
        return st;
    }
    Rank2 upd{u1, v1, u2, v2, nullptr, lda};
    if (N > 0)  // s = A_hat^T y (zero when M == 0)
        st = run<T, T>(M, N, A, lda, 0, nullptr, 0, y, 0, nullptr, 0, s, 0, 1, stream,
                       dmv::kOutS, &upd);
    const int64_t bx = N > 0 ? (N + 255) / 256 : 0, bw = M > 0 ? (M + 255) / 256 : 0;
    if (st == DUALMV_SUCCESS && N > 0) {
        dmv::gemver_x_kernel<T><<<(unsigned)(bx > 4096 ? 4096 : bx), 256, 0, stream>>>(
            x, s, z, N, beta);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) st = cuda_fail(e);
    }
    if (st == DUALMV_SUCCESS && M > 0) {  // t = A_hat x (zero when N == 0)
        upd.a_out = update_A ? A : nullptr;
        st = run<T, T>(M, N, A, lda, 0, x, 0, nullptr, 0, t, 0, nullptr, 0, 1, stream,
                       dmv::kOutQ, &upd);
    }
    if (st == DUALMV_SUCCESS && M > 0) {
        dmv::gemver_w_kernel<T><<<(unsigned)(bw > 4096 ? 4096 : bw), 256, 0, stream>>>(
            w, t, M, alpha);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) st = cuda_fail(e);
    }
    cudaError_t e1 = cudaFreeAsync(s, stream), e2 = cudaFreeAsync(t, stream);
    if (st == DUALMV_SUCCESS && (e1 != cudaSuccess || e2 != cudaSuccess))
        st = cuda_fail(e1 != cudaSuccess ? e1 : e2);
    return st;
}

// ----------------------------------------------------------------- tuner --
//
// The performance-feedback loop of Section 3.2 over the compiled variants:
// candidates near the current baseline, a functional-equivalence gate
// (Eq. 4), the trimmed mean of repeated timings as the score (Eq. 3), and
// the fastest feasible candidate as the next baseline (Eq. 5).

bool trimmed_mean_of(std::vector<double> t, int64_t k, double *out) {
    const int64_t R = (int64_t)t.size();
    if (k < 0 || R <= 2 * k) return false;
    std::sort(t.begin(), t.end());
    double sum = 0.0;
    for (int64_t i = k; i < R - k; ++i) sum += t[i];
    *out = sum / (double)(R - 2 * k);
    return true;
}

// Reads and clears the device fault word after synchronising `stream`.
cudaError_t take_fault_word(cudaStream_t stream, unsigned int *word) {
    cudaError_t e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return e;
    e = cudaMemcpyFromSymbol(word, dmv::g_fault_word, sizeof *word);
    if (e != cudaSuccess || *word == 0) return e;
    const unsigned int zero = 0;
    return cudaMemcpyToSymbol(dmv::g_fault_word, &zero, sizeof zero);
}

template <typename T> constexpr double fe_tolerance() {
    return std::is_same<T, float>::value ? 1e-5 : std::is_same<T, double>::value ? 1e-12 : 0.0;
}

template <typename T, typename Out>
class Tuner {
  public:
    // One problem (batch 1) or a strided batch; strides in elements.  With
    // outputs kOutQ or kOutS, single-sided passes of one problem (the
    // other side's pointers unused).
    Tuner(int64_t M, int64_t N, int64_t batch, const T *A, int64_t lda, int64_t strideA,
          const T *p, int64_t strideP, const T *r, int64_t strideR, Out *q, int64_t strideQ,
          Out *s, int64_t strideS, const dualmv_tune_config_t &cfg, cudaStream_t stream,
          uint32_t outputs = dmv::kOutBoth)
        : M_(M), N_(N), batch_(batch), A_(A), lda_(lda), strideA_(strideA), p_(p),
          strideP_(strideP), r_(r), strideR_(strideR), q_(q), strideQ_(strideQ), s_(s),
          strideS_(strideS), cfg_(cfg), stream_(stream), outputs_(outputs),
          want_q_((outputs & dmv::kOutQ) != 0), want_s_((outputs & dmv::kOutS) != 0) {}

    ~Tuner() {
        for (cudaEvent_t ev : events_) cudaEventDestroy(ev);
        void *bufs[] = {q_base_, s_base_, den_q_, den_s_, fe_word_, flush_};
        for (void *b : bufs)
            if (b) cudaFreeAsync(b, stream_);
        cudaStreamSynchronize(stream_);
    }

    dualmv_status setup() {
        dualmv_status st = DUALMV_SUCCESS;
        if (want_q_) st = pool_alloc(&q_base_, batch_ * M_, stream_);
        if (st == DUALMV_SUCCESS && want_s_) st = pool_alloc(&s_base_, batch_ * N_, stream_);
        if (st == DUALMV_SUCCESS) st = pool_alloc(&fe_word_, 1, stream_);
        constexpr bool kExact = std::is_same<T, int32_t>::value;
        if (!kExact) {
            if (st == DUALMV_SUCCESS && want_q_) st = pool_alloc(&den_q_, batch_ * M_, stream_);
            if (st == DUALMV_SUCCESS && want_s_) st = pool_alloc(&den_s_, batch_ * N_, stream_);
        }
        if (st != DUALMV_SUCCESS) return st;
        int dev = 0, l2 = 0, sms = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return cuda_fail(e);
        if (cfg_.flush_l2) {
            flush_bytes_ = 2 * (int64_t)l2;
            st = pool_alloc(&flush_, flush_bytes_, stream_);
            if (st != DUALMV_SUCCESS) return st;
        }
        events_.resize(2 * (size_t)cfg_.repeats, nullptr);
        for (cudaEvent_t &ev : events_) {
            e = cudaEventCreate(&ev);
            if (e != cudaSuccess) return cuda_fail(e);
        }
        if (!kExact) {  // magnitude sums for the equivalence bar, once per problem
            const int64_t bc = (N_ + 255) / 256;
            for (int64_t b = 0; b < batch_; ++b) {
                if (want_q_)
                    dmv::abs_rows_kernel<T><<<4 * sms, 256, 0, stream_>>>(
                        A_ + b * strideA_, M_, N_, lda_, p_ + b * strideP_, den_q_ + b * M_);
                if (want_s_)
                    dmv::abs_cols_kernel<T>
                        <<<(unsigned)(bc < 65535 ? bc : 65535), 256, 0, stream_>>>(
                            A_ + b * strideA_, M_, N_, lda_, r_ + b * strideR_, den_s_ + b * N_);
                e = cudaGetLastError();
                if (e != cudaSuccess) return cuda_fail(e);
            }
        }
        return DUALMV_SUCCESS;
    }

    // One call of variant `v` into q, s (or the baseline buffers, packed).
    dualmv_status call(int32_t v, bool into_base) {
        Out *q = into_base ? q_base_ : q_, *s = into_base ? s_base_ : s_;
        const int64_t sq = into_base ? M_ : strideQ_, ss = into_base ? N_ : strideS_;
        return run<T, Out>(M_, N_, A_, lda_, strideA_, p_, strideP_, r_, strideR_, q, sq, s, ss,
                           batch_, stream_, outputs_, nullptr, v);
    }

    // Score of Eq. 3: `repeats` timed calls, trimmed mean of their times.
    dualmv_status score(int32_t v, double *ms) {
        const int R = cfg_.repeats;
        for (int i = 0; i < R; ++i) {
            cudaError_t e = cudaSuccess;
            if (flush_) e = cudaMemsetAsync(flush_, i & 0xff, (size_t)flush_bytes_, stream_);
            if (e == cudaSuccess) e = cudaEventRecord(events_[2 * i], stream_);
            if (e != cudaSuccess) return cuda_fail(e);
            dualmv_status st = call(v, false);
            if (st != DUALMV_SUCCESS) return st;
            e = cudaEventRecord(events_[2 * i + 1], stream_);
            if (e != cudaSuccess) return cuda_fail(e);
        }
        dualmv_status st = check_fault();
        if (st != DUALMV_SUCCESS) return st;
        std::vector<double> t((size_t)R);
        for (int i = 0; i < R; ++i) {
            float f = 0.f;
            cudaError_t e = cudaEventElapsedTime(&f, events_[2 * i], events_[2 * i + 1]);
            if (e != cudaSuccess) return cuda_fail(e);
            t[(size_t)i] = f;
        }
        trimmed_mean_of(t, cfg_.trim, ms);
        return DUALMV_SUCCESS;
    }

    // Eq. 4: the largest per-element error of q, s against the baseline's.
    dualmv_status equivalence(double *err) {
        cudaError_t e = cudaMemsetAsync(fe_word_, 0, sizeof(unsigned long long), stream_);
        const unsigned gq = (unsigned)std::min<int64_t>((M_ + 255) / 256, 1024);
        const unsigned gs = (unsigned)std::min<int64_t>((N_ + 255) / 256, 1024);
        for (int64_t b = 0; b < batch_ && e == cudaSuccess; ++b) {
            if (want_q_)
                dmv::fe_max_kernel<Out><<<gq, 256, 0, stream_>>>(
                    q_ + b * strideQ_, q_base_ + b * M_, den_q_ ? den_q_ + b * M_ : nullptr, M_,
                    fe_word_);
            if (want_s_)
                dmv::fe_max_kernel<Out><<<gs, 256, 0, stream_>>>(
                    s_ + b * strideS_, s_base_ + b * N_, den_s_ ? den_s_ + b * N_ : nullptr, N_,
                    fe_word_);
            e = cudaGetLastError();
        }
        unsigned long long bits = 0;
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(&bits, fe_word_, sizeof bits, cudaMemcpyDeviceToHost, stream_);
        if (e == cudaSuccess) e = cudaStreamSynchronize(stream_);
        if (e != cudaSuccess) return cuda_fail(e);
        std::memcpy(err, &bits, sizeof bits);
        return DUALMV_SUCCESS;
    }

    dualmv_status check_fault() {
        unsigned int word = 0;
        cudaError_t e = take_fault_word(stream_, &word);
        if (e != cudaSuccess) return cuda_fail(e);
        return word ? DUALMV_ERR_TIMEOUT : DUALMV_SUCCESS;
    }

    // A planted mistake in a candidate's outputs, for testing the gate.
    dualmv_status plant_mistake() {
        cudaError_t e = cudaMemsetAsync(want_q_ ? q_ : s_, 0x7f, sizeof(Out), stream_);
        return e == cudaSuccess ? DUALMV_SUCCESS : cuda_fail(e);
    }

  private:
    int64_t M_, N_, batch_;
    const T *A_;
    int64_t lda_, strideA_;
    const T *p_;
    int64_t strideP_;
    const T *r_;
    int64_t strideR_;
    Out *q_;
    int64_t strideQ_;
    Out *s_;
    int64_t strideS_;
    dualmv_tune_config_t cfg_;
    cudaStream_t stream_;
    uint32_t outputs_;
    bool want_q_, want_s_;
    Out *q_base_ = nullptr, *s_base_ = nullptr;
    double *den_q_ = nullptr, *den_s_ = nullptr;
    unsigned long long *fe_word_ = nullptr;
    unsigned char *flush_ = nullptr;
    int64_t flush_bytes_ = 0;
    std::vector<cudaEvent_t> events_;
};

// The loop of Section 3.2 for one problem (batch 1) or a strided batch (the
// candidates then are the variants with a batched instance); with outputs
// kOutQ or kOutS, for a single-sided pass of one problem (the candidates are
// the variants with single-sided instances).
template <typename T, typename Out>
dualmv_status tune_run(int64_t M, int64_t N, int64_t batch, const T *A, int64_t lda,
                       int64_t strideA, const T *p, int64_t strideP, const T *r,
                       int64_t strideR, Out *q, int64_t strideQ, Out *s, int64_t strideS,
                       const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
                       cudaStream_t stream, uint32_t outputs = dmv::kOutBoth) {
    if (cfg == nullptr || res == nullptr) return DUALMV_ERR_INVALID_VALUE;
    if (cfg->trim < 0 || cfg->repeats <= 2 * cfg->trim || cfg->max_rounds < 0 ||
        cfg->candidates < 1 || !(cfg->min_gain >= 0.0))
        return DUALMV_ERR_INVALID_VALUE;
    const bool sided = outputs != dmv::kOutBoth;
    if (sided && (batch != 1 || std::is_same<T, int32_t>::value)) return DUALMV_ERR_INVALID_VALUE;
    dualmv_status st = validate(M, N, A, lda, strideA, p, strideP, r, strideR, q, strideQ, s,
                                strideS, batch, outputs);
    if (st != DUALMV_SUCCESS) return st;
    std::memset(res, 0, sizeof *res);
    const int64_t es = sizeof(T);
    const bool batched = batch > 1;
    const bool eligible = M > 0 && N > 0 && batch > 0 && g_path != DUALMV_PATH_DIRECT &&
                          g_path != DUALMV_PATH_TMA_NATIVE_F64 &&
                          reinterpret_cast<uintptr_t>(A) % 16 == 0 && (lda * es) % 16 == 0 &&
                          (!batched || (strideA * es) % 16 == 0) && M < INT32_MAX &&
                          N < INT32_MAX && batch < INT32_MAX;
    if (!eligible)
        return run<T, Out>(M, N, A, lda, strideA, p, strideP, r, strideR, q, strideQ, s, strideS,
                           batch, stream, outputs);
    if (fault_injected_alloc()) return DUALMV_ERR_ALLOC;

    const int32_t dtype = dtype_code<T>();
    const std::vector<Variant> &tab = *variant_table(dtype);
    constexpr double tol = fe_tolerance<T>();
    const bool plant = fault_injected("fe");
    Tuner<T, Out> tu(M, N, batch, A, lda, strideA, p, strideP, r, strideR, q, strideQ, s,
                     strideS, *cfg, stream, outputs);
    st = tu.setup();
    if (st != DUALMV_SUCCESS) return st;

    // K^(0): the variant an untuned call of this shape uses; its outputs are
    // the reference for Eq. 4.
    int32_t base = batched ? 0
                   : sided ? sided_default_variant(dtype)
                           : default_variant(dtype, A, lda * es);
    res->initial = base;
    st = tu.call(base, true);
    if (st == DUALMV_SUCCESS) st = tu.score(base, &res->baseline_ms);
    if (st != DUALMV_SUCCESS) return st;
    double base_ms = res->baseline_ms;
    std::vector<bool> tried(tab.size(), false);
    tried[base] = true;

    for (int32_t d = 0; d < cfg->max_rounds; ++d) {
        std::vector<int32_t> cands;
        for (const Variant &v : tab)
            if (!tried[v.info.index] && (!batched || v.launch3d != nullptr) &&
                (!sided || v.launch_q != nullptr) && neighbours(v.info, tab[base].info) &&
                (int32_t)cands.size() < cfg->candidates)
                cands.push_back(v.info.index);
        if (cands.empty()) break;
        res->rounds = d + 1;
        int32_t best = -1;
        double best_ms = 0.0;
        for (int32_t c : cands) {
            tried[c] = true;
            ++res->evaluated;
            dualmv_tune_step_t *step = nullptr;
            if (res->trace_len < DUALMV_TUNE_MAX_TRACE) {
                step = &res->trace[res->trace_len++];
                step->index = c;
                step->round = d;
            }
            st = tu.call(c, false);
            if (st == DUALMV_SUCCESS && plant) st = tu.plant_mistake();
            if (st == DUALMV_SUCCESS) st = tu.check_fault();
            double err = 0.0;
            if (st == DUALMV_SUCCESS) st = tu.equivalence(&err);
            if (st != DUALMV_SUCCESS) return st;
            if (step) step->fe = err;
            if (!(err <= tol)) {  // Eq. 4: not in the feasible set
                ++res->rejected;
                continue;
            }
            if (err > res->worst_fe) res->worst_fe = err;
            double ms = 0.0;
            st = tu.score(c, &ms);
            if (st != DUALMV_SUCCESS) return st;
            if (step) {
                step->feasible = 1;
                step->ms = ms;
            }
            if (best < 0 || ms < best_ms) {  // Eq. 5
                best = c;
                best_ms = ms;
            }
        }
        if (best < 0 || !(best_ms < base_ms * (1.0 - cfg->min_gain))) break;
        base = best;
        base_ms = best_ms;
        st = tu.call(base, true);  // the new baseline's outputs, for Eq. 4
        if (st != DUALMV_SUCCESS) return st;
    }
    res->best = base;
    res->best_ms = base_ms;
    {
        std::lock_guard<std::mutex> lk(g_tuned_mu);
        g_tuned[std::make_tuple(dtype, M, N, lda, batched ? batch : (int64_t)1, outputs)] = base;
        g_tuned_count.store((int)g_tuned.size(), std::memory_order_release);
    }
    st = tu.call(base, false);  // leave the chosen variant's outputs in q, s
    if (st != DUALMV_SUCCESS) return st;
    return tu.check_fault();
}

// ------------------------------------------------- no-allocation variant --
//
// Some callers cannot allocate device memory while they run dualmv: code
// inside a framework that owns every device allocation (a fixed memory
// budget, or a custom allocator that dualmv cannot see), real-time loops
// that must not call into the allocator, and code that must not add
// synchronising or pool-growing calls on a hot stream.  dualmv_f32_noalloc
// serves them: its scratch (the band partials of q and segment partials of s
// that the combine kernel reads) lives in this fixed device array, which
// every GPU that loads the library holds until the process exits.
constexpr int64_t kNoallocScratchBytes = 8ll << 20;  // 8 MiB
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

struct NoallocDevice {
    std::once_flag once;
    cudaError_t error = cudaSuccess;
    int sms = 0;
    void *scratch = nullptr;  // device address of g_noalloc_scratch
};
NoallocDevice g_noalloc_dev[kMaxDevices];

// Once per device, with that device current: the SM count and the device
// address of the scratch array (in host code the array's name is only a
// stand-in, never a device address).
cudaError_t noalloc_setup(int dev, NoallocDevice **out) {
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    NoallocDevice &nd = g_noalloc_dev[dev];
    std::call_once(nd.once, [&]() {
        cudaError_t e = cudaDeviceGetAttribute(&nd.sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) { nd.error = e; return; }
        void *ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
        if (e != cudaSuccess) { nd.error = e; return; }
        nd.scratch = ptr;
    });
    *out = &nd;
    return nd.error;
}

dualmv_status run_f32_noalloc(int64_t M, int64_t N, const float *A, int64_t lda,
                              const float *p, const float *r, float *q, float *s,
                              cudaStream_t stream) {
    using T = float;
    using Acc = float;
    dualmv_status st = validate(M, N, A, lda, 0, p, 0, r, 0, q, 0, s, 0, 1);
    if (st != DUALMV_SUCCESS) return st;
    if (M == 0 || N == 0) {
        cudaError_t e = zero_fill(q, M, M, 1, stream);
        if (e == cudaSuccess) e = zero_fill(s, N, N, 1, stream);
        return e == cudaSuccess ? DUALMV_SUCCESS : cuda_fail(e);
    }
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e);
    NoallocDevice *nd = nullptr;
    e = noalloc_setup(dev, &nd);
    if (e != cudaSuccess) return cuda_fail(e);

    const int64_t es = sizeof(T);
    bool tma = g_path != DUALMV_PATH_DIRECT &&
               (reinterpret_cast<uintptr_t>(A) % 16 == 0) && ((lda * es) % 16 == 0) &&
               M < INT32_MAX && N < INT32_MAX;
    CUtensorMap map;
    std::memset(&map, 0, sizeof map);
    if (tma) tma = encode_a<T>(&map, A, M, N, lda, M * lda, 1, kBandCols, kWarps * kRpw4, false);
    dualmv_plan_t pl;
    st = make_plan(M, N, 1, es, sizeof(Acc),
                   (int64_t)nd->sms * (tma ? 1 : kDirectCtasPerSm),
                   tma ? Kind::kTma : Kind::kDirect, &pl);
    if (st != DUALMV_SUCCESS) return st;
    if (pl.workspace_bytes > kNoallocScratchBytes) return DUALMV_ERR_TOO_LARGE;

    // Every scratch word the combine kernel reads is written earlier in the
    // same call, so nothing needs clearing between calls.
    Params prm;
    std::memset(&prm, 0, sizeof prm);
    prm.ph_n = 1;
    prm.A = A; prm.lda = lda; prm.strideA = M * lda;
    prm.p = p; prm.strideP = N;
    prm.r = r; prm.strideR = M;
    prm.q = q; prm.strideQ = M;
    prm.s = s; prm.strideS = N;
    prm.M = M; prm.N = N; prm.batch = 1;
    prm.outputs = dmv::kOutBoth;
    prm.u1 = prm.v1 = prm.u2 = prm.v2 = nullptr;
    prm.a_out = nullptr;
    prm.lda_out = 0;
    prm.band_cols = pl.band_cols;
    prm.bands = pl.bands; prm.stripes = pl.stripes; prm.tiles = pl.tiles;
    prm.grid = pl.grid; prm.max_seg = pl.max_segments;
    const int64_t q_ws_bytes = pl.bands > 1 ? pl.bands * M * (int64_t)sizeof(Acc) : 0;
    prm.q_ws = pl.bands > 1 ? nd->scratch : nullptr;
    prm.s_ws = static_cast<unsigned char *>(nd->scratch) + ((q_ws_bytes + 255) / 256) * 256;

    e = tma ? launch_stream<T, true, false>(map, prm, pl, dev, stream)
            : launch_stream<T, false, false>(map, prm, pl, dev, stream);
    if (e == cudaSuccess) e = launch_combine<Acc>(prm, stream);
    return e == cudaSuccess ? DUALMV_SUCCESS : cuda_fail(e);
}

}  // namespace

// ================================================================ C ABI ===

// One single-sided pass: DUALMV_PASS_ROWS (out = A x) or DUALMV_PASS_COLS
// (out = A^T x), through the same tuner loop.
template <typename T>
dualmv_status tune_pass(int64_t M, int64_t N, const T *A, int64_t lda, int32_t pass,
                        const T *x, T *out, const dualmv_tune_config_t *cfg,
                        dualmv_tune_result_t *res, dualmv_stream_t stream) {
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (pass == DUALMV_PASS_ROWS)
        return tune_run<T, T>(M, N, 1, A, lda, 0, x, 0, nullptr, 0, out, 0, nullptr, 0, cfg, res,
                              st, dmv::kOutQ);
    if (pass == DUALMV_PASS_COLS)
        return tune_run<T, T>(M, N, 1, A, lda, 0, nullptr, 0, x, 0, nullptr, 0, out, 0, cfg, res,
                              st, dmv::kOutS);
    return DUALMV_ERR_INVALID_VALUE;
}

extern "C" {

dualmv_status dualmv_f32(int64_t M, int64_t N, const float *A, int64_t lda, const float *p,
                         const float *r, float *q, float *s, dualmv_stream_t stream) {
    return run<float, float>(M, N, A, lda, 0, p, 0, r, 0, q, 0, s, 0, 1,
                             reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                         const double *p, const double *r, double *q, double *s,
                         dualmv_stream_t stream) {
    return run<double, double>(M, N, A, lda, 0, p, 0, r, 0, q, 0, s, 0, 1,
                               reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_i32(int64_t M, int64_t N, const int32_t *A, int64_t lda,
                         const int32_t *p, const int32_t *r, int64_t *q, int64_t *s,
                         dualmv_stream_t stream) {
    return run<int32_t, int64_t>(M, N, A, lda, 0, p, 0, r, 0, q, 0, s, 0, 1,
                                 reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_f32_strided_batched(int64_t M, int64_t N, const float *A, int64_t lda,
                                         int64_t strideA, const float *p, int64_t strideP,
                                         const float *r, int64_t strideR, float *q,
                                         int64_t strideQ, float *s, int64_t strideS,
                                         int64_t batch, dualmv_stream_t stream) {
    return run<float, float>(M, N, A, lda, strideA, p, strideP, r, strideR, q, strideQ, s,
                             strideS, batch, reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_f64_strided_batched(int64_t M, int64_t N, const double *A, int64_t lda,
                                         int64_t strideA, const double *p, int64_t strideP,
                                         const double *r, int64_t strideR, double *q,
                                         int64_t strideQ, double *s, int64_t strideS,
                                         int64_t batch, dualmv_stream_t stream) {
    return run<double, double>(M, N, A, lda, strideA, p, strideP, r, strideR, q, strideQ, s,
                               strideS, batch, reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_i32_strided_batched(int64_t M, int64_t N, const int32_t *A,
                                         int64_t lda, int64_t strideA, const int32_t *p,
                                         int64_t strideP, const int32_t *r, int64_t strideR,
                                         int64_t *q, int64_t strideQ, int64_t *s,
                                         int64_t strideS, int64_t batch,
                                         dualmv_stream_t stream) {
    return run<int32_t, int64_t>(M, N, A, lda, strideA, p, strideP, r, strideR, q, strideQ,
                                 s, strideS, batch, reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_gesummv_f32(int64_t M, int64_t N, float alpha, const float *A,
                                 int64_t lda, float beta, const float *B, int64_t ldb,
                                 const float *x, float *y, dualmv_stream_t stream) {
    return gesummv_run<float>(M, N, alpha, A, lda, beta, B, ldb, x, y,
                              reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_gesummv_f64(int64_t M, int64_t N, double alpha, const double *A,
                                 int64_t lda, double beta, const double *B, int64_t ldb,
                                 const double *x, double *y, dualmv_stream_t stream) {
    return gesummv_run<double>(M, N, alpha, A, lda, beta, B, ldb, x, y,
                               reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_atax_f32(int64_t M, int64_t N, const float *A, int64_t lda,
                              const float *x, float *y, dualmv_stream_t stream) {
    return atax_run<float>(M, N, A, lda, x, y, reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_atax_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                              const double *x, double *y, dualmv_stream_t stream) {
    return atax_run<double>(M, N, A, lda, x, y, reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_gemver_f32(int64_t M, int64_t N, float alpha, float beta, float *A,
                                int64_t lda, int update_A, const float *u1, const float *v1,
                                const float *u2, const float *v2, float *w, float *x,
                                const float *y, const float *z, dualmv_stream_t stream) {
    return gemver_run<float>(M, N, alpha, beta, A, lda, update_A, u1, v1, u2, v2, w, x, y, z,
                             reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_gemver_f64(int64_t M, int64_t N, double alpha, double beta, double *A,
                                int64_t lda, int update_A, const double *u1, const double *v1,
                                const double *u2, const double *v2, double *w, double *x,
                                const double *y, const double *z, dualmv_stream_t stream) {
    return gemver_run<double>(M, N, alpha, beta, A, lda, update_A, u1, v1, u2, v2, w, x, y, z,
                              reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_f32_noalloc(int64_t M, int64_t N, const float *A, int64_t lda,
                                 const float *p, const float *r, float *q, float *s,
                                 dualmv_stream_t stream) {
    return run_f32_noalloc(M, N, A, lda, p, r, q, s, reinterpret_cast<cudaStream_t>(stream));
}

int64_t dualmv_f32_noalloc_scratch_bytes(void) { return kNoallocScratchBytes; }

const char *dualmv_status_string(dualmv_status status) {
    switch (status) {
    case DUALMV_SUCCESS: return "success";
    case DUALMV_ERR_INVALID_VALUE: return "invalid argument";
    case DUALMV_ERR_ALLOC: return "workspace allocation failed";
    case DUALMV_ERR_LAUNCH: return "CUDA launch or runtime error";
    case DUALMV_ERR_TIMEOUT: return "a device-side bounded wait timed out";
    case DUALMV_ERR_UNSUPPORTED: return "unsupported configuration";
    case DUALMV_ERR_TOO_LARGE:
        return "problem needs more scratch than the no-allocation entry point holds";
    }
    return "unknown status";
}

int dualmv_last_cuda_error(void) { return g_last_cuda_error; }

dualmv_status dualmv_device_fault(dualmv_stream_t stream) {
    cudaError_t e = cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e);
    unsigned int word = 0, zero = 0;
    e = cudaMemcpyFromSymbol(&word, dmv::g_fault_word, sizeof word);
    if (e != cudaSuccess) return cuda_fail(e);
    if (word != 0) {
        e = cudaMemcpyToSymbol(dmv::g_fault_word, &zero, sizeof zero);
        if (e != cudaSuccess) return cuda_fail(e);
        return DUALMV_ERR_TIMEOUT;
    }
    return DUALMV_SUCCESS;
}

dualmv_status dualmv_read_probe(const void *buf, int64_t bytes, uint32_t *out,
                                dualmv_stream_t stream) {
    if (bytes < 0 || bytes % 16 != 0 || reinterpret_cast<uintptr_t>(buf) % 16 != 0 ||
        out == nullptr || (bytes > 0 && buf == nullptr))
        return DUALMV_ERR_INVALID_VALUE;
    if (bytes == 0) return DUALMV_SUCCESS;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e);
    DeviceState *ds = nullptr;
    e = device_state(dev, &ds);
    if (e != cudaSuccess) return cuda_fail(e);
    // Four blocks of 512 threads fill an SM's 2048 thread slots.
    dmv::read_probe_kernel<<<(unsigned)(4 * ds->sms), dmv::kProbeThreads, 0,
                             reinterpret_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint4 *>(buf), bytes / 16, out);
    e = cudaGetLastError();
    return e == cudaSuccess ? DUALMV_SUCCESS : cuda_fail(e);
}

dualmv_status dualmv_selftest_wait_timeout(int cluster_scope, int32_t *waited,
                                          dualmv_stream_t stream) {
    if (waited == nullptr) return DUALMV_ERR_INVALID_VALUE;
    dmv::wait_selftest_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        cluster_scope != 0 ? 1 : 0, waited);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? DUALMV_SUCCESS : cuda_fail(e);
}

dualmv_status dualmv_pool_usage(int device, int64_t *reserved_bytes, int64_t *used_high_bytes,
                                int reset_high) {
    if (device < 0 || device >= kMaxDevices || reserved_bytes == nullptr ||
        used_high_bytes == nullptr)
        return DUALMV_ERR_INVALID_VALUE;
    *reserved_bytes = 0;
    *used_high_bytes = 0;
    DeviceState *ds = nullptr;
    cudaError_t e = device_state(device, &ds);
    if (e != cudaSuccess) return cuda_fail(e);
    uint64_t reserved = 0, high = 0;
    e = cudaMemPoolGetAttribute(ds->pool, cudaMemPoolAttrReservedMemCurrent, &reserved);
    if (e == cudaSuccess)
        e = cudaMemPoolGetAttribute(ds->pool, cudaMemPoolAttrUsedMemHigh, &high);
    if (e == cudaSuccess && reset_high) {
        uint64_t zero = 0;  // resets the high-water mark to the current use
        e = cudaMemPoolSetAttribute(ds->pool, cudaMemPoolAttrUsedMemHigh, &zero);
    }
    if (e != cudaSuccess) return cuda_fail(e);
    *reserved_bytes = (int64_t)reserved;
    *used_high_bytes = (int64_t)high;
    return DUALMV_SUCCESS;
}

void dualmv_record_kernel_events(void *start, void *stop) {
    g_kernel_ev_start = static_cast<cudaEvent_t>(start);
    g_kernel_ev_stop = static_cast<cudaEvent_t>(stop);
}

int dualmv_gemver_set_onthefly(int onthefly) {
    const int old = g_gemver_onthefly;
    g_gemver_onthefly = onthefly ? 1 : 0;
    return old;
}

int dualmv_atax_set_two_pass(int two_pass) {
    const int old = g_atax_two_pass;
    g_atax_two_pass = two_pass ? 1 : 0;
    return old;
}

int dualmv_set_path(int path) {
    if (path != DUALMV_PATH_AUTO && path != DUALMV_PATH_TMA && path != DUALMV_PATH_DIRECT &&
        path != DUALMV_PATH_TMA_NATIVE_F64)
        return -1;
    const int old = g_path;
    g_path = path;
    return old;
}

dualmv_status dualmv_plan(int64_t M, int64_t N, int64_t batch, int64_t elem_bytes,
                          int64_t acc_bytes, int64_t num_sms, dualmv_plan_t *out) {
    return make_plan(M, N, batch, elem_bytes, acc_bytes, num_sms,
                     elem_bytes == 8 ? Kind::kF64e : Kind::kTma, out);
}

int32_t dualmv_variant_count(int32_t dtype) {
    const std::vector<Variant> *tab = variant_table(dtype);
    return tab ? (int32_t)tab->size() : -1;
}

dualmv_status dualmv_variant_info(int32_t dtype, int32_t index, dualmv_variant_t *out) {
    const std::vector<Variant> *tab = variant_table(dtype);
    if (tab == nullptr || out == nullptr || index < 0 || index >= (int32_t)tab->size())
        return DUALMV_ERR_INVALID_VALUE;
    *out = (*tab)[index].info;
    return DUALMV_SUCCESS;
}

int32_t dualmv_set_variant(int32_t dtype, int32_t index) {
    const std::vector<Variant> *tab = variant_table(dtype);
    if (tab == nullptr || index < -1 || index >= (int32_t)tab->size()) return -2;
    return g_forced_variant[dtype].exchange(index);
}

int32_t dualmv_tuned_variant(int32_t dtype, int64_t M, int64_t N, int64_t lda) {
    return tuned_lookup(dtype, M, N, lda);
}

int32_t dualmv_tuned_variant_batched(int32_t dtype, int64_t M, int64_t N, int64_t lda,
                                     int64_t batch) {
    return tuned_lookup(dtype, M, N, lda, batch > 1 ? batch : 1);
}

int32_t dualmv_tuned_variant_pass(int32_t dtype, int64_t M, int64_t N, int64_t lda, int32_t pass) {
    if (pass != DUALMV_PASS_ROWS && pass != DUALMV_PASS_COLS) return -1;
    return tuned_lookup(dtype, M, N, lda, 1,
                        pass == DUALMV_PASS_ROWS ? (uint32_t)dmv::kOutQ : (uint32_t)dmv::kOutS);
}

int32_t dualmv_last_variant(void) { return g_last_variant; }

int32_t dualmv_last_kernel(void) { return g_last_kernel; }

int32_t dualmv_atax_last_path(void) { return g_last_atax_path; }

int32_t dualmv_gemver_last_path(void) { return g_last_gemver_path; }

void dualmv_tune_clear(void) {
    std::lock_guard<std::mutex> lk(g_tuned_mu);
    g_tuned.clear();
    g_tuned_count.store(0, std::memory_order_release);
}

dualmv_status dualmv_trimmed_mean(const double *t, int64_t R, int64_t k, double *out) {
    if (t == nullptr || out == nullptr || R < 0) return DUALMV_ERR_INVALID_VALUE;
    std::vector<double> v(t, t + R);
    return trimmed_mean_of(std::move(v), k, out) ? DUALMV_SUCCESS : DUALMV_ERR_INVALID_VALUE;
}

dualmv_status dualmv_tune_f32(int64_t M, int64_t N, const float *A, int64_t lda, const float *p,
                              const float *r, float *q, float *s,
                              const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
                              dualmv_stream_t stream) {
    return tune_run<float, float>(M, N, 1, A, lda, 0, p, 0, r, 0, q, 0, s, 0, cfg, res,
                                  reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_tune_pass_f32(int64_t M, int64_t N, const float *A, int64_t lda,
                                   int32_t pass, const float *x, float *out,
                                   const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
                                   dualmv_stream_t stream) {
    return tune_pass<float>(M, N, A, lda, pass, x, out, cfg, res, stream);
}

dualmv_status dualmv_tune_pass_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                                   int32_t pass, const double *x, double *out,
                                   const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
                                   dualmv_stream_t stream) {
    return tune_pass<double>(M, N, A, lda, pass, x, out, cfg, res, stream);
}

dualmv_status dualmv_tune_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                              const double *p, const double *r, double *q, double *s,
                              const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
                              dualmv_stream_t stream) {
    return tune_run<double, double>(M, N, 1, A, lda, 0, p, 0, r, 0, q, 0, s, 0, cfg, res,
                                    reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_tune_i32(int64_t M, int64_t N, const int32_t *A, int64_t lda,
                              const int32_t *p, const int32_t *r, int64_t *q, int64_t *s,
                              const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
                              dualmv_stream_t stream) {
    return tune_run<int32_t, int64_t>(M, N, 1, A, lda, 0, p, 0, r, 0, q, 0, s, 0, cfg, res,
                                      reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_tune_f32_strided_batched(
    int64_t M, int64_t N, const float *A, int64_t lda, int64_t strideA, const float *p,
    int64_t strideP, const float *r, int64_t strideR, float *q, int64_t strideQ, float *s,
    int64_t strideS, int64_t batch, const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
    dualmv_stream_t stream) {
    return tune_run<float, float>(M, N, batch, A, lda, strideA, p, strideP, r, strideR, q,
                                  strideQ, s, strideS, cfg, res,
                                  reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_tune_f64_strided_batched(
    int64_t M, int64_t N, const double *A, int64_t lda, int64_t strideA, const double *p,
    int64_t strideP, const double *r, int64_t strideR, double *q, int64_t strideQ, double *s,
    int64_t strideS, int64_t batch, const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
    dualmv_stream_t stream) {
    return tune_run<double, double>(M, N, batch, A, lda, strideA, p, strideP, r, strideR, q,
                                    strideQ, s, strideS, cfg, res,
                                    reinterpret_cast<cudaStream_t>(stream));
}

dualmv_status dualmv_tune_i32_strided_batched(
    int64_t M, int64_t N, const int32_t *A, int64_t lda, int64_t strideA, const int32_t *p,
    int64_t strideP, const int32_t *r, int64_t strideR, int64_t *q, int64_t strideQ, int64_t *s,
    int64_t strideS, int64_t batch, const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
    dualmv_stream_t stream) {
    return tune_run<int32_t, int64_t>(M, N, batch, A, lda, strideA, p, strideP, r, strideR, q,
                                      strideQ, s, strideS, cfg, res,
                                      reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"
