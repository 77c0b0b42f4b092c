// Device code of the fused dual matrix-vector product (BICG, Tables 1-2):
//     q = A p,  s = A^T r,  one pass over a row-major A.
//
// Work decomposition
//   A (one problem, or each problem of a strided batch) is cut into column
//   bands of kBandCols = 256 columns and row stripes of BM rows; a tile is
//   one stripe of one band.  Tiles are numbered band-major
//   (problem, band, stripe) and CTA c of a persistent grid of G CTAs owns the
//   contiguous range [c*T/G, (c+1)*T/G), so every CTA streams the same number
//   of tiles to within one.
//
// Inside a CTA (TMA path)
//   one producer warp issues one 2-D/3-D TMA box (256 columns x BM rows) per
//   tile into a ring of kStages shared-memory buffers, tracked by mbarriers;
//   W consumer warps each take RPW consecutive rows of every tile.  Lane l
//   holds 8 columns of the band (two or four 16-byte vectors) and the
//   matching 8 entries of p in registers.
//     * q: each row's 8-term partial is reduced across the warp with a
//       reduce-scatter butterfly (RPW rows share log2 steps), which yields
//       the complete band partial of that row; it goes to q directly when
//       the matrix is one band wide, else to the band-partial workspace.
//     * s: each lane accumulates its 8 columns over the rows of the tile,
//       then over a group of tiles, then over the segment (the run of
//       stripes of one band that this CTA owns).  At a segment end the W
//       warps' partials are summed in warp order through shared memory and
//       written to s (segment covers the whole band) or to the segment
//       workspace.
//   A second kernel adds band partials (q) in ascending band order and
//   segment partials (s) in ascending CTA order.  Every sum has a fixed
//   order, so floating-point results are identical run to run.
//
// Plain-load path: the same schedule and arithmetic, but each consumer warp
// reads its rows straight from global memory with bounds checks.  It serves
// inputs the TMA unit cannot address (unaligned base or leading dimension).
//
// Every wait on an mbarrier is bounded in time.  A warp that gives up sets
// the device fault word and stops waiting, but keeps the same control flow
// (so no named barrier is left short of a participant) and the producer
// still waits, bounded, for the copies it issued before the CTA exits.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

namespace dmv {

// What a stream kernel computes: the row sums q = A p, the column sums
// s = A^T r, or both (the dual product).  The single-sided modes serve the
// operations built from one matrix-vector product (ATAX, GESUMMV).
constexpr int kOutQ = 1;
constexpr int kOutS = 2;
constexpr int kOutBoth = kOutQ | kOutS;

constexpr int kBandCols = 256;          // columns per band = TMA box width
constexpr int kLaneCols = kBandCols / 32;  // columns per lane = 8
constexpr int kGroupTiles = 16;         // tiles summed before the segment sum
constexpr unsigned long long kWaitTimeoutNs = 2000000000ull;  // 2 s

// Device fault word: bit 0 = a bounded wait timed out.  Read and cleared by
// the host through dualmv_device_fault().
__device__ unsigned int g_fault_word;

template <typename T> struct Traits;
template <> struct Traits<float> {
    using Acc = float;
    using Vec = float4;
    static constexpr int kVecElems = 4;
};
template <> struct Traits<double> {
    using Acc = double;
    using Vec = double2;
    static constexpr int kVecElems = 2;
};
// int32 inputs: exact 64-bit products, sums modulo 2^64 (unsigned, so the
// wrap-around is defined), reinterpreted as int64 on output.
template <> struct Traits<int32_t> {
    using Acc = unsigned long long;
    using Vec = int4;
    static constexpr int kVecElems = 4;
};

// ------------------------------------------------------------ arithmetic --

__device__ __forceinline__ float mul_acc(float a, float x, float acc) {
    return fmaf(a, x, acc);
}
__device__ __forceinline__ double mul_acc(double a, double x, double acc) {
    return fma(a, x, acc);
}
__device__ __forceinline__ unsigned long long mul_acc(int32_t a, int32_t x,
                                                      unsigned long long acc) {
    return acc + (unsigned long long)((long long)a * (long long)x);
}

template <typename Acc>
__device__ __forceinline__ Acc shfl_xor(Acc v, int off) {
    return __shfl_xor_sync(0xffffffffu, v, off);
}

// Element e of a 16-byte vector.
__device__ __forceinline__ float vget(const float4 &v, int e) {
    return e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w;
}
__device__ __forceinline__ double vget(const double2 &v, int e) {
    return e == 0 ? v.x : v.y;
}
__device__ __forceinline__ int32_t vget(const int4 &v, int e) {
    return e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w;
}

// Band-relative column of element e of vector v held by `lane`.
template <typename T>
__device__ __forceinline__ int lane_col(int v, int lane, int e) {
    return (v * 32 + lane) * Traits<T>::kVecElems + e;
}

// Reduce-scatter butterfly over RPW row partials held by every lane.  On
// return, v[0] of lane l is the full warp sum of row
// (l >> (5 - log2 RPW)) & (RPW - 1).  Step k exchanges half of the
// remaining values across lane bit (4 - k); the remaining bits are summed
// with plain xor steps.  Fixed order, so deterministic.
template <int RPW, typename Acc>
__device__ __forceinline__ void warp_rows_reduce(Acc (&v)[RPW], int lane) {
    int off = 16;
#pragma unroll
    for (int h = RPW / 2; h >= 1; h /= 2) {
        const bool upper = (lane & off) != 0;
#pragma unroll
        for (int k = 0; k < h; ++k) {
            const Acc send = upper ? v[k] : v[k + h];
            const Acc keep = upper ? v[k + h] : v[k];
            v[k] = keep + shfl_xor(send, off);
        }
        off >>= 1;
    }
#pragma unroll
    for (; off >= 1; off >>= 1) v[0] = v[0] + shfl_xor(v[0], off);
}

template <int RPW>
__device__ __forceinline__ int butterfly_row(int lane) {
    constexpr int L = RPW == 1 ? 0 : RPW == 2 ? 1 : RPW == 4 ? 2 : RPW == 8 ? 3 : 4;
    return (lane >> (5 - L)) & (RPW - 1);
}
template <int RPW>
__device__ __forceinline__ bool butterfly_writer(int lane) {
    constexpr int L = RPW == 1 ? 0 : RPW == 2 ? 1 : RPW == 4 ? 2 : RPW == 8 ? 3 : 4;
    return (lane & ((32 >> L) - 1)) == 0;
}

// --------------------------------------------------- mbarrier and TMA ----

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Bytes to skip so that the dynamic shared memory base is kAlign-aligned.
// Callers offset the __shared__ array itself by this amount (pointer
// arithmetic keeps the shared address space visible to the compiler, so
// tile reads stay shared-memory loads rather than generic ones).
template <int kAlign>
__device__ __forceinline__ uint32_t shared_align_pad(const void *base) {
    return (uint32_t)(kAlign - (smem_u32(base) & (kAlign - 1))) & (uint32_t)(kAlign - 1);
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile(
        "{\n\t.reg .b64 st;\n\t"
        "mbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(bar)
        : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile(
        "{\n\t.reg .b64 st;\n\t"
        "mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(bar),
        "r"(bytes)
        : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Slow path of mbar_wait_bounded: keeps polling for at most kWaitTimeoutNs,
// then sets the device fault word and returns false.
__device__ __forceinline__ bool mbar_wait_slow(uint32_t bar, uint32_t parity) {
    const unsigned long long t0 = global_ns();
    for (;;) {
        for (int i = 0; i < 64; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (global_ns() - t0 > kWaitTimeoutNs) {
            atomicOr(&g_fault_word, 1u);
            return false;
        }
    }
}

// Wait for the phase of `bar` with parity `parity`, bounded in time.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    return mbar_wait_slow(bar, parity);
}

__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map,
                                            int x, int y, uint32_t bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(pol)
        : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map,
                                            int x, int y, int z, uint32_t bar,
                                            uint64_t pol) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
        ".L2::cache_hint [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar),
        "l"(pol)
        : "memory");
}

__device__ __forceinline__ void named_barrier(int id, int threads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

__device__ __forceinline__ void pdl_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ------------------------------------------------------------ parameters --

struct Params {
    const void *A;
    int64_t lda, strideA;
    const void *p;
    int64_t strideP;
    const void *r;
    int64_t strideR;
    void *q;
    int64_t strideQ;
    void *s;
    int64_t strideS;
    int64_t M, N, batch;
    // GEMVER's rank-2 update, applied to every element as it is streamed:
    // A_hat = A + u1 v1^T + u2 v2^T (u1, u2 of length M, v1, v2 of length
    // N); with a_out set, A_hat is also written there (row stride lda_out).
    const void *u1, *v1, *u2, *v2;
    void *a_out;
    int64_t lda_out;
    uint32_t outputs;   // kOutQ | kOutS: which of q and s this call computes
    int64_t band_cols;  // columns per band (the stream kernel's tile width)
    int64_t bands, stripes, tiles, grid, max_seg;
    void *q_ws;  // [batch][bands][M] band partials of q (bands > 1 only)
    void *s_ws;  // [grid][max_seg][kBandCols] segment partials of s
    // Rows whose stride (or base) is not 16-byte aligned, read through tensor
    // maps per row phase (dualmv_stream_phased_kernel): row r is in phase
    // r % ph_n, and its columns start at element ph_off[phase] of its box
    // row.  ph_n = 1 and zeros otherwise.
    int32_t ph_n;
    int32_t ph_off[4];
    // Late wait: a single-sided pass launched as a programmatic dependent of
    // a kernel that triggers its dependents only after its own wait, so that
    // every grid before that kernel has completed when this one starts.
    // That kernel touches none of this pass's memory, so the pass reads and
    // writes without waiting, and waits for that kernel's grid only before
    // it exits: its completion still implies that kernel's.  GEMVER's
    // columns pass runs this way beside the u . y dot-product kernel, and
    // GESUMMV's pass over B after its pass over A.  A late-wait pass lets
    // its own dependents launch at its start, so no late-wait pass may
    // follow it.
    int32_t pdl_late;
};

// Phased tensor maps: two per phase, over the same rows: m[2 ph] with
// 256-column boxes, m[2 ph + 1] with 16-byte boxes (the columns that the
// phase's offset pushes past the band's box).
constexpr int kMaxPhases = 4;
struct TmapSet {
    CUtensorMap m[2 * kMaxPhases];
};

// First tile of CTA c, and the CTA that owns tile t (inverse of the split).
__host__ __device__ __forceinline__ int64_t cta_first_tile(int64_t c, int64_t T,
                                                           int64_t G) {
    return (c * T) / G;
}
__host__ __device__ __forceinline__ int64_t cta_of_tile(int64_t t, int64_t T,
                                                        int64_t G) {
    return ((t + 1) * G - 1) / T;
}

// Dynamic shared memory of the stream kernel, the single definition used by
// both the kernel (offsets) and the host (launch size).  TMA path: a
// 1024-byte-aligned ring of STAGES tiles, the warp scratch for the s flush,
// then the full/empty mbarriers.  Plain-load path: the scratch only.
// Coordinates of a tile in band-major order, advanced one tile at a time so
// that the per-tile loop does no 64-bit division.
struct TileCursor {
    int64_t g;       // global band index: b * bands + band
    int64_t b;       // problem
    int64_t band;    // band within the problem
    int64_t stripe;  // stripe within the band
    __device__ __forceinline__ void init(int64_t t, int64_t S, int64_t bands) {
        g = t / S;
        stripe = t - g * S;
        b = g / bands;
        band = g - b * bands;
    }
    __device__ __forceinline__ void advance(int64_t S, int64_t bands) {
        if (++stripe == S) {
            stripe = 0;
            ++g;
            if (++band == bands) {
                band = 0;
                ++b;
            }
        }
    }
    // The tile before (for a CTA that walks its range backwards).
    __device__ __forceinline__ void retreat(int64_t S, int64_t bands) {
        if (stripe-- == 0) {
            stripe = S - 1;
            --g;
            if (band-- == 0) {
                band = bands - 1;
                --b;
            }
        }
    }
};

// The same in 32 bits, for kernels whose launch guarantees fewer than 2^31
// tiles (the double-float fp64 kernel, where the registers it saves pay).
struct TileCursor32 {
    int g, b, band, stripe;
    __device__ __forceinline__ void init(int t, int S, int bands) {
        g = t / S;
        stripe = t - g * S;
        b = g / bands;
        band = g - b * bands;
    }
    __device__ __forceinline__ void advance(int S, int bands) {
        if (++stripe == S) {
            stripe = 0;
            ++g;
            if (++band == bands) {
                band = 0;
                ++b;
            }
        }
    }
    __device__ __forceinline__ void retreat(int S, int bands) {
        if (stripe-- == 0) {
            stripe = S - 1;
            --g;
            if (band-- == 0) {
                band = bands - 1;
                --b;
            }
        }
    }
};

template <typename T, int W, int RPW, int STAGES, bool kTma, int NPH = 0>
struct SmemLayout {
    using Acc = typename Traits<T>::Acc;
    // NPH > 0 (phased maps): per phase, its W * RPW / NPH rows of the band's
    // box (1 KiB a row for 4-byte elements), then their 16 bytes each from
    // the small box, padded to 128 bytes so that every copy lands 128-byte
    // aligned.  kTileTx is what a tile's copies deliver, kTileBytes its slot.
    static constexpr int kRowBytes = kBandCols * (int)sizeof(T);
    static constexpr int kPhaseRows = NPH > 0 ? W * RPW / NPH : W * RPW;
    static constexpr int kPhaseBytes =
        kPhaseRows * kRowBytes + (NPH > 0 ? (kPhaseRows * 16 + 127) / 128 * 128 : 0);
    static constexpr int kTileBytes = (NPH > 0 ? NPH : 1) * kPhaseBytes;
    static constexpr int kTileTx = W * RPW * (kRowBytes + (NPH > 0 ? 16 : 0));
    static constexpr int kAlign = kTma ? 1024 : 16;
    static constexpr int kRing = kTma ? STAGES * kTileBytes : 0;
    static constexpr int kScratch = W * kBandCols * (int)sizeof(Acc);
    static constexpr int kBars = kTma ? 2 * STAGES * 8 : 0;
    // kAlign bytes of slack let the kernel round the dynamic base up.
    static constexpr int kTotal = kAlign + kRing + kScratch + kBars;
};

// ------------------------------------------------------------ main kernel --
//
// Template: element type T, W consumer warps, RPW rows per warp per tile,
// STAGES ring depth, kTma = TMA producer (else plain loads), kBatched3d =
// 3-D tensor map (batch as the outer coordinate).
// The plain-load path keeps its loads in registers and hides their latency
// with warps.  Its int32 form (64-bit sums) would otherwise take 168
// registers and one CTA per SM; it asks for two (128 registers), as the
// float forms get by themselves.
// The kernel body, shared by dualmv_stream_kernel (one tensor map, NPH = 0)
// and dualmv_stream_phased_kernel (NPH phase maps, tmaps[0 .. NPH - 1]).
template <typename T, int W, int RPW, int STAGES, bool kTma, bool kBatched3d, int kOut,
          bool kRank2, int NPH, bool kRev = false>
__device__ __forceinline__ void stream_body(const CUtensorMap *tmaps, const Params &prm) {
    using Acc = typename Traits<T>::Acc;
    static_assert(!kRank2 || !std::is_same<T, int32_t>::value, "rank-2 update: floats only");
    // kRev: each CTA walks its tile range backwards (last tile first), so a
    // pass that follows another over the same A starts on the tiles that
    // pass read last, which may still be in L2.  Rows-only passes only.
    static_assert(!kRev || kOut == kOutQ, "backward walk: rows-only passes");
    constexpr bool kQ = (kOut & kOutQ) != 0;  // row sums q = A p
    constexpr bool kS = (kOut & kOutS) != 0;  // column sums s = A^T r
    // Integer sums are exact modulo 2^64 in any order, so the int32 path adds
    // its band and segment partials straight into q and s with atomics (the
    // result is the same bits on every run) and needs no workspace and no
    // combine kernel.  q and s are zeroed by a preceding kernel, whose
    // completion the consumers await (programmatic dependent launch) before
    // their first write.
    constexpr bool kAtomicOut = std::is_same<T, int32_t>::value;
    using Vec = typename Traits<T>::Vec;
    constexpr int VE = Traits<T>::kVecElems;
    constexpr int VPL = kLaneCols / VE;  // 16-byte vectors per lane per row
    constexpr int BM = W * RPW;
    using L = SmemLayout<T, W, RPW, STAGES, kTma, NPH>;
    constexpr int ROW_BYTES = L::kRowBytes;  // smem pitch of a tile row (the band's box)
    constexpr int TILE_BYTES = L::kTileBytes;
    static_assert(NPH == 0 || (kTma && !kBatched3d && !kRank2 && RPW % NPH == 0 &&
                               BM % NPH == 0 && NPH <= kMaxPhases),
                  "phased maps: one unbatched problem, each warp's rows in whole phase groups");
    // Phased maps: per phase, the band's box (BM / NPH rows of ROW_BYTES) and
    // then the small box (BM / NPH rows of 16 bytes).
    constexpr int PH = NPH > 0 ? NPH : 1;
    constexpr int PHASE_ROWS = BM / PH;
    constexpr int PHASE_BYTES = L::kPhaseBytes;
    static_assert(PHASE_ROWS == L::kPhaseRows && PHASE_BYTES % 128 == 0,
                  "phased maps: every copy must land 128-byte aligned");

    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_raw + shared_align_pad<L::kAlign>(smem_raw);
    unsigned char *ring = smem;
    Acc *scratch = reinterpret_cast<Acc *>(smem + L::kRing);
    uint64_t *full_bar = reinterpret_cast<uint64_t *>(smem + L::kRing + L::kScratch);
    uint64_t *empty_bar = full_bar + STAGES;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t T_ = prm.tiles, G = prm.grid, S = prm.stripes;
    const int64_t c = blockIdx.x;
    const int64_t t0 = cta_first_tile(c, T_, G);
    const int64_t t1 = cta_first_tile(c + 1, T_, G);
    const int64_t ntiles = t1 - t0;
    const int64_t g_first = t0 / S;

    if constexpr (kTma) {
        if (threadIdx.x == 0) {
            for (int i = 0; i < STAGES; ++i) {
                mbar_init(smem_u32(&full_bar[i]), 1);
                mbar_init(smem_u32(&empty_bar[i]), W);
            }
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        __syncthreads();
    }
    // Dependent grids (the combine kernel) may start launching now; they
    // wait for this grid's completion before reading anything it writes.
    pdl_launch_dependents();

    // ------------------------------------------------------ producer ----
    if constexpr (kTma) {
        if (warp == W) {
            if (lane == 0) {
                const uint64_t pol = policy_evict_first();
                bool ok = true;
                int64_t issued = 0;
                TileCursor cur;
                cur.init(kRev ? t1 - 1 : t0, S, prm.bands);
                int stage = 0;
                uint32_t phase = 0;  // parity of the ring pass, flips each pass
                for (int64_t k = 0; k < ntiles; ++k) {
                    // Before the second pass over the ring, wait until the
                    // consumers released the previous tile in this stage.
                    if (ok && k >= STAGES)
                        ok = mbar_wait_bounded(smem_u32(&empty_bar[stage]), phase ^ 1u);
                    if (!ok) break;
                    const uint32_t fb = smem_u32(&full_bar[stage]);
                    mbar_arrive_expect_tx(fb, L::kTileTx);
                    const uint32_t dst = smem_u32(ring + (size_t)stage * TILE_BYTES);
                    const int x = (int)(cur.band * kBandCols), y = (int)(cur.stripe * BM);
                    if constexpr (NPH > 0) {
                        // Per phase: the band's columns of its BM / NPH rows
                        // (shifted by the phase's offset) and the 16 bytes after.
#pragma unroll
                        for (int ph = 0; ph < NPH; ++ph) {
                            const uint32_t d = dst + (uint32_t)(ph * PHASE_BYTES);
                            tma_load_2d(d, &tmaps[2 * ph], x, y / NPH, fb, pol);
                            tma_load_2d(d + (uint32_t)(PHASE_ROWS * ROW_BYTES), &tmaps[2 * ph + 1],
                                        x + kBandCols, y / NPH, fb, pol);
                        }
                    } else if constexpr (kBatched3d) {
                        tma_load_3d(dst, &tmaps[0], x, y, (int)cur.b, fb, pol);
                    } else {
                        tma_load_2d(dst, &tmaps[0], x, y, fb, pol);
                    }
                    issued = k + 1;
                    if constexpr (kRev)
                        cur.retreat(S, prm.bands);
                    else
                        cur.advance(S, prm.bands);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                // Before the CTA exits, every copy it issued must have landed
                // (bounded): the last min(STAGES, ntiles) issued stages.
                for (int64_t k = issued > STAGES ? issued - STAGES : 0; k < issued; ++k) {
                    const int stage = (int)(k % STAGES);
                    mbar_wait_bounded(smem_u32(&full_bar[stage]),
                                      (uint32_t)(k / STAGES) & 1u);
                }
            }
            return;
        }
    }

    // ----------------------------------------------------- consumers ----
    const T *__restrict__ Ag = static_cast<const T *>(prm.A);
    const T *__restrict__ pg = static_cast<const T *>(prm.p);
    const T *__restrict__ rg = static_cast<const T *>(prm.r);
    const int nthreads_c = W * 32;

    T pv[kLaneCols];
    T v1v[kRank2 ? kLaneCols : 1], v2v[kRank2 ? kLaneCols : 1];  // GEMVER columns
    Acc grp[kLaneCols], seg[kLaneCols];
#pragma unroll
    for (int e = 0; e < kLaneCols; ++e) {
        pv[e] = T(0);
        grp[e] = Acc(0);
        seg[e] = Acc(0);
    }
    int ngrp = 0;
    int64_t seg_start_stripe = 0;
    bool ok = true;

    TileCursor cur;
    cur.init(kRev ? t1 - 1 : t0, S, prm.bands);
    // r for this warp's RPW rows of the next tile (lane i < RPW holds row
    // row0 + i), loaded one tile ahead so its latency hides behind a tile.
    T r_next = T(0), u1_next = T(0), u2_next = T(0);
    if constexpr (kS) {
        const int64_t row = cur.stripe * BM + (int64_t)warp * RPW + lane;
        if (lane < RPW && row < prm.M) r_next = rg[cur.b * prm.strideR + row];
    }
    if constexpr (kRank2) {
        const int64_t row = cur.stripe * BM + (int64_t)warp * RPW + lane;
        if (lane < RPW && row < prm.M) {
            u1_next = static_cast<const T *>(prm.u1)[row];
            u2_next = static_cast<const T *>(prm.u2)[row];
        }
    }
    int stage = 0;
    uint32_t phase = 0;
    if constexpr (kAtomicOut) pdl_wait();  // q and s zeroed before any add

    for (int64_t k = 0; k < ntiles; ++k) {
        const int64_t g = cur.g;
        const int64_t stripe = cur.stripe;
        const int64_t band = cur.band;
        const int64_t b = cur.b;
        const int64_t col0 = band * kBandCols;
        const int64_t row0 = stripe * BM + (int64_t)warp * RPW;
        const T rmine = r_next, u1mine = u1_next, u2mine = u2_next;
        if constexpr (kRev)
            cur.retreat(S, prm.bands);
        else
            cur.advance(S, prm.bands);
        if (kS && k + 1 < ntiles) {
            const int64_t row = cur.stripe * BM + (int64_t)warp * RPW + lane;
            r_next = (lane < RPW && row < prm.M) ? rg[cur.b * prm.strideR + row] : T(0);
        }
        if (kRank2 && k + 1 < ntiles) {
            const int64_t row = cur.stripe * BM + (int64_t)warp * RPW + lane;
            const bool in = lane < RPW && row < prm.M;
            u1_next = in ? static_cast<const T *>(prm.u1)[row] : T(0);
            u2_next = in ? static_cast<const T *>(prm.u2)[row] : T(0);
        }
        if (kRank2 && (k == 0 || stripe == 0)) {  // a new segment: v1, v2 of this band
#pragma unroll
            for (int v = 0; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) {
                    const int64_t col = col0 + lane_col<T>(v, lane, e);
                    v1v[v * VE + e] = col < prm.N ? static_cast<const T *>(prm.v1)[col] : T(0);
                    v2v[v * VE + e] = col < prm.N ? static_cast<const T *>(prm.v2)[col] : T(0);
                }
        }

        // A new segment: the CTA's first tile, or a band entered (at its
        // first stripe walking forwards, its last walking backwards).
        const bool seg_start = k == 0 || stripe == (kRev ? S - 1 : 0);
        if (seg_start) seg_start_stripe = stripe;
        if (kQ && seg_start) {  // a new segment: this band's p
            const T *pb = pg + b * prm.strideP;
#pragma unroll
            for (int v = 0; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) {
                    const int64_t col = col0 + lane_col<T>(v, lane, e);
                    pv[v * VE + e] = col < prm.N ? pb[col] : T(0);
                }
        }

        Acc qp[RPW];
        Acc tacc[kLaneCols];
#pragma unroll
        for (int e = 0; e < kLaneCols; ++e) tacc[e] = Acc(0);

        if constexpr (kTma) {
            if (ok) ok = mbar_wait_bounded(smem_u32(&full_bar[stage]), phase);
        }
        // One-map TMA tiles: the warp copies its rows of the stage into
        // registers and releases the stage before any arithmetic, so the
        // producer refills it while the warp computes.  (With the release
        // after the products the f32 16384^2 kernel ran at 0.99 of the
        // measured copy bandwidth; with it here, and four stages, 1.01-1.03.)
        constexpr bool kEarly = kTma && NPH == 0 && !kRank2;
        Vec tile[kEarly ? RPW : 1][VPL];
        if constexpr (kEarly) {
#pragma unroll
            for (int i = 0; i < RPW; ++i) {
                const Vec *rowp = reinterpret_cast<const Vec *>(
                    ring + (size_t)stage * TILE_BYTES + (size_t)(warp * RPW + i) * ROW_BYTES);
#pragma unroll
                for (int v = 0; v < VPL; ++v) tile[i][v] = rowp[v * 32 + lane];
            }
            // Every lane's reads of the stage come before lane 0's arrival
            // (the warp barrier orders them; the arrival releases them).
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&empty_bar[stage]));
        }
#pragma unroll
        for (int i = 0; i < RPW; ++i) {
            Vec a[VPL];
            if constexpr (kEarly) {
#pragma unroll
                for (int v = 0; v < VPL; ++v) a[v] = tile[i][v];
            } else if constexpr (NPH > 0) {
                // Tile row warp * RPW + i: phase i % NPH (RPW is a multiple of
                // NPH), row (warp * RPW + i) / NPH of that phase's box, its
                // columns from element ph_off of the box row.
                const int ph = i % PH;
                const int off = prm.ph_off[ph];
                // The box row (16-byte aligned); the row's element j is at box
                // position j + off, off < VE.
                const int prow = (warp * RPW + i) / PH;
                const unsigned char *phb = ring + (size_t)stage * TILE_BYTES + (size_t)ph * PHASE_BYTES;
                const Vec *boxrow = reinterpret_cast<const Vec *>(phb + (size_t)prow * ROW_BYTES);
                if (off == 0) {
#pragma unroll
                    for (int v = 0; v < VPL; ++v) a[v] = boxrow[v * 32 + lane];
                } else {
                    // Lane l's vector v is the tail of aligned vector v * 32 + l
                    // and the head of the next one (lane 31's last: the row's 16
                    // bytes of the small box).  Both are read as aligned 16-byte
                    // vectors (consecutive lanes, consecutive vectors: no bank
                    // conflicts), and the row's elements picked from them.
                    const Vec *tailrow = reinterpret_cast<const Vec *>(
                        phb + (size_t)PHASE_ROWS * ROW_BYTES + (size_t)prow * 16);
#pragma unroll
                    for (int v = 0; v < VPL; ++v) {
                        const Vec cur = boxrow[v * 32 + lane];
                        const Vec nxt = (v == VPL - 1 && lane == 31) ? *tailrow
                                                                     : boxrow[v * 32 + lane + 1];
                        if constexpr (VE == 4) {
                            if (off == 1) a[v] = Vec{cur.y, cur.z, cur.w, nxt.x};
                            else if (off == 2) a[v] = Vec{cur.z, cur.w, nxt.x, nxt.y};
                            else a[v] = Vec{cur.w, nxt.x, nxt.y, nxt.z};
                        } else {
                            a[v] = Vec{cur.y, nxt.x};
                        }
                    }
                }
            } else if constexpr (kTma) {
                const Vec *rowp = reinterpret_cast<const Vec *>(
                    ring + (size_t)stage * TILE_BYTES +
                    (size_t)(warp * RPW + i) * ROW_BYTES);
#pragma unroll
                for (int v = 0; v < VPL; ++v) a[v] = rowp[v * 32 + lane];
            } else {
                const int64_t row = row0 + i;
                const T *arow = Ag + b * prm.strideA + row * prm.lda;
#pragma unroll
                for (int v = 0; v < VPL; ++v) {
                    T tmp[VE];
#pragma unroll
                    for (int e = 0; e < VE; ++e) {
                        const int64_t col = col0 + lane_col<T>(v, lane, e);
                        tmp[e] = (row < prm.M && col < prm.N) ? arow[col] : T(0);
                    }
                    if constexpr (VE == 4) a[v] = Vec{tmp[0], tmp[1], tmp[2], tmp[3]};
                    else a[v] = Vec{tmp[0], tmp[1]};
                }
            }
            const T ri = kS ? __shfl_sync(0xffffffffu, rmine, i) : T(0);
            if constexpr (kRank2) {
                // A_hat = A + u1 v1^T + u2 v2^T, element by element; written
                // back when asked (in place is fine: each element is read
                // before it is written, by the same thread).
                const T u1i = __shfl_sync(0xffffffffu, u1mine, i);
                const T u2i = __shfl_sync(0xffffffffu, u2mine, i);
                const int64_t row = row0 + i;
#pragma unroll
                for (int v = 0; v < VPL; ++v) {
                    T tmp[VE];
#pragma unroll
                    for (int e = 0; e < VE; ++e)
                        tmp[e] = mul_acc(u2i, v2v[v * VE + e],
                                         mul_acc(u1i, v1v[v * VE + e], vget(a[v], e)));
                    if constexpr (VE == 4) a[v] = Vec{tmp[0], tmp[1], tmp[2], tmp[3]};
                    else a[v] = Vec{tmp[0], tmp[1]};
                    if (prm.a_out != nullptr && row < prm.M) {
                        T *orow = static_cast<T *>(prm.a_out) + row * prm.lda_out;
#pragma unroll
                        for (int e = 0; e < VE; ++e) {
                            const int64_t col = col0 + lane_col<T>(v, lane, e);
                            if (col < prm.N) orow[col] = tmp[e];
                        }
                    }
                }
            }
            Acc dot = Acc(0);
#pragma unroll
            for (int v = 0; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) {
                    const T av = vget(a[v], e);
                    if constexpr (kQ) dot = mul_acc(av, pv[v * VE + e], dot);
                    if constexpr (kS) tacc[v * VE + e] = mul_acc(av, ri, tacc[v * VE + e]);
                }
            qp[i] = dot;
        }
        if constexpr (kTma && !kEarly) {
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&empty_bar[stage]));
        }
        if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
        }

        // q: complete band partial of each of this warp's rows.
        if constexpr (kQ) warp_rows_reduce<RPW>(qp, lane);
        if (kQ && butterfly_writer<RPW>(lane)) {
            const int64_t row = row0 + butterfly_row<RPW>(lane);
            if (row < prm.M) {
                if (prm.bands == 1) {
                    Acc *qo = static_cast<Acc *>(prm.q);
                    qo[b * prm.strideQ + row] = qp[0];
                } else if constexpr (kAtomicOut) {
                    atomicAdd(static_cast<Acc *>(prm.q) + b * prm.strideQ + row, qp[0]);
                } else {
                    Acc *qw = static_cast<Acc *>(prm.q_ws);
                    qw[(b * prm.bands + band) * prm.M + row] = qp[0];
                }
            }
        }

        // s: tile -> group -> segment accumulation.
        if constexpr (kS) {
    #pragma unroll
            for (int e = 0; e < kLaneCols; ++e) grp[e] = grp[e] + tacc[e];
            if (++ngrp == kGroupTiles) {
    #pragma unroll
                for (int e = 0; e < kLaneCols; ++e) {
                    seg[e] = seg[e] + grp[e];
                    grp[e] = Acc(0);
                }
                ngrp = 0;
            }

            if (stripe == S - 1 || k == ntiles - 1) {  // segment end: flush s
    #pragma unroll
                for (int e = 0; e < kLaneCols; ++e) seg[e] = seg[e] + grp[e];
                Acc *sw = scratch + warp * kBandCols;
    #pragma unroll
                for (int v = 0; v < VPL; ++v)
    #pragma unroll
                    for (int e = 0; e < VE; ++e) sw[lane_col<T>(v, lane, e)] = seg[v * VE + e];
                named_barrier(1, nthreads_c);
                const bool whole_band = (seg_start_stripe == 0 && stripe == S - 1);
                for (int col = threadIdx.x; col < kBandCols; col += nthreads_c) {
                    Acc acc = scratch[col];
    #pragma unroll
                    for (int w = 1; w < W; ++w) acc = acc + scratch[w * kBandCols + col];
                    if (whole_band) {
                        if (col0 + col < prm.N) {
                            Acc *so = static_cast<Acc *>(prm.s);
                            so[b * prm.strideS + col0 + col] = acc;
                        }
                    } else if constexpr (kAtomicOut) {
                        if (col0 + col < prm.N)
                            atomicAdd(static_cast<Acc *>(prm.s) + b * prm.strideS + col0 + col, acc);
                    } else {
                        Acc *sws = static_cast<Acc *>(prm.s_ws);
                        sws[((c * prm.max_seg) + (g - g_first)) * kBandCols + col] = acc;
                    }
                }
                named_barrier(1, nthreads_c);
    #pragma unroll
                for (int e = 0; e < kLaneCols; ++e) {
                    grp[e] = Acc(0);
                    seg[e] = Acc(0);
                }
                ngrp = 0;
            }
        }
    }
}

template <typename T, int W, int RPW, int STAGES, bool kTma, bool kBatched3d,
          int kOut = kOutBoth, bool kRank2 = false, bool kRev = false>
__global__ void __launch_bounds__((W + (kTma ? 1 : 0)) * 32,
                                  (!kTma && std::is_same<T, int32_t>::value) ? 2 : 1)
dualmv_stream_kernel(const __grid_constant__ CUtensorMap tmap, const Params prm) {
    stream_body<T, W, RPW, STAGES, kTma, kBatched3d, kOut, kRank2, 0, kRev>(&tmap, prm);
    if (prm.pdl_late) pdl_wait();  // see Params::pdl_late
}

// The same kernel for one problem whose row stride or base is not 16-byte
// aligned (the TMA unit cannot take it as one 2-D tensor): row phase ph (rows
// r = ph mod NPH) is its own 2-D tensor with the base rounded down to 16
// bytes, so that its row stride NPH * lda * size is a multiple of 16 bytes.
// NPH = 1 covers an unaligned base alone.
template <typename T, int W, int RPW, int STAGES, int NPH>
__global__ void __launch_bounds__((W + 1) * 32, 1)
dualmv_stream_phased_kernel(const __grid_constant__ TmapSet maps, const Params prm) {
    stream_body<T, W, RPW, STAGES, true, false, kOutBoth, false, NPH>(maps.m, prm);
    if (prm.pdl_late) pdl_wait();  // see Params::pdl_late
}

// ------------------------------------------------------- combine arithmetic --
// The two sums the combine kernel forms, as device functions, so that a kernel
// that takes over a pass's combine (GEMVER's vector updates) adds the
// partials in the same order and gets the same bits.

// Output i of problem b from its band partials: C interleaved chunks (chunk y
// adds bands y, y + C, ... in ascending order), then the chunks in order.
template <typename Acc>
__device__ __forceinline__ Acc q_band_sum(const Params &prm, int64_t b, int64_t i, int C) {
    const Acc *base = static_cast<const Acc *>(prm.q_ws) + (b * prm.bands) * prm.M + i;
    Acc tot = Acc(0);
    for (int y = 0; y < C; ++y) {
        Acc acc = Acc(0);
        int64_t k = y;
        if (k < prm.bands) {
            acc = base[k * prm.M];
            k += C;
        }
        for (; k < prm.bands; k += C) acc = acc + base[k * prm.M];
        tot = y == 0 ? acc : tot + acc;
    }
    return tot;
}

// The CTAs holding stripes of global band g (b * bands + band): c_lo .. c_hi.
// When they are one CTA, that CTA wrote the band's s directly.
__device__ __forceinline__ void band_ctas_of(const Params &prm, int64_t g, int64_t &c_lo,
                                             int64_t &c_hi) {
    const int64_t S = prm.stripes;
    c_lo = cta_of_tile(g * S, prm.tiles, prm.grid);
    c_hi = cta_of_tile(g * S + S - 1, prm.tiles, prm.grid);
}

// Column col of global band g (split between CTAs c_lo < c_hi): its segment
// partials added in CTA order.  CTA cc's segment of band g is g minus the
// band of its first tile; every CTA after c_lo starts inside band g, so the
// band is its segment 0, and only c_lo's segment needs a division: the loads
// do not wait on one another (a running segment count between them had made
// the combine of the 1024^2 workload take 5 of its 8 us).
template <typename Acc>
__device__ __forceinline__ Acc s_segment_sum(const Params &prm, int64_t g, int col, int64_t c_lo,
                                             int64_t c_hi) {
    const Acc *src = static_cast<const Acc *>(prm.s_ws) + col;
    const int64_t seg0 = g - ((c_lo * prm.tiles) / prm.grid) / prm.stripes;
    const int64_t pitch = prm.max_seg * prm.band_cols;
    Acc acc = src[c_lo * pitch + seg0 * prm.band_cols];
#pragma unroll 8
    for (int64_t cc = c_lo + 1; cc <= c_hi; ++cc) acc = acc + src[cc * pitch];
    return acc;
}

// --------------------------------------------------------- combine kernel --
//
// Adds the band partials of q and the segment partials of s in a fixed
// order, for the outputs the stream kernel could not finish alone.  Launched
// as a programmatic dependent of the stream kernel: it waits for that grid to
// complete before reading the workspace.  256 threads per block.
//   Blocks [0, q_blocks): rows of q.  A block takes R = 256 / C consecutive
//     outputs (over batch * M) and C chunks; chunk y adds bands y, y + C,
//     y + 2C, ... in ascending order, then the C chunk sums are added in
//     ascending chunk order.  C depends only on the band count, so the
//     order (and the rounding) is the same on every call.
//   Blocks [q_blocks, q_blocks + batch * bands): one band of s each (band
//     width prm.band_cols <= 256); the segments of a band split between
//     CTAs are added in ascending CTA order.
template <typename Acc>
__global__ void __launch_bounds__(256)
dualmv_combine_kernel(const Params prm, int64_t q_blocks, int q_chunks) {
    // The next call's fp64 streaming kernel may launch once every block of
    // this grid has started (it waits for this grid's completion before it
    // reads or writes anything).
    pdl_launch_dependents();
    pdl_wait();
    __shared__ Acc part[256];
    const Acc *qw = static_cast<const Acc *>(prm.q_ws);
    if ((int64_t)blockIdx.x < q_blocks) {  // (q_blocks is 0 unless q is computed)
        const int C = q_chunks, R = 256 / C;
        const int x = threadIdx.x % R, y = threadIdx.x / R;
        const int64_t idx = (int64_t)blockIdx.x * R + x;
        const bool valid = idx < prm.batch * prm.M;
        int64_t b = 0, i = 0;
        Acc acc = Acc(0);
        if (valid) {
            b = idx / prm.M;
            i = idx - b * prm.M;
            const Acc *base = qw + (b * prm.bands) * prm.M + i;
            int64_t k = y;
            if (k < prm.bands) {
                acc = base[k * prm.M];
                k += C;
            }
#pragma unroll 4
            for (; k < prm.bands; k += C) acc = acc + base[k * prm.M];
        }
        part[threadIdx.x] = acc;
        __syncthreads();
        if (y == 0 && valid) {
            Acc tot = part[x];
            for (int yy = 1; yy < C; ++yy) tot = tot + part[yy * R + x];
            static_cast<Acc *>(prm.q)[b * prm.strideQ + i] = tot;
        }
        return;
    }
    const int64_t g = (int64_t)blockIdx.x - q_blocks;  // b * bands + band
    const int64_t b = g / prm.bands, band = g - b * prm.bands;
    int64_t c_lo, c_hi;
    band_ctas_of(prm, g, c_lo, c_hi);
    if (c_lo == c_hi) return;  // written directly by the stream kernel
    const int col = threadIdx.x;
    if (col >= prm.band_cols) return;
    const int64_t j = band * prm.band_cols + col;
    if (j >= prm.N) return;
    static_cast<Acc *>(prm.s)[b * prm.strideS + j] = s_segment_sum<Acc>(prm, g, col, c_lo, c_hi);
}

// Zeroes q and s (strided batches) ahead of a stream kernel that adds into
// them atomically; lets that kernel launch at once (programmatic dependent
// launch) so its prologue and first copies overlap this one.
template <typename Acc>
__global__ void dualmv_zero_outputs_kernel(Acc *q, int64_t M, int64_t strideQ, Acc *s,
                                           int64_t N, int64_t strideS, int64_t batch) {
    pdl_launch_dependents();
    const int64_t nq = M * batch, total = nq + N * batch;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        if (idx < nq) {
            const int64_t b = idx / M, i = idx - b * M;
            q[b * strideQ + i] = Acc(0);
        } else {
            const int64_t js = idx - nq;
            const int64_t b = js / N, j = js - b * N;
            s[b * strideS + j] = Acc(0);
        }
    }
}

// y = alpha * t + beta * y (the GESUMMV epilogue).
// Zero-fill of strided outputs (empty problems).
template <typename Acc>
__global__ void dualmv_zero_kernel(Acc *out, int64_t len, int64_t stride, int64_t batch) {
    const int64_t total = len * batch;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int64_t b = idx / len, i = idx - b * len;
        out[b * stride + i] = Acc(0);
    }
}

}  // namespace dmv
