// Wide-tile streaming kernel for int32 inputs (q = A p, s = A^T r, sums
// exact modulo 2^64).
//
// Why a second tile shape: when the row stride of A is not a multiple of
// 128 bytes, a 256-column box row (1 KiB) of most rows starts inside a
// 128-byte line and touches nine lines instead of eight.  The line that
// straddles two 256-column bands is fetched once for each band, and with
// band-major tiles the two fetches are far apart in time, so DRAM moves up
// to 12.5% more than A.  Here a tile is RPW rows by W * 256 columns and
// consumer warp w takes the 256-column sub-band w of the same RPW rows, so
// a tile reads W KiB of each of its rows contiguously and only the line
// shared with the next wide band is fetched twice (1/64 of a row segment at
// W = 8).
//
// Integer sums are exact in any order, so the warps need not combine their
// partials: each warp adds its row partials into q and, at the end of a
// segment (the stripes of one wide band this CTA owns), its 256 column sums
// into s with 64-bit atomics; a preceding kernel zeroes q and s and this
// kernel, its programmatic dependent, waits for it before the first add.
// Tiles are numbered band-major over (wide band, stripe) and split into
// contiguous per-CTA ranges exactly as in the main kernel.  Every mbarrier
// wait is bounded (see dualmv_kernels.cuh).
#pragma once

#include "dualmv_kernels.cuh"

namespace dmv {

template <int W, int RPW, int STAGES>
struct WideLayout {
    static constexpr int kBoxBytes = RPW * kBandCols * 4;  // one warp's sub-band
    static constexpr int kTileBytes = W * kBoxBytes;
    static constexpr int kAlign = 1024;
    static constexpr int kRing = STAGES * kTileBytes;
    static constexpr int kBars = 2 * STAGES * 8;
    static constexpr int kTotal = kAlign + kRing + kBars;
};

template <int W, int RPW, int STAGES>
__global__ void __launch_bounds__((W + 1) * 32, 1)
dualmv_wide_i32_kernel(const __grid_constant__ CUtensorMap tmap, const Params prm) {
    using T = int32_t;
    using Acc = unsigned long long;
    using Vec = int4;
    constexpr int VE = 4;
    constexpr int VPL = kLaneCols / VE;  // 16-byte vectors per lane per row
    constexpr int ROW_BYTES = kBandCols * (int)sizeof(T);
    constexpr int64_t WIDE = (int64_t)W * kBandCols;  // columns per wide band
    using L = WideLayout<W, RPW, STAGES>;
    static_assert(L::kBoxBytes == RPW * ROW_BYTES, "box size mismatch");

    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_raw + shared_align_pad<L::kAlign>(smem_raw);
    unsigned char *ring = smem;
    uint64_t *full_bar = reinterpret_cast<uint64_t *>(smem + L::kRing);
    uint64_t *empty_bar = full_bar + STAGES;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t T_ = prm.tiles, G = prm.grid, S = prm.stripes;
    const int64_t c = blockIdx.x;
    const int64_t t0 = cta_first_tile(c, T_, G);
    const int64_t ntiles = cta_first_tile(c + 1, T_, G) - t0;

    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(smem_u32(&full_bar[i]), 1);
            mbar_init(smem_u32(&empty_bar[i]), W);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    // ---------------------------------------------------------- producer ----
    if (warp == W) {
        if (lane == 0) {
            const uint64_t pol = policy_evict_first();
            bool ok = true;
            int64_t issued = 0;
            TileCursor cur;
            cur.init(t0, S, prm.bands);
            int stage = 0;
            uint32_t phase = 0;
            for (int64_t k = 0; k < ntiles; ++k) {
                if (ok && k >= STAGES)
                    ok = mbar_wait_bounded(smem_u32(&empty_bar[stage]), phase ^ 1u);
                if (!ok) break;
                // Sub-bands wholly past column N are not loaded (their warps
                // skip them), so the byte count covers the live ones only.
                const int64_t x0 = cur.band * WIDE;
                const int64_t left = prm.N - x0;
                const int live = left >= WIDE ? W : (int)((left + kBandCols - 1) / kBandCols);
                const uint32_t fb = smem_u32(&full_bar[stage]);
                mbar_arrive_expect_tx(fb, (uint32_t)(live * L::kBoxBytes));
                const uint32_t dst = smem_u32(ring + (size_t)stage * L::kTileBytes);
                const int y = (int)(cur.stripe * RPW);
                for (int w = 0; w < live; ++w)
                    tma_load_2d(dst + (uint32_t)(w * L::kBoxBytes), &tmap,
                                (int)(x0 + (int64_t)w * kBandCols), y, fb, pol);
                issued = k + 1;
                cur.advance(S, prm.bands);
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            for (int64_t k = issued > STAGES ? issued - STAGES : 0; k < issued; ++k)
                mbar_wait_bounded(smem_u32(&full_bar[(int)(k % STAGES)]),
                                  (uint32_t)(k / STAGES) & 1u);
        }
        return;
    }

    // --------------------------------------------------------- consumers ----
    const T *__restrict__ pg = static_cast<const T *>(prm.p);
    const T *__restrict__ rg = static_cast<const T *>(prm.r);
    Acc *__restrict__ qo = static_cast<Acc *>(prm.q);
    Acc *__restrict__ so = static_cast<Acc *>(prm.s);

    T pv[kLaneCols];
    Acc grp[kLaneCols], seg[kLaneCols];
#pragma unroll
    for (int e = 0; e < kLaneCols; ++e) {
        pv[e] = 0;
        grp[e] = 0;
        seg[e] = 0;
    }
    int ngrp = 0;
    int64_t seg_start_stripe = 0;
    bool ok = true;

    TileCursor cur;
    cur.init(t0, S, prm.bands);
    T r_next = 0;
    {
        const int64_t row = cur.stripe * RPW + lane;
        if (lane < RPW && row < prm.M) r_next = rg[row];
    }
    int stage = 0;
    uint32_t phase = 0;
    pdl_wait();  // q and s zeroed before any add

    for (int64_t k = 0; k < ntiles; ++k) {
        const int64_t stripe = cur.stripe;
        const int64_t col0 = cur.band * WIDE + (int64_t)warp * kBandCols;
        const int64_t row0 = stripe * RPW;
        const bool live = col0 < prm.N;  // this warp's sub-band holds columns
        const T rmine = r_next;
        cur.advance(S, prm.bands);
        if (k + 1 < ntiles) {
            const int64_t row = cur.stripe * RPW + lane;
            r_next = (lane < RPW && row < prm.M) ? rg[row] : 0;
        }
        if (k == 0 || stripe == 0) {  // a new segment: this sub-band's p
            seg_start_stripe = stripe;
#pragma unroll
            for (int v = 0; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) {
                    const int64_t col = col0 + lane_col<T>(v, lane, e);
                    pv[v * VE + e] = col < prm.N ? pg[col] : 0;
                }
        }

        Acc qp[RPW];
        Acc tacc[kLaneCols];
#pragma unroll
        for (int e = 0; e < kLaneCols; ++e) tacc[e] = 0;
#pragma unroll
        for (int i = 0; i < RPW; ++i) qp[i] = 0;

        if (ok) ok = mbar_wait_bounded(smem_u32(&full_bar[stage]), phase);
        if (live) {
            const unsigned char *box =
                ring + (size_t)stage * L::kTileBytes + (size_t)warp * L::kBoxBytes;
#pragma unroll
            for (int i = 0; i < RPW; ++i) {
                const Vec *rowp = reinterpret_cast<const Vec *>(box + (size_t)i * ROW_BYTES);
                Vec a[VPL];
#pragma unroll
                for (int v = 0; v < VPL; ++v) a[v] = rowp[v * 32 + lane];
                const T ri = __shfl_sync(0xffffffffu, rmine, i);
                Acc dot = 0;
#pragma unroll
                for (int v = 0; v < VPL; ++v)
#pragma unroll
                    for (int e = 0; e < VE; ++e) {
                        const T av = vget(a[v], e);
                        dot = mul_acc(av, pv[v * VE + e], dot);
                        tacc[v * VE + e] = mul_acc(av, ri, tacc[v * VE + e]);
                    }
                qp[i] = dot;
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&empty_bar[stage]));
        if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
        }

        if (live) {
            // q: this sub-band's partial of each of the RPW rows.
            warp_rows_reduce<RPW>(qp, lane);
            if (butterfly_writer<RPW>(lane)) {
                const int64_t row = row0 + butterfly_row<RPW>(lane);
                if (row < prm.M) atomicAdd(qo + row, qp[0]);
            }
            // s: tile -> group -> segment, then the segment's column sums.
#pragma unroll
            for (int e = 0; e < kLaneCols; ++e) grp[e] += tacc[e];
            if (++ngrp == kGroupTiles) {
#pragma unroll
                for (int e = 0; e < kLaneCols; ++e) {
                    seg[e] += grp[e];
                    grp[e] = 0;
                }
                ngrp = 0;
            }
            if (stripe == S - 1 || k == ntiles - 1) {
                const bool whole_band = seg_start_stripe == 0 && stripe == S - 1;
#pragma unroll
                for (int v = 0; v < VPL; ++v)
#pragma unroll
                    for (int e = 0; e < VE; ++e) {
                        const int64_t col = col0 + lane_col<T>(v, lane, e);
                        const Acc val = seg[v * VE + e] + grp[v * VE + e];
                        if (col < prm.N) {
                            if (whole_band) so[col] = val;
                            else atomicAdd(so + col, val);
                        }
                    }
#pragma unroll
                for (int e = 0; e < kLaneCols; ++e) {
                    grp[e] = 0;
                    seg[e] = 0;
                }
                ngrp = 0;
            }
        }
    }
}

}  // namespace dmv
