// ATAX (Table 1: y = A^T (A x)) with one read of A from HBM, for fp64.
//
// The cluster scheme of atax_cluster_kernel (dualmv_atax.cuh) with the
// double-float arithmetic of dualmv_stream_f64e_kernel (dualmv_f64e.cuh):
// a cluster of C CTAs streams one stripe of R rows at a time, each warp a
// 256-column sub-band of doubles (lane l: columns 2l, 2l+1, +64, +128,
// +192), and keeps it in shared memory until t = A x of those rows is known.
//
//   1. Row phase (stripe j): each element a is split into a_hi + a_lo
//      (integer operations, as split_f64), the row products with x (split
//      once per kernel) are formed and summed in packed double-float pairs,
//      and the split is written back over the element in shared memory
//      (a_hi, a_lo as two floats: the same 8 bytes).  The warp's row
//      partials (reduce-scatter butterfly, rounded to fp64) are added over
//      the warps in warp order and sent to every CTA of the cluster
//      (st.async into distributed shared memory).
//   2. After the partials of stripe j - 1 have all arrived: t_i as their
//      fp64 sum in CTA-rank order (bit-identical in every CTA), split once.
//   3. Column phase (stripe j - 1): y_j += t_i a_ij from the split still in
//      shared memory, in double-float pairs (tile -> group of kGroupTiles ->
//      fp64 segment in shared memory).
//
// Warps are not held in step by CTA-wide barriers (the row phase of a warp
// may run a stripe ahead of another's column phase).  A control warp (warp
// W) does the exchange: for stripe j it waits until every compute warp has
// written its row partials (mbarrier wfull[j % 4], W arrivals), sends the
// CTA's partials, and, for stripe j - 1, waits for the cluster's partials,
// forms and splits t and releases it (mbarrier tready[(j - 1) % 4]).  It
// takes stripe j - 1's partials out of their slot before it sends stripe j,
// so no peer can write a slot that is still unread (a peer's stripe j + 3
// needs t of stripe j, hence this CTA's stripe j).
//
// Range.  The double-float forms are exact only while |a|, |x_j| and |t_i|
// lie in [2^-40, 2^40) or are zero.  x is checked once; a warp whose tile
// holds anything else (a cheap bound, then an exact re-check that lets zeros
// pass) takes both phases of that stripe in native fp64, reading its rows
// again from global memory (the shared copy now holds the split); a stripe
// whose t has a value out of range takes its column phase in native fp64.
//
// Waits are bounded as in the fp32 kernel, every CTA reaches the same
// cluster barriers, and a CTA leaves only after the last one.
#pragma once

#include "dualmv_atax.cuh"
#include "dualmv_f64e.cuh"

namespace dmv {

struct AtaxParams64 {
    const double *A;   // only for the native fallback (rows re-read)
    int64_t lda;
    const double *x;
    double *y_ws;      // [clusters][N] column sums of each cluster's stripes
    int64_t M, N;
    int64_t stripes;   // ceil(M / R)
    int64_t clusters;  // clusters launched
    int64_t bands;     // ceil(N / BAND) sub-bands
};

template <int W, int R, int STAGES, int BAND = kBandCols>
struct AtaxLayout64 {
    static constexpr int kBoxBytes = R * BAND * 8;  // one warp's sub-band, R rows
    static constexpr int kAlign = 1024;
    static constexpr int kRing = W * STAGES * kBoxBytes;
    static constexpr int kWarpPart = kAtaxSlots * W * R * 8;               // [slot][W][R] fp64
    static constexpr int kPart = kAtaxSlots * kAtaxMaxCluster * R * 8;     // [slot][C][R] fp64
    // [slot][R] t (fp64), [slot][R] its split (float2), [slot] out-of-range flag
    static constexpr int kT = kAtaxSlots * (R * 8 + R * 8 + 8);
    static constexpr int kSeg = W * BAND * 8;                              // [W][BAND] fp64
    // full[W][STAGES], part[slot], wfull[slot], tready[slot]
    static constexpr int kBars = (W * STAGES + 3 * kAtaxSlots) * 8;
    static constexpr int kTotal = kAlign + kRing + kWarpPart + kPart + kT + kSeg + kBars;
};

// 8 bytes into a peer's shared memory, counted on the peer's mbarrier.
__device__ __forceinline__ void st_async_f64(uint32_t raddr, double v, uint32_t rbar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b64 [%0], %1, [%2];"
                 ::"r"(raddr), "l"(__double_as_longlong(v)), "r"(rbar) : "memory");
}

template <int W, int R, int STAGES, int BAND = kBandCols>
__global__ void __launch_bounds__((W + 1) * 32, 1)
atax_cluster_f64_kernel(const __grid_constant__ CUtensorMap tmap, const AtaxParams64 prm) {
    using L = AtaxLayout64<W, R, STAGES, BAND>;
    using Vec = double2;
    constexpr int VE = 2, LANE_COLS = BAND / 32, VPL = LANE_COLS / VE;
    constexpr int ROW_BYTES = BAND * 8;
    static_assert(L::kBoxBytes == R * ROW_BYTES, "box size mismatch");
    static_assert(VPL == 2 || VPL == 4, "a sub-band of 128 or 256 columns");
    static_assert(kAtaxMaxCluster * R <= 64, "the control warp sends two values a lane");

    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_raw + shared_align_pad<L::kAlign>(smem_raw);
    unsigned char *ring = smem;
    double *wpart = reinterpret_cast<double *>(smem + L::kRing);  // [slot][W][R]
    double *part = wpart + kAtaxSlots * W * R;                    // [slot][kMax][R]
    double *tvec = part + kAtaxSlots * kAtaxMaxCluster * R;       // [slot][R]
    float2 *tsplit = reinterpret_cast<float2 *>(tvec + kAtaxSlots * R);  // [slot][R]
    uint32_t *tflag = reinterpret_cast<uint32_t *>(tsplit + kAtaxSlots * R);  // [slot]
    double *segs = reinterpret_cast<double *>(reinterpret_cast<unsigned char *>(tvec) + L::kT);
    uint64_t *full_bar = reinterpret_cast<uint64_t *>(smem + L::kRing + L::kWarpPart +
                                                      L::kPart + L::kT + L::kSeg);
    uint64_t *part_bar = full_bar + W * STAGES;
    uint64_t *wfull_bar = part_bar + kAtaxSlots;
    uint64_t *tready_bar = wfull_bar + kAtaxSlots;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t crank = cluster_rank(), csize = cluster_size();
    const int64_t cl = cluster_id();
    const int64_t s0 = cl * prm.stripes / prm.clusters;
    const int64_t ns = (cl + 1) * prm.stripes / prm.clusters - s0;

    if (threadIdx.x == 0) {
        for (int i = 0; i < W * STAGES; ++i) mbar_init(smem_u32(&full_bar[i]), 1);
        for (int i = 0; i < kAtaxSlots; ++i) {
            mbar_init(smem_u32(&part_bar[i]), 1);
            mbar_init(smem_u32(&wfull_bar[i]), W);
            mbar_init(smem_u32(&tready_bar[i]), 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    // Every CTA's barriers exist before any peer sends to them.
    cluster_sync();
    // A programmatic dependent of the kernel before it (see atax_cluster_kernel).
    pdl_wait();
    pdl_launch_dependents();

    // ---------------------------------------------------- control warp ----
    if (warp == W) {
        bool ok = true;
        for (int64_t j = 0; j <= ns; ++j) {
            if (j < ns && lane == 0)
                mbar_arrive_expect_tx(smem_u32(&part_bar[j % kAtaxSlots]), csize * R * 8u);
            if (j >= 1) {
                // t of stripe j - 1: the C partials of each row in CTA-rank order.
                const int64_t jp = j - 1;
                const int bp = (int)(jp % kAtaxSlots);
                if (!mbar_wait_cluster_bounded(smem_u32(&part_bar[bp]),
                                               (uint32_t)(jp / kAtaxSlots) & 1u))
                    ok = false;
                bool bad = false;
                if (lane < R) {
                    double tt = part[(bp * kAtaxMaxCluster) * R + lane];
                    for (uint32_t k = 1; k < csize; ++k)
                        tt += part[(bp * kAtaxMaxCluster + k) * R + lane];
                    float th, tl;
                    split_f64(tt, th, tl);
                    bad = !f64e_in_range(tt);
                    tvec[bp * R + lane] = tt;
                    tsplit[bp * R + lane] = make_float2(th, tl);
                }
                const bool any_bad = __any_sync(0xffffffffu, bad);
                if (lane == 0) tflag[bp] = any_bad ? 1u : 0u;
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&tready_bar[bp]));
            }
            if (j < ns) {
                // The CTA's partial of each row (warp order), sent to every
                // CTA of the cluster (this one included) into slot [b][crank].
                const int b = (int)(j % kAtaxSlots);
                if (ok && !mbar_wait_bounded(smem_u32(&wfull_bar[b]),
                                             (uint32_t)(j / kAtaxSlots) & 1u))
                    ok = false;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int idx = lane + 32 * h;
                    if (idx < (int)(csize * R)) {
                        const int i = idx % R;
                        const uint32_t peer = (uint32_t)idx / R;
                        const double *wp = wpart + b * W * R;
                        double cp = wp[i];
#pragma unroll
                        for (int w = 1; w < W; ++w) cp += wp[w * R + i];
                        const uint32_t slot_addr =
                            smem_u32(&part[(b * kAtaxMaxCluster + crank) * R + i]);
                        st_async_f64(peer_addr(slot_addr, peer), cp,
                                     peer_addr(smem_u32(&part_bar[b]), peer));
                    }
                }
            }
        }
        // No CTA leaves while a peer may still write into its shared memory.
        cluster_sync();
        return;
    }

    // --------------------------------------------------- compute warps ----
    const int64_t sb = (int64_t)crank * W + warp;  // this warp's sub-band
    const bool live = sb < prm.bands;
    const int64_t col0 = sb * BAND;
    double *segp = segs + warp * BAND;  // this warp's fp64 column sums

    // x of this warp's columns, split once; its range checked once.
    float2 xh2[VPL], xl2[VPL];
    bool x_bad = false;
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
        float h[VE], l[VE];
#pragma unroll
        for (int e = 0; e < VE; ++e) {
            const int64_t col = col0 + lane_col<double>(v, lane, e);
            const double xv = (live && col < prm.N) ? prm.x[col] : 0.0;
            split_f64(xv, h[e], l[e]);
            x_bad |= !f64e_in_range(xv);
            segp[lane_col<double>(v, lane, e)] = 0.0;
        }
        xh2[v] = make_float2(h[0], h[1]);
        xl2[v] = make_float2(l[0], l[1]);
    }
    const bool warp_x_bad = __any_sync(0xffffffffu, x_bad);

    // Self-loading: lane 0 issues this warp's boxes, STAGES stripes ahead.
    uint64_t pol = 0;
    int64_t issued = 0;
    auto issue = [&](int64_t j) {
        const int slot = warp * STAGES + (int)(j % STAGES);
        const uint32_t fb = smem_u32(&full_bar[slot]);
        mbar_arrive_expect_tx(fb, L::kBoxBytes);
        tma_load_2d(smem_u32(ring + (size_t)slot * L::kBoxBytes), &tmap, (int)col0,
                    (int)((s0 + j) * R), fb, pol);
        ++issued;
    };
    if (live && lane == 0) {
        pol = policy_evict_first();
        for (int64_t j = 0; j < STAGES && j < ns; ++j) issue(j);
    }

    // Elements re-read from global memory by the native fallback.
    auto a_at = [&](int64_t row, int64_t col) -> double {
        return (row < prm.M && col < prm.N) ? prm.A[row * prm.lda + col] : 0.0;
    };

    DF2 grp2[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) grp2[v].s = grp2[v].c = make_float2(0.f, 0.f);
    int ngrp = 0;
    bool ok = true;
    int64_t confirmed = 0;      // boxes of this warp seen landed, in stripe order
    uint32_t stage_native = 0;  // bit s: the stripe in stage s took the native row phase
    const int perm = butterfly_row<R>(lane);

    for (int64_t j = 0; j <= ns; ++j) {
        if (j < ns) {
            // 1. Row partials of stripe j over this sub-band.
            const int b = (int)(j % kAtaxSlots);
            double *wp = wpart + (b * W + warp) * R;
            if (live) {
                const int st = (int)(j % STAGES);
                const int slot = warp * STAGES + st;
                if (ok) {
                    ok = mbar_wait_bounded(smem_u32(&full_bar[slot]),
                                           (uint32_t)(j / STAGES) & 1u);
                    if (ok) confirmed = j + 1;
                }
                unsigned char *box = ring + (size_t)slot * L::kBoxBytes;
                const int64_t row0 = (s0 + j) * R;
                DF q[R];
                // Range keys: one running max per column vector (independent
                // chains; one chain through the stripe serialises the warp).
                uint32_t span = 0;
                uint32_t spanv[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                for (int i = 0; i < R; ++i) {
                    // Slot i of this lane is row i ^ perm (warp_rows_reduce_df_perm).
                    const int ri = i ^ perm;
                    Vec *rowp = reinterpret_cast<Vec *>(box + (size_t)ri * ROW_BYTES);
                    Vec a[VPL];
#pragma unroll
                    for (int v = 0; v < VPL; ++v) a[v] = rowp[v * 32 + lane];
                    DF2 qp[VPL];
#pragma unroll
                    for (int v = 0; v < VPL; ++v) {
                        float ah0, al0, ah1, al1;
                        split_f64(a[v].x, ah0, al0);
                        split_f64(a[v].y, ah1, al1);
                        spanv[v] = __vimax3_u32(spanv[v], f64e_range_key(a[v].x),
                                                f64e_range_key(a[v].y));
                        const float2 ah = make_float2(ah0, ah1), al = make_float2(al0, al1);
                        df_prod2(ah, al, xh2[v], xl2[v], qp[v].s, qp[v].c);
                        // The column phase reads the split, not the double.
                        reinterpret_cast<float4 *>(rowp)[v * 32 + lane] =
                            make_float4(ah0, ah1, al0, al1);
                    }
                    DF2 h;
                    if constexpr (VPL == 4)
                        h = df_add2(df_add2(qp[0], qp[1]), df_add2(qp[2], qp[3]));
                    else
                        h = df_add2(qp[0], qp[1]);
                    DF lo, hi;
                    lo.s = h.s.x;
                    lo.c = h.c.x;
                    hi.s = h.s.y;
                    hi.c = h.c.y;
                    q[i] = df_add(lo, hi);
                }
                if constexpr (VPL == 4)
                    span = max(max(spanv[0], spanv[1]), max(spanv[2], spanv[3]));
                else
                    span = max(spanv[0], spanv[1]);
                bool native = warp_x_bad;
                if (!native && __any_sync(0xffffffffu, span >= kF64eRangeSpan)) {
                    // Exact re-check from global memory: zeros pass.
                    bool bad = false;
#pragma unroll
                    for (int i = 0; i < R; ++i)
#pragma unroll
                        for (int v = 0; v < VPL; ++v)
#pragma unroll
                            for (int e = 0; e < VE; ++e)
                                bad |= !f64e_in_range(
                                    a_at(row0 + i, col0 + lane_col<double>(v, lane, e)));
                    native = __any_sync(0xffffffffu, bad);
                }
                if (!native) {
                    stage_native &= ~(1u << st);
                    warp_rows_reduce_df_perm<R>(q);
                    if (butterfly_writer<R>(lane)) wp[butterfly_row<R>(lane)] = df_to_double(q[0]);
                } else {
                    stage_native |= 1u << st;
                    double qd[R];
#pragma unroll
                    for (int i = 0; i < R; ++i) {
                        double dot = 0.0;
#pragma unroll
                        for (int v = 0; v < VPL; ++v)
#pragma unroll
                            for (int e = 0; e < VE; ++e) {
                                const int64_t col = col0 + lane_col<double>(v, lane, e);
                                const double xv = col < prm.N ? prm.x[col] : 0.0;
                                dot = fma(a_at(row0 + i, col), xv, dot);
                            }
                        qd[i] = dot;
                    }
                    warp_rows_reduce<R>(qd, lane);
                    if (butterfly_writer<R>(lane)) wp[butterfly_row<R>(lane)] = qd[0];
                }
            } else if (lane < R) {
                wp[lane] = 0.0;
            }
            // The partials are written: release them to the control warp.
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&wfull_bar[b]));
        }
        if (j >= 1) {
            // 2. Column sums of stripe j - 1, once its t is known.
            const int64_t jp = j - 1;
            const int bp = (int)(jp % kAtaxSlots);
            if (!mbar_wait_bounded(smem_u32(&tready_bar[bp]), (uint32_t)(jp / kAtaxSlots) & 1u))
                ok = false;
            if (live) {
                const int st = (int)(jp % STAGES);
                const int slot = warp * STAGES + st;
                const unsigned char *box = ring + (size_t)slot * L::kBoxBytes;
                if (tflag[bp] == 0u && !(stage_native & (1u << st))) {
                    DF2 tacc2[VPL];
#pragma unroll
                    for (int i = 0; i < R; ++i) {
                        const float2 t = tsplit[bp * R + i];
                        const float2 th2 = make_float2(t.x, t.x), tl2 = make_float2(t.y, t.y);
                        const float4 *rowp =
                            reinterpret_cast<const float4 *>(box + (size_t)i * ROW_BYTES);
#pragma unroll
                        for (int v = 0; v < VPL; ++v) {
                            const float4 f = rowp[v * 32 + lane];
                            float2 p0, p1;
                            df_prod2(make_float2(f.x, f.y), make_float2(f.z, f.w), th2, tl2,
                                     p0, p1);
                            if (i == 0) {
                                tacc2[v].s = p0;
                                tacc2[v].c = p1;
                            } else {
                                df_acc2(tacc2[v], p0, p1);
                            }
                        }
                    }
#pragma unroll
                    for (int v = 0; v < VPL; ++v) grp2[v] = df_add2(grp2[v], tacc2[v]);
                } else {
                    // Native fp64 from global memory (the shared copy holds the
                    // split, which is garbage for values out of range).
                    const int64_t row0 = (s0 + jp) * R;
#pragma unroll
                    for (int v = 0; v < VPL; ++v)
#pragma unroll
                        for (int e = 0; e < VE; ++e) {
                            const int c = lane_col<double>(v, lane, e);
                            double acc = 0.0;
#pragma unroll
                            for (int i = 0; i < R; ++i)
                                acc = fma(a_at(row0 + i, col0 + c), tvec[bp * R + i], acc);
                            segp[c] += acc;
                        }
                }
                if (++ngrp == kGroupTiles || jp == ns - 1) {
#pragma unroll
                    for (int v = 0; v < VPL; ++v)
#pragma unroll
                        for (int e = 0; e < VE; ++e) {
                            DF x;
                            x.s = e == 0 ? grp2[v].s.x : grp2[v].s.y;
                            x.c = e == 0 ? grp2[v].c.x : grp2[v].c.y;
                            segp[lane_col<double>(v, lane, e)] += df_to_double(x);
                        }
#pragma unroll
                    for (int v = 0; v < VPL; ++v) grp2[v].s = grp2[v].c = make_float2(0.f, 0.f);
                    ngrp = 0;
                }
                // The stage is free: refill it with the stripe STAGES ahead.
                __syncwarp();
                if (lane == 0 && ok && jp + STAGES < ns) {
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    issue(jp + STAGES);
                }
            }
        }
    }

    // This cluster's column sums of the sub-band.
    if (live) {
        __syncwarp();
        double *yw = prm.y_ws + cl * prm.N;
#pragma unroll
        for (int v = 0; v < VPL; ++v)
#pragma unroll
            for (int e = 0; e < VE; ++e) {
                const int c = lane_col<double>(v, lane, e);
                if (col0 + c < prm.N) yw[col0 + c] = segp[c];
            }
    }
    // After a timeout, boxes issued but never seen landed must land before
    // the CTA exits (bounded).
    if (live && lane == 0)
        for (int64_t kk = confirmed; kk < issued; ++kk)
            mbar_wait_bounded(smem_u32(&full_bar[warp * STAGES + (int)(kk % STAGES)]),
                              (uint32_t)(kk / STAGES) & 1u);
    // No CTA leaves while a peer may still write into its shared memory.
    cluster_sync();
}


// ---- warp-specialised form -----------------------------------------------
// The same stripes, exchange and arithmetic, with the row and column phases
// of a sub-band on two warps that share its ring of stages: row warp w
// (warps 0 .. W-1) splits each element, forms the row partials and writes
// the split back; column warp W + w takes the stage once its split is
// written (mbarrier ready[w][stage]) and t of the stripe is known, forms
// y_j += t_i a_ij, and refills the stage with the stripe STAGES ahead.  The
// control warp (warp 2W) is unchanged.  A row warp may run up to STAGES - 1
// stripes ahead of its column warp, so the exchange of a stripe hides
// behind that much row work, and each SM sub-partition holds four warps of
// double-float work where the single-warp form holds two.  Whether a
// stripe's row phase went native (out-of-range values) passes to the column
// warp in shared memory, written before ready[w][stage] is arrived on.
//
// Slots: a row warp's stripe j + 4 needs its stage back from stripe j + 1's
// column phase, which needs t of stripe j + 1, which the control warp forms
// only after it has taken stripe j's row partials and cluster partials out
// of their slots, so four slots remain enough.  Row warps of sub-bands past
// the matrix have no stage to wait for: they do not take part (their
// partials stay zero and wfull counts the live row warps only).
template <int W, int R, int STAGES, int BAND = kBandCols>
struct AtaxLayout64WS {
    static constexpr int kBoxBytes = R * BAND * 8;
    static constexpr int kAlign = 1024;
    static constexpr int kRing = W * STAGES * kBoxBytes;
    static constexpr int kWarpPart = kAtaxSlots * W * R * 8;               // [slot][W][R] fp64
    static constexpr int kPart = kAtaxSlots * kAtaxMaxCluster * R * 8;     // [slot][C][R] fp64
    static constexpr int kT = kAtaxSlots * (R * 8 + R * 8 + 8);
    static constexpr int kSeg = W * BAND * 8;                              // [W][BAND] fp64
    // stage_native[W][STAGES], col_issued[W] (u32), rounded to 8 bytes
    static constexpr int kFlags = ((W * STAGES + W) * 4 + 7) / 8 * 8;
    // full[W][STAGES], ready[W][STAGES], part[slot], wfull[slot], tready[slot]
    static constexpr int kBars = (2 * W * STAGES + 3 * kAtaxSlots) * 8;
    static constexpr int kTotal =
        kAlign + kRing + kWarpPart + kPart + kT + kSeg + kFlags + kBars;
};

template <int W, int R, int STAGES, int BAND = kBandCols, int NV = 0>
__global__ void __launch_bounds__((2 * W + 1) * 32, 1)
atax_cluster_f64_ws_kernel(const __grid_constant__ CUtensorMap tmap, const AtaxParams64 prm) {
    using L = AtaxLayout64WS<W, R, STAGES, BAND>;
    using Vec = double2;
    constexpr int VE = 2, LANE_COLS = BAND / 32, VPL = LANE_COLS / VE;
    constexpr int ROW_BYTES = BAND * 8;
    // The last NV of each lane's VPL column vectors take their column sums
    // in native fp64 (DFMA on the otherwise idle FP64 pipe, one chain per
    // column over the CTA's stripes); the row warp leaves those vectors as
    // doubles in the stage instead of writing their split.
    static_assert(NV >= 0 && NV < VPL, "native column vectors: 0 .. VPL - 1");
    constexpr int VS = VPL - NV;  // vectors in double-float
    static_assert(L::kBoxBytes == R * ROW_BYTES, "box size mismatch");
    static_assert(VPL == 2 || VPL == 4, "a sub-band of 128 or 256 columns");
    static_assert(kAtaxMaxCluster * R <= 64, "the control warp sends two values a lane");

    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_raw + shared_align_pad<L::kAlign>(smem_raw);
    unsigned char *ring = smem;
    double *wpart = reinterpret_cast<double *>(smem + L::kRing);  // [slot][W][R]
    double *part = wpart + kAtaxSlots * W * R;                    // [slot][kMax][R]
    double *tvec = part + kAtaxSlots * kAtaxMaxCluster * R;       // [slot][R]
    float2 *tsplit = reinterpret_cast<float2 *>(tvec + kAtaxSlots * R);  // [slot][R]
    uint32_t *tflag = reinterpret_cast<uint32_t *>(tsplit + kAtaxSlots * R);  // [slot]
    double *segs = reinterpret_cast<double *>(reinterpret_cast<unsigned char *>(tvec) + L::kT);
    uint32_t *stage_native = reinterpret_cast<uint32_t *>(
        reinterpret_cast<unsigned char *>(segs) + L::kSeg);        // [W][STAGES]
    uint32_t *col_issued = stage_native + W * STAGES;              // [W]
    uint64_t *full_bar = reinterpret_cast<uint64_t *>(
        smem + L::kRing + L::kWarpPart + L::kPart + L::kT + L::kSeg + L::kFlags);
    uint64_t *ready_bar = full_bar + W * STAGES;
    uint64_t *part_bar = ready_bar + W * STAGES;
    uint64_t *wfull_bar = part_bar + kAtaxSlots;
    uint64_t *tready_bar = wfull_bar + kAtaxSlots;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t crank = cluster_rank(), csize = cluster_size();
    const int64_t cl = cluster_id();
    const int64_t s0 = cl * prm.stripes / prm.clusters;
    const int64_t ns = (cl + 1) * prm.stripes / prm.clusters - s0;

    // Sub-bands of this CTA inside the matrix (at least one: C = ceil(bands / W)).
    const int64_t live_left = prm.bands - (int64_t)crank * W;
    const int nlive = live_left >= W ? W : (int)live_left;
    if (threadIdx.x == 0) {
        for (int i = 0; i < W * STAGES; ++i) {
            mbar_init(smem_u32(&full_bar[i]), 1);
            mbar_init(smem_u32(&ready_bar[i]), 1);
        }
        for (int i = 0; i < kAtaxSlots; ++i) {
            mbar_init(smem_u32(&part_bar[i]), 1);
            mbar_init(smem_u32(&wfull_bar[i]), nlive);
            mbar_init(smem_u32(&tready_bar[i]), 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    // Row partials of sub-bands past the matrix stay zero; only live row
    // warps arrive on wfull (a row warp with nothing to wait for would run
    // ahead and arrive for later stripes).
    for (int i = threadIdx.x; i < kAtaxSlots * W * R; i += blockDim.x) wpart[i] = 0.0;
    // Every CTA's barriers exist before any peer sends to them.
    cluster_sync();
    // A programmatic dependent of the kernel before it (see atax_cluster_kernel).
    pdl_wait();
    pdl_launch_dependents();

    // ---------------------------------------------------- control warp ----
    if (warp == 2 * W) {
        bool ok = true;
        for (int64_t j = 0; j <= ns; ++j) {
            if (j < ns && lane == 0)
                mbar_arrive_expect_tx(smem_u32(&part_bar[j % kAtaxSlots]), csize * R * 8u);
            if (j >= 1) {
                // t of stripe j - 1: the C partials of each row in CTA-rank order.
                const int64_t jp = j - 1;
                const int bp = (int)(jp % kAtaxSlots);
                if (!mbar_wait_cluster_bounded(smem_u32(&part_bar[bp]),
                                               (uint32_t)(jp / kAtaxSlots) & 1u))
                    ok = false;
                bool bad = false;
                if (lane < R) {
                    double tt = part[(bp * kAtaxMaxCluster) * R + lane];
                    for (uint32_t k = 1; k < csize; ++k)
                        tt += part[(bp * kAtaxMaxCluster + k) * R + lane];
                    float th, tl;
                    split_f64(tt, th, tl);
                    bad = !f64e_in_range(tt);
                    tvec[bp * R + lane] = tt;
                    tsplit[bp * R + lane] = make_float2(th, tl);
                }
                const bool any_bad = __any_sync(0xffffffffu, bad);
                if (lane == 0) tflag[bp] = any_bad ? 1u : 0u;
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&tready_bar[bp]));
            }
            if (j < ns) {
                // The CTA's partial of each row (warp order), sent to every
                // CTA of the cluster (this one included) into slot [b][crank].
                const int b = (int)(j % kAtaxSlots);
                if (ok && !mbar_wait_bounded(smem_u32(&wfull_bar[b]),
                                             (uint32_t)(j / kAtaxSlots) & 1u))
                    ok = false;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int idx = lane + 32 * h;
                    if (idx < (int)(csize * R)) {
                        const int i = idx % R;
                        const uint32_t peer = (uint32_t)idx / R;
                        const double *wp = wpart + b * W * R;
                        double cp = wp[i];
#pragma unroll
                        for (int w = 1; w < W; ++w) cp += wp[w * R + i];
                        const uint32_t slot_addr =
                            smem_u32(&part[(b * kAtaxMaxCluster + crank) * R + i]);
                        st_async_f64(peer_addr(slot_addr, peer), cp,
                                     peer_addr(smem_u32(&part_bar[b]), peer));
                    }
                }
            }
        }
        // No CTA leaves while a peer may still write into its shared memory.
        cluster_sync();
        return;
    }

    const bool is_row = warp < W;
    const int sbw = is_row ? warp : warp - W;       // this CTA's sub-band of the pair
    const int64_t sb = (int64_t)crank * W + sbw;    // this pair's sub-band
    const bool live = sb < prm.bands;
    const int64_t col0 = sb * BAND;

    uint64_t pol = 0;
    auto issue = [&](int64_t j) {
        const int slot = sbw * STAGES + (int)(j % STAGES);
        const uint32_t fb = smem_u32(&full_bar[slot]);
        mbar_arrive_expect_tx(fb, L::kBoxBytes);
        tma_load_2d(smem_u32(ring + (size_t)slot * L::kBoxBytes), &tmap, (int)col0,
                    (int)((s0 + j) * R), fb, pol);
    };
    // Elements re-read from global memory by the native fallbacks.
    auto a_at = [&](int64_t row, int64_t col) -> double {
        return (row < prm.M && col < prm.N) ? prm.A[row * prm.lda + col] : 0.0;
    };
    const int64_t prologue = live ? (ns < STAGES ? ns : STAGES) : 0;

    if (is_row) {
        // ---------------------------------------------------- row warps ----
        // x of this sub-band, split once; its range checked once.
        float2 xh2[VPL], xl2[VPL];
        bool x_bad = false;
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
            float h[VE], l[VE];
#pragma unroll
            for (int e = 0; e < VE; ++e) {
                const int64_t col = col0 + lane_col<double>(v, lane, e);
                const double xv = (live && col < prm.N) ? prm.x[col] : 0.0;
                split_f64(xv, h[e], l[e]);
                x_bad |= !f64e_in_range(xv);
            }
            xh2[v] = make_float2(h[0], h[1]);
            xl2[v] = make_float2(l[0], l[1]);
        }
        const bool warp_x_bad = __any_sync(0xffffffffu, x_bad);
        if (live && lane == 0) {
            pol = policy_evict_first();
            for (int64_t j = 0; j < prologue; ++j) issue(j);
        }
        bool ok = true;
        int64_t confirmed = 0;  // boxes of this sub-band seen landed, in stripe order
        const int perm = butterfly_row<R>(lane);
        for (int64_t j = 0; live && j < ns; ++j) {
            const int b = (int)(j % kAtaxSlots);
            double *wp = wpart + (b * W + sbw) * R;
            const int slot = sbw * STAGES + (int)(j % STAGES);
            if (live) {
                if (ok) {
                    ok = mbar_wait_bounded(smem_u32(&full_bar[slot]),
                                           (uint32_t)(j / STAGES) & 1u);
                    if (ok) confirmed = j + 1;
                }
                unsigned char *box = ring + (size_t)slot * L::kBoxBytes;
                const int64_t row0 = (s0 + j) * R;
                DF q[R];
                uint32_t spanv[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                for (int i = 0; i < R; ++i) {
                    // Slot i of this lane is row i ^ perm (warp_rows_reduce_df_perm).
                    const int ri = i ^ perm;
                    Vec *rowp = reinterpret_cast<Vec *>(box + (size_t)ri * ROW_BYTES);
                    Vec a[VPL];
#pragma unroll
                    for (int v = 0; v < VPL; ++v) a[v] = rowp[v * 32 + lane];
                    DF2 qp[VPL];
#pragma unroll
                    for (int v = 0; v < VPL; ++v) {
                        float ah0, al0, ah1, al1;
                        split_f64(a[v].x, ah0, al0);
                        split_f64(a[v].y, ah1, al1);
                        spanv[v] = __vimax3_u32(spanv[v], f64e_range_key(a[v].x),
                                                f64e_range_key(a[v].y));
                        const float2 ah = make_float2(ah0, ah1), al = make_float2(al0, al1);
                        df_prod2(ah, al, xh2[v], xl2[v], qp[v].s, qp[v].c);
                        // The column warp reads the split, not the double
                        // (except in its native vectors).
                        if (v < VS)
                            reinterpret_cast<float4 *>(rowp)[v * 32 + lane] =
                                make_float4(ah0, ah1, al0, al1);
                    }
                    DF2 h;
                    if constexpr (VPL == 4)
                        h = df_add2(df_add2(qp[0], qp[1]), df_add2(qp[2], qp[3]));
                    else
                        h = df_add2(qp[0], qp[1]);
                    DF lo, hi;
                    lo.s = h.s.x;
                    lo.c = h.c.x;
                    hi.s = h.s.y;
                    hi.c = h.c.y;
                    q[i] = df_add(lo, hi);
                }
                uint32_t span;
                if constexpr (VPL == 4)
                    span = max(max(spanv[0], spanv[1]), max(spanv[2], spanv[3]));
                else
                    span = max(spanv[0], spanv[1]);
                bool native = warp_x_bad;
                if (!native && __any_sync(0xffffffffu, span >= kF64eRangeSpan)) {
                    // Exact re-check from global memory: zeros pass.
                    bool bad = false;
#pragma unroll
                    for (int i = 0; i < R; ++i)
#pragma unroll
                        for (int v = 0; v < VPL; ++v)
#pragma unroll
                            for (int e = 0; e < VE; ++e)
                                bad |= !f64e_in_range(
                                    a_at(row0 + i, col0 + lane_col<double>(v, lane, e)));
                    native = __any_sync(0xffffffffu, bad);
                }
                if (!native) {
                    warp_rows_reduce_df_perm<R>(q);
                    if (butterfly_writer<R>(lane)) wp[butterfly_row<R>(lane)] = df_to_double(q[0]);
                } else {
                    double qd[R];
#pragma unroll
                    for (int i = 0; i < R; ++i) {
                        double dot = 0.0;
#pragma unroll
                        for (int v = 0; v < VPL; ++v)
#pragma unroll
                            for (int e = 0; e < VE; ++e) {
                                const int64_t col = col0 + lane_col<double>(v, lane, e);
                                const double xv = col < prm.N ? prm.x[col] : 0.0;
                                dot = fma(a_at(row0 + i, col), xv, dot);
                            }
                        qd[i] = dot;
                    }
                    warp_rows_reduce<R>(qd, lane);
                    if (butterfly_writer<R>(lane)) wp[butterfly_row<R>(lane)] = qd[0];
                }
                if (lane == 0) stage_native[slot] = native ? 1u : 0u;
            }
            // The partials and the split are written: release them to the
            // control warp and to this sub-band's column warp.  The column
            // warp refills the stage by TMA after it, so the split's
            // generic writes are ordered before that async-proxy write here.
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(smem_u32(&wfull_bar[b]));
                mbar_arrive(smem_u32(&ready_bar[slot]));
            }
        }
        // The column warps have recorded how many boxes they issued.
        named_barrier(1, 2 * W * 32);
        // After a timeout, boxes issued but never seen landed must land
        // before the CTA exits (bounded).
        if (live && lane == 0) {
            const int64_t issued = prologue + (int64_t)col_issued[sbw];
            for (int64_t kk = confirmed; kk < issued; ++kk)
                mbar_wait_bounded(smem_u32(&full_bar[sbw * STAGES + (int)(kk % STAGES)]),
                                  (uint32_t)(kk / STAGES) & 1u);
        }
    } else {
        // ------------------------------------------------- column warps ----
        double *segp = segs + sbw * BAND;  // this sub-band's fp64 column sums
#pragma unroll
        for (int v = 0; v < VPL; ++v)
#pragma unroll
            for (int e = 0; e < VE; ++e) segp[lane_col<double>(v, lane, e)] = 0.0;
        if (live && lane == 0) pol = policy_evict_first();
        DF2 grp2[VPL];
#pragma unroll
        for (int v = 0; v < VPL; ++v) grp2[v].s = grp2[v].c = make_float2(0.f, 0.f);
        double nacc[NV > 0 ? NV : 1][VE];  // native column sums (vectors VS ..)
#pragma unroll
        for (int v = 0; v < (NV > 0 ? NV : 1); ++v) nacc[v][0] = nacc[v][1] = 0.0;
        int ngrp = 0;
        uint32_t nissued = 0;
        bool ok = true;
        for (int64_t jp = 0; live && jp < ns; ++jp) {
            const int bp = (int)(jp % kAtaxSlots);
            const int slot = sbw * STAGES + (int)(jp % STAGES);
            if (!mbar_wait_bounded(smem_u32(&tready_bar[bp]), (uint32_t)(jp / kAtaxSlots) & 1u))
                ok = false;
            if (ok && !mbar_wait_bounded(smem_u32(&ready_bar[slot]),
                                         (uint32_t)(jp / STAGES) & 1u))
                ok = false;
            const unsigned char *box = ring + (size_t)slot * L::kBoxBytes;
            if (tflag[bp] == 0u && stage_native[slot] == 0u) {
                DF2 tacc2[VPL];
#pragma unroll
                for (int i = 0; i < R; ++i) {
                    const float2 t = tsplit[bp * R + i];
                    const float2 th2 = make_float2(t.x, t.x), tl2 = make_float2(t.y, t.y);
                    const float4 *rowp =
                        reinterpret_cast<const float4 *>(box + (size_t)i * ROW_BYTES);
                    if constexpr (NV > 0) {
                        const double td = tvec[bp * R + i];
                        const double2 *rowd = reinterpret_cast<const double2 *>(rowp);
#pragma unroll
                        for (int v = VS; v < VPL; ++v) {
                            const double2 a = rowd[v * 32 + lane];
                            nacc[v - VS][0] = fma(a.x, td, nacc[v - VS][0]);
                            nacc[v - VS][1] = fma(a.y, td, nacc[v - VS][1]);
                        }
                    }
#pragma unroll
                    for (int v = 0; v < VS; ++v) {
                        const float4 f = rowp[v * 32 + lane];
                        float2 p0, p1;
                        df_prod2(make_float2(f.x, f.y), make_float2(f.z, f.w), th2, tl2, p0,
                                 p1);
                        if (i == 0) {
                            tacc2[v].s = p0;
                            tacc2[v].c = p1;
                        } else {
                            df_acc2(tacc2[v], p0, p1);
                        }
                    }
                }
#pragma unroll
                for (int v = 0; v < VS; ++v) grp2[v] = df_add2(grp2[v], tacc2[v]);
            } else {
                // Native fp64 from global memory (the shared copy holds the
                // split, which is garbage for values out of range).
                const int64_t row0 = (s0 + jp) * R;
#pragma unroll
                for (int v = 0; v < VPL; ++v)
#pragma unroll
                    for (int e = 0; e < VE; ++e) {
                        const int c = lane_col<double>(v, lane, e);
                        double acc = 0.0;
#pragma unroll
                        for (int i = 0; i < R; ++i)
                            acc = fma(a_at(row0 + i, col0 + c), tvec[bp * R + i], acc);
                        segp[c] += acc;
                    }
            }
            if (++ngrp == kGroupTiles || jp == ns - 1) {
#pragma unroll
                for (int v = 0; v < VS; ++v)
#pragma unroll
                    for (int e = 0; e < VE; ++e) {
                        DF x;
                        x.s = e == 0 ? grp2[v].s.x : grp2[v].s.y;
                        x.c = e == 0 ? grp2[v].c.x : grp2[v].c.y;
                        segp[lane_col<double>(v, lane, e)] += df_to_double(x);
                    }
#pragma unroll
                for (int v = 0; v < VS; ++v) grp2[v].s = grp2[v].c = make_float2(0.f, 0.f);
                ngrp = 0;
            }
            // The stage is free: refill it with the stripe STAGES ahead.
            __syncwarp();
            if (lane == 0 && ok && jp + STAGES < ns) {
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                issue(jp + STAGES);
                ++nissued;
            }
        }
        // The native columns' chains join their sums of the native stripes.
        if constexpr (NV > 0) {
#pragma unroll
            for (int v = VS; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) segp[lane_col<double>(v, lane, e)] += nacc[v - VS][e];
        }
        // This cluster's column sums of the sub-band.
        if (live) {
            __syncwarp();
            double *yw = prm.y_ws + cl * prm.N;
#pragma unroll
            for (int v = 0; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) {
                    const int c = lane_col<double>(v, lane, e);
                    if (col0 + c < prm.N) yw[col0 + c] = segp[c];
                }
        }
        if (lane == 0) col_issued[sbw] = nissued;
        named_barrier(1, 2 * W * 32);
    }
    // No CTA leaves while a peer may still write into its shared memory.
    cluster_sync();
}

}  // namespace dmv
