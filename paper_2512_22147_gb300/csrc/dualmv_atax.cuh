// ATAX (Table 1: y = A^T (A x)) with one read of A from HBM, for fp32.
//
// The second product needs all of t = A x, and t_i is complete only after
// its whole row has been read.  A thread-block cluster of C CTAs therefore
// streams the same row stripe (R rows) at once, each CTA a slice of the
// columns (W 256-column sub-bands, one per warp), and keeps the slice in
// shared memory until t of those rows is known:
//
//   1. each warp forms the partial dot products of the R rows over its
//      sub-band (warp butterfly), the W warps' partials are added in warp
//      order, and the CTA sends its R partials to every CTA of the cluster
//      with st.async into distributed shared memory; the arrival of all C
//      contributions completes a local mbarrier;
//   2. every CTA adds the C partials of each row in CTA-rank order, so all
//      of them hold bit-identical t_i;
//   3. each warp forms y_j += t_i a_ij for its columns from the copy still
//      in shared memory (tile -> group -> segment sums, as in the main
//      kernel).
// The exchange of stripe s overlaps the row work of stripe s + 1: a CTA
// waits for the partials of s only after it has sent those of s + 1, so the
// exchange latency hides behind a whole stripe.  Peers can then run up to
// three stripes ahead of a CTA's reads, so partials land in four rotating
// slots, each with its own mbarrier.  Each
// cluster owns a contiguous range of stripes and writes its column sums to
// a workspace row; a second kernel adds the clusters' rows in order.  Every
// sum has a fixed order, so results are identical run to run.
//
// Waits on mbarriers are bounded (2 s) and set the device fault word on
// timeout while keeping the control flow, so every CTA of a cluster reaches
// the same cluster barriers.  A CTA leaves only after a cluster barrier, so
// no peer writes into shared memory that is gone.
#pragma once

#include "dualmv_kernels.cuh"

namespace dmv {

struct AtaxParams {
    const float *x;
    float *y_ws;       // [clusters][N] column sums of each cluster's stripes
    int64_t M, N;
    int64_t stripes;   // ceil(M / R)
    int64_t clusters;  // clusters launched
    int64_t bands;     // ceil(N / 256) sub-bands
};

constexpr int kAtaxMaxCluster = 16;
constexpr int kAtaxSlots = 4;  // partial-sum slots (stripes in flight)

template <int W, int R, int STAGES>
struct AtaxLayout {
    static constexpr int kBoxBytes = R * kBandCols * 4;  // one warp's sub-band, R rows
    static constexpr int kAlign = 1024;
    static constexpr int kRing = W * STAGES * kBoxBytes;
    static constexpr int kWarpPart = W * R * 4;                 // [W][R]
    static constexpr int kPart = kAtaxSlots * kAtaxMaxCluster * R * 4;  // [slot][C][R]
    static constexpr int kT = 2 * R * 4;                                // [R], padded
    static constexpr int kBars = (W * STAGES + kAtaxSlots) * 8;
    static constexpr int kTotal = kAlign + kRing + kWarpPart + kPart + kT + kBars;
};

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t cluster_size() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t cluster_id() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t peer_addr(uint32_t local, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
    return r;
}
// 4 bytes into a peer's shared memory, counted on the peer's mbarrier.
__device__ __forceinline__ void st_async_f32(uint32_t raddr, float v, uint32_t rbar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];"
                 ::"r"(raddr), "r"(__float_as_uint(v)), "r"(rbar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// As mbar_wait_bounded, with cluster-scope acquire (the data came from
// other CTAs of the cluster).
__device__ __forceinline__ bool mbar_wait_cluster_bounded(uint32_t bar, uint32_t parity) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    for (;;) {
        for (int i = 0; i < 64; ++i)
            if (mbar_try_wait_cluster(bar, parity)) return true;
        if (global_ns() - t0 > kWaitTimeoutNs) {
            atomicOr(&g_fault_word, 1u);
            return false;
        }
    }
}

template <int W, int R, int STAGES>
__global__ void __launch_bounds__(W * 32, 1)
atax_cluster_kernel(const __grid_constant__ CUtensorMap tmap, const AtaxParams prm) {
    using L = AtaxLayout<W, R, STAGES>;
    constexpr int VE = 4, VPL = kLaneCols / VE;
    constexpr int ROW_BYTES = kBandCols * 4;
    static_assert(L::kBoxBytes == R * ROW_BYTES, "box size mismatch");

    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_raw + shared_align_pad<L::kAlign>(smem_raw);
    unsigned char *ring = smem;
    float *wpart = reinterpret_cast<float *>(smem + L::kRing);  // [W][R]
    float *part = wpart + W * R;                                // [slot][kMax][R]
    float *tvec = part + kAtaxSlots * kAtaxMaxCluster * R;      // [R]
    uint64_t *full_bar = reinterpret_cast<uint64_t *>(smem + L::kRing + L::kWarpPart +
                                                      L::kPart + L::kT);
    uint64_t *part_bar = full_bar + W * STAGES;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t crank = cluster_rank(), csize = cluster_size();
    const int64_t cl = cluster_id();
    const int64_t s0 = cl * prm.stripes / prm.clusters;
    const int64_t ns = (cl + 1) * prm.stripes / prm.clusters - s0;
    const int64_t sb = (int64_t)crank * W + warp;  // this warp's sub-band
    const bool live = sb < prm.bands;
    const int64_t col0 = sb * kBandCols;

    if (threadIdx.x == 0) {
        for (int i = 0; i < W * STAGES; ++i) mbar_init(smem_u32(&full_bar[i]), 1);
        for (int i = 0; i < kAtaxSlots; ++i) mbar_init(smem_u32(&part_bar[i]), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    // Every CTA's barriers exist before any peer sends to them.
    cluster_sync();
    // A programmatic dependent of the kernel before it: its launch and the
    // set-up above overlap that kernel; nothing in global memory is touched
    // before that grid has completed.  The sum kernel after it may launch.
    pdl_wait();
    pdl_launch_dependents();

    float xv[kLaneCols];
#pragma unroll
    for (int v = 0; v < VPL; ++v)
#pragma unroll
        for (int e = 0; e < VE; ++e) {
            const int64_t col = col0 + lane_col<float>(v, lane, e);
            xv[v * VE + e] = (live && col < prm.N) ? prm.x[col] : 0.f;
        }

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

    float grp[kLaneCols], seg[kLaneCols];
#pragma unroll
    for (int e = 0; e < kLaneCols; ++e) grp[e] = seg[e] = 0.f;
    int ngrp = 0;
    bool ok = true;
    int64_t confirmed = 0;  // boxes of this warp seen landed, in stripe order

    for (int64_t j = 0; j <= ns; ++j) {
        const int b = (int)(j % kAtaxSlots);
        if (j < ns) {
            if (threadIdx.x == 0)
                mbar_arrive_expect_tx(smem_u32(&part_bar[b]), csize * R * 4u);
            // 1. Partial dot products of stripe j's rows over this sub-band.
            float qp[R];
#pragma unroll
            for (int i = 0; i < R; ++i) qp[i] = 0.f;
            if (live) {
                const int slot = warp * STAGES + (int)(j % STAGES);
                if (ok) {
                    ok = mbar_wait_bounded(smem_u32(&full_bar[slot]),
                                           (uint32_t)(j / STAGES) & 1u);
                    if (ok) confirmed = j + 1;
                }
                const unsigned char *box = ring + (size_t)slot * L::kBoxBytes;
#pragma unroll
                for (int i = 0; i < R; ++i) {
                    const float4 *rowp = reinterpret_cast<const float4 *>(box + i * ROW_BYTES);
                    float dot = 0.f;
#pragma unroll
                    for (int v = 0; v < VPL; ++v) {
                        const float4 a = rowp[v * 32 + lane];
                        dot = fmaf(a.x, xv[v * VE + 0], dot);
                        dot = fmaf(a.y, xv[v * VE + 1], dot);
                        dot = fmaf(a.z, xv[v * VE + 2], dot);
                        dot = fmaf(a.w, xv[v * VE + 3], dot);
                    }
                    qp[i] = dot;
                }
            }
            warp_rows_reduce<R>(qp, lane);
            if (butterfly_writer<R>(lane)) wpart[warp * R + butterfly_row<R>(lane)] = qp[0];
        }
        // (Also when j == ns: every warp is past its reads of t before t is
        // rewritten below.)
        named_barrier(1, W * 32);
        if (j < ns && threadIdx.x < (int)(csize * R)) {
            // 2. The CTA's partial of each row (warp order), sent to every
            // CTA of the cluster (this one included) into slot [b][crank].
            const int i = threadIdx.x % R;
            const uint32_t peer = (uint32_t)threadIdx.x / R;
            float cp = 0.f;
#pragma unroll
            for (int w = 0; w < W; ++w) cp += wpart[w * R + i];
            const uint32_t slot_addr = smem_u32(&part[(b * kAtaxMaxCluster + crank) * R + i]);
            st_async_f32(peer_addr(slot_addr, peer), cp, peer_addr(smem_u32(&part_bar[b]), peer));
        }
        if (j >= 1) {
            // 3. Stripe j - 1: all C partials are here; t in CTA-rank order.
            const int64_t jp = j - 1;
            const int bp = (int)(jp % kAtaxSlots);
            if (!mbar_wait_cluster_bounded(smem_u32(&part_bar[bp]),
                                           (uint32_t)(jp / kAtaxSlots) & 1u))
                ok = false;
            if (threadIdx.x < R) {
                float tt = 0.f;
                for (uint32_t k = 0; k < csize; ++k)
                    tt += part[(bp * kAtaxMaxCluster + k) * R + threadIdx.x];
                tvec[threadIdx.x] = tt;
            }
            named_barrier(1, W * 32);
            // 4. Column sums of stripe j - 1 from its copy in shared memory.
            if (live) {
                const int slot = warp * STAGES + (int)(jp % STAGES);
                const unsigned char *box = ring + (size_t)slot * L::kBoxBytes;
                float tacc[kLaneCols];
#pragma unroll
                for (int e = 0; e < kLaneCols; ++e) tacc[e] = 0.f;
#pragma unroll
                for (int i = 0; i < R; ++i) {
                    const float ti = tvec[i];
                    const float4 *rowp = reinterpret_cast<const float4 *>(box + i * ROW_BYTES);
#pragma unroll
                    for (int v = 0; v < VPL; ++v) {
                        const float4 a = rowp[v * 32 + lane];
                        tacc[v * VE + 0] = fmaf(a.x, ti, tacc[v * VE + 0]);
                        tacc[v * VE + 1] = fmaf(a.y, ti, tacc[v * VE + 1]);
                        tacc[v * VE + 2] = fmaf(a.z, ti, tacc[v * VE + 2]);
                        tacc[v * VE + 3] = fmaf(a.w, ti, tacc[v * VE + 3]);
                    }
                }
#pragma unroll
                for (int e = 0; e < kLaneCols; ++e) grp[e] += tacc[e];
                if (++ngrp == kGroupTiles) {
#pragma unroll
                    for (int e = 0; e < kLaneCols; ++e) {
                        seg[e] += grp[e];
                        grp[e] = 0.f;
                    }
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
        float *yw = prm.y_ws + cl * prm.N;
#pragma unroll
        for (int v = 0; v < VPL; ++v)
#pragma unroll
            for (int e = 0; e < VE; ++e) {
                const int64_t col = col0 + lane_col<float>(v, lane, e);
                if (col < prm.N) yw[col] = seg[v * VE + e] + grp[v * VE + e];
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

// y = sum over clusters of their column sums, in cluster order.
template <typename T>
__global__ void __launch_bounds__(256) atax_sum_kernel(const T *y_ws, T *y, int64_t N,
                                                       int64_t clusters) {
    // A programmatic dependent of the cluster kernel: waits for its grid.
    pdl_launch_dependents();
    pdl_wait();
    const int64_t threads = (int64_t)gridDim.x * blockDim.x;
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < N; j += threads) {
        T acc = T(0);
        for (int64_t c = 0; c < clusters; ++c) acc += y_ws[c * N + j];
        y[j] = acc;
    }
}

}  // namespace dmv
