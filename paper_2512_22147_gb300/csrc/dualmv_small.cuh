// Small fp32 dual products (BICG, Tables 1-2) in one thread-block cluster.
//
// For a matrix of a few MiB the streaming kernel's call is latency, not
// bandwidth: one wave of one-tile CTAs, then the combine kernel, and the
// dependency between the two kernels costs as much as either.  Here one
// cluster of kSmallCluster CTAs does the whole call, with no workspace and
// no second kernel:
//   * CTA k of the cluster owns rows [k M / C, (k + 1) M / C): every q_i is
//     complete inside one CTA (a row's products summed by each lane in four
//     chains, one per element of its float4s, then across the warp by a
//     butterfly) and is kept in shared memory until the first barrier;
//   * each lane keeps the column sums of its columns over its warp's rows;
//     the warps' sums are added in warp order through shared memory, giving
//     the CTA's partial of s;
//   * after a cluster barrier, CTA k writes its q, adds the C partials of
//     its share of the columns, reading them from the peers' shared memory
//     in CTA-rank order, and writes s; a second barrier keeps every CTA's
//     shared memory alive until its peers have read it.
// Every sum has a fixed order, so results are the same bits on every call.
// Loads of A and p are plain 16-byte global loads (A and p 16-byte aligned,
// lda and N multiples of 4); lane l holds columns 4 (v 32 + l) .. + 3 for
// v < VPL, so N is at most 128 VPL.  A CTA holds at most kSmallMaxRows rows.
#pragma once

#include <cstdint>

#include "dualmv_atax.cuh"
#include "dualmv_kernels.cuh"

namespace dmv {

constexpr int kSmallCluster = 16;  // CTAs of the cluster (non-portable size)
constexpr int kSmallWarps = 8;
constexpr int kSmallMaxRows = 512;  // rows of one CTA: 8 MiB over 16 CTAs at N >= 256

template <int VPL>
struct SmallLayout {
    static constexpr int kCols = 128 * VPL;                      // most columns
    static constexpr int kWarpPart = kSmallWarps * kCols * 4;    // [W][cols] fp32
    static constexpr int kCtaPart = kCols * 4;                   // [cols] fp32
    static constexpr int kQ = kSmallMaxRows * 4;                 // [rows] fp32
    static constexpr int kTotal = kWarpPart + kCtaPart + kQ;
};

// barrier.cluster with no memory ordering: the last barrier only keeps
// every CTA's shared memory alive until its peers' reads of it have
// returned (their values are used before the peer arrives).
__device__ __forceinline__ void cluster_sync_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;\n\t"
                 "barrier.cluster.wait.aligned;" ::: "memory");
}

template <int VPL, int D>
__global__ void __launch_bounds__(kSmallWarps * 32, 1)
dualmv_small_cluster_kernel(const Params prm) {
    using L = SmallLayout<VPL>;
    extern __shared__ __align__(16) unsigned char small_smem[];
    float *wpart = reinterpret_cast<float *>(small_smem);
    float *cpart = reinterpret_cast<float *>(small_smem + L::kWarpPart);
    float *qrow = reinterpret_cast<float *>(small_smem + L::kWarpPart + L::kCtaPart);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_rank();
    const int64_t M = prm.M, N = prm.N, lda = prm.lda;
    const int64_t n4 = N / 4;
    const float *A = static_cast<const float *>(prm.A);
    const float4 *p4g = static_cast<const float4 *>(prm.p);
    const float *rg = static_cast<const float *>(prm.r);
    float *q = static_cast<float *>(prm.q);
    float *s = static_cast<float *>(prm.s);

    // A programmatic dependent of the kernel before it: launched while that
    // kernel runs, it touches global memory only once that grid is done.
    pdl_wait();
    pdl_launch_dependents();

    float4 p4[VPL], s4[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
        const int64_t c4 = (int64_t)v * 32 + lane;
        p4[v] = c4 < n4 ? p4g[c4] : make_float4(0.f, 0.f, 0.f, 0.f);
        s4[v] = make_float4(0.f, 0.f, 0.f, 0.f);
    }

    // This CTA's rows; warp w takes rows r0 + w, r0 + w + W, ...  Each warp
    // keeps D rows in flight in a register ring: the loads of row i + D W
    // are issued as soon as row i is done, so that the few SMs of the
    // cluster keep enough bytes in flight to hide the memory latency.
    const int64_t r0 = (int64_t)rank * M / kSmallCluster;
    const int64_t r1 = ((int64_t)rank + 1) * M / kSmallCluster;
    float4 buf[D][VPL];
    float rbuf[D];
    auto load_row = [&](int d, int64_t row) {
        const float4 *arow = reinterpret_cast<const float4 *>(A + row * lda);
        rbuf[d] = rg[row];
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
            const int64_t c4 = (int64_t)v * 32 + lane;
            buf[d][v] = c4 < n4 ? arow[c4] : make_float4(0.f, 0.f, 0.f, 0.f);
        }
    };
#pragma unroll
    for (int d = 0; d < D; ++d) {
        const int64_t row = r0 + warp + (int64_t)d * kSmallWarps;
        if (row < r1) load_row(d, row);
    }
    for (int64_t base = r0 + warp; base < r1; base += (int64_t)D * kSmallWarps) {
#pragma unroll
        for (int d = 0; d < D; ++d) {
            const int64_t row = base + (int64_t)d * kSmallWarps;
            if (row < r1) {
                const float ri = rbuf[d];
                // A lane's products of the row in four chains, one per
                // element of its float4s, added pairwise at the end.
                float dx = 0.f, dy = 0.f, dz = 0.f, dw = 0.f;
#pragma unroll
                for (int v = 0; v < VPL; ++v) {
                    const float4 a = buf[d][v];
                    dx = fmaf(a.x, p4[v].x, dx);
                    dy = fmaf(a.y, p4[v].y, dy);
                    dz = fmaf(a.z, p4[v].z, dz);
                    dw = fmaf(a.w, p4[v].w, dw);
                    s4[v].x = fmaf(a.x, ri, s4[v].x);
                    s4[v].y = fmaf(a.y, ri, s4[v].y);
                    s4[v].z = fmaf(a.z, ri, s4[v].z);
                    s4[v].w = fmaf(a.w, ri, s4[v].w);
                }
                const int64_t next = row + (int64_t)D * kSmallWarps;
                if (next < r1) load_row(d, next);
                float dot = (dx + dy) + (dz + dw);
#pragma unroll
                for (int off = 16; off >= 1; off >>= 1)
                    dot += __shfl_xor_sync(0xffffffffu, dot, off);
                if (lane == 0) qrow[row - r0] = dot;
            }
        }
    }

    // The warps' column sums, added in warp order: the CTA's partial of s.
#pragma unroll
    for (int v = 0; v < VPL; ++v)
        reinterpret_cast<float4 *>(wpart + warp * L::kCols)[v * 32 + lane] = s4[v];
    __syncthreads();
    for (int64_t j = threadIdx.x; j < N; j += kSmallWarps * 32) {
        float acc = wpart[j];
#pragma unroll
        for (int w = 1; w < kSmallWarps; ++w) acc += wpart[w * L::kCols + j];
        cpart[j] = acc;
    }
    // Every CTA's partial is in its shared memory before any peer reads it.
    // No global store is outstanding here, so the release is cheap; q goes
    // out after it.
    cluster_sync();
    for (int64_t i = threadIdx.x; i < r1 - r0; i += kSmallWarps * 32) q[r0 + i] = qrow[i];
    // This CTA's share of the columns: the C partials in CTA-rank order.
    const int64_t j0 = (int64_t)rank * N / kSmallCluster;
    const int64_t j1 = ((int64_t)rank + 1) * N / kSmallCluster;
    for (int64_t j = j0 + threadIdx.x; j < j1; j += kSmallWarps * 32) {
        const uint32_t local = smem_u32(&cpart[j]);
        float acc = 0.f;
#pragma unroll
        for (int c = 0; c < kSmallCluster; ++c) {
            float v;
            asm volatile("ld.shared::cluster.f32 %0, [%1];"
                         : "=f"(v)
                         : "r"(peer_addr(local, (uint32_t)c)));
            acc = c == 0 ? v : acc + v;
        }
        s[j] = acc;
    }
    // No CTA leaves while a peer may still read its shared memory.
    cluster_sync_relaxed();
}

}  // namespace dmv
