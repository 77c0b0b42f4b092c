// Read-only bandwidth probe: the ceiling a kernel that only streams A can
// reach on this GPU, measured beside the copy bandwidth (which moves every
// byte twice, once read and once written).  Not part of the method.
//
// A grid-stride loop of 16-byte loads, eight independent loads in flight
// per thread and a full SM of threads, so the memory system, not latency,
// bounds it.  Loads are read-only and bypass L1.  Each thread folds what it read into
// one word; the block's words are folded and xor-ed into *out, so the
// loads cannot be removed (the value itself means nothing).
#pragma once

#include <cstdint>

#include "dualmv_atax.cuh"
#include "dualmv_kernels.cuh"

namespace dmv {

constexpr int kProbeThreads = 512;
constexpr int kProbeUnroll = 8;

__device__ __forceinline__ uint4 ld_stream16(const uint4 *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__global__ void __launch_bounds__(kProbeThreads)
read_probe_kernel(const uint4 *__restrict__ src, int64_t n16, uint32_t *out) {
    const int64_t stride = (int64_t)gridDim.x * kProbeThreads;
    int64_t i = (int64_t)blockIdx.x * kProbeThreads + threadIdx.x;
    uint32_t acc = 0;
    for (; i + (kProbeUnroll - 1) * stride < n16; i += kProbeUnroll * stride) {
        uint4 v[kProbeUnroll];
#pragma unroll
        for (int k = 0; k < kProbeUnroll; ++k) v[k] = ld_stream16(src + i + k * stride);
#pragma unroll
        for (int k = 0; k < kProbeUnroll; ++k) acc ^= v[k].x ^ v[k].y ^ v[k].z ^ v[k].w;
    }
    for (; i < n16; i += stride) {
        const uint4 v = ld_stream16(src + i);
        acc ^= v.x ^ v.y ^ v.z ^ v.w;
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) acc ^= __shfl_xor_sync(0xffffffffu, acc, off);
    if ((threadIdx.x & 31) == 0) atomicXor(out, acc);
}

// Wait self-test, for the failure-detection tests: thread 0 waits for phase
// 0 of an mbarrier that nothing arrives on, through the bounded waits of the
// streaming kernels (CTA scope) or of the cluster kernels (cluster scope;
// this CTA is a cluster of one).  After kWaitTimeoutNs the wait sets the
// device fault word and returns false, and the kernel exits as the
// library's kernels do after a timeout.  *waited = 1 if the wait returned
// true (nothing can make it), 0 if it ran out.
__global__ void __launch_bounds__(32) wait_selftest_kernel(int cluster_scope, int32_t *waited) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncwarp();
    if (threadIdx.x == 0) {
        const bool ok = cluster_scope ? mbar_wait_cluster_bounded(smem_u32(&bar), 0u)
                                      : mbar_wait_bounded(smem_u32(&bar), 0u);
        *waited = ok ? 1 : 0;
    }
}

}  // namespace dmv
