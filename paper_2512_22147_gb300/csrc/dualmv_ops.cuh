// Vector kernels of the operations built on the dual product's passes:
// GESUMMV's combination of its two row passes, and GEMVER's updates of x
// and w with the dot products of its factorised rank-2 update.  None of
// them reads A.
#pragma once

#include <cstdint>

#include "dualmv_kernels.cuh"

namespace dmv {

// GESUMMV's last step with both passes' combines folded in: row i of each
// pass from its band partials, added as the combine kernel adds them (C
// threads per row, thread y adding bands y, y + C, ..., then the C chunk
// sums in order: the combine's bits), or read from the pass's output when
// it wrote q itself; then y = alpha * t_A + beta * t_B.  Both passes have
// the same bands, so one C.  Blocks of 256
// threads over 256 / C rows; launched as a programmatic dependent of the
// second pass.
template <typename T>
__global__ void __launch_bounds__(256)
gesummv_final_kernel(const Params pa, int a_direct, const Params pb, int b_direct, int C, T *y,
                     int64_t m, T alpha, T beta) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ T chunk_a[256], chunk_b[256];
    const int R = 256 / C, xr = threadIdx.x % R, yc = threadIdx.x / R;
    const int64_t i = (int64_t)blockIdx.x * R + xr;
    const bool valid = i < m;
    auto chunk = [&](const Params &pp) -> T {
        const T *base = static_cast<const T *>(pp.q_ws) + i;
        T acc = T(0);
        int64_t k = yc;
        if (k < pp.bands) {
            acc = base[k * pp.M];
            k += C;
        }
#pragma unroll 4
        for (; k < pp.bands; k += C) acc = acc + base[k * pp.M];
        return acc;
    };
    chunk_a[threadIdx.x] = (valid && !a_direct) ? chunk(pa) : T(0);
    chunk_b[threadIdx.x] = (valid && !b_direct) ? chunk(pb) : T(0);
    __syncthreads();
    if (yc == 0 && valid) {
        T ta, tb;
        if (a_direct) {
            ta = static_cast<const T *>(pa.q)[i];
        } else {
            ta = chunk_a[xr];
            for (int c = 1; c < C; ++c) ta = ta + chunk_a[c * R + xr];
        }
        if (b_direct) {
            tb = static_cast<const T *>(pb.q)[i];
        } else {
            tb = chunk_b[xr];
            for (int c = 1; c < C; ++c) tb = tb + chunk_b[c * R + xr];
        }
        y[i] = alpha * ta + beta * tb;
    }
}

// GEMVER vector steps: x = (x + beta * s) + z, then w = w + alpha * t.
template <typename T>
__global__ void gemver_x_kernel(T *x, const T *s, const T *z, int64_t n, T beta) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        x[i] = (x[i] + beta * s[i]) + z[i];
}
template <typename T>
__global__ void gemver_w_kernel(T *w, const T *t, int64_t n, T alpha) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        w[i] = w[i] + alpha * t[i];
}

// ---- GEMVER with the rank-2 update factorised ----------------------------
//   A_hat^T y = A^T y + v1 (u1 . y) + v2 (u2 . y)
//   A_hat x   = A x   + u1 (v1 . x) + u2 (v2 . x)
// Two dot products per side (a . c and b . c), deterministic: kDotChunks
// blocks per product each take one contiguous chunk (thread k: elements
// k, k + 256, ... of the chunk, in order), sum it with TwoProduct/TwoSum in
// double, round that compensated sum once, and add the threads' sums in a
// fixed tree of plain fp64 adds; the kernel that uses the products adds the
// chunk sums in a fixed tree too.  Along any path there are at most 16
// roundings after the compensated thread sums, so the error stays within
// about 16 u sum |a_k c_k|: each term's error is inside the bar, whose
// denominator holds |u1| (|u1| . |y|) and the like.  GB300's FP64 pipe is
// narrow, so the work is spread over many SMs and the trees take one add
// per level (TwoSum trees, eight operations per level, cost the x update
// 11 us of its call at 8192^2).
constexpr int kDotChunks = 64;

__device__ __forceinline__ void two_sum_d(double a, double b, double &s, double &e) {
    s = a + b;
    const double bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

// s + cc += x y, compensated (TwoProduct, TwoSum).
__device__ __forceinline__ void dot2_step(double x, double y, double &s, double &cc) {
    const double p = x * y;
    const double pe = fma(x, y, -p);  // exact rounding error of the product
    double t, e;
    two_sum_d(s, p, t, e);
    s = t;
    cc += e + pe;
}

// The sum of v over a warp's 32 lanes in a fixed tree; lane 0 holds it.
__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
    return v;
}

// The sum of v over lanes 0-7 in a fixed tree; lane 0 holds it.
__device__ __forceinline__ double warp_sum8_d(double v) {
#pragma unroll
    for (int off = 4; off >= 1; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
    return v;
}

// The block's 256 thread sums in a fixed tree (each warp's, then the 8
// warps' in warp 0); thread 0 writes the block's sum to part[slot].
// hs: 8 doubles.
__device__ __forceinline__ void dot_block_store(double v, double *hs, double *part, int slot) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum_d(v);
    if (lane == 0) hs[warp] = v;
    __syncthreads();
    if (warp == 0) {
        v = warp_sum8_d(lane < 8 ? hs[lane] : 0.0);
        if (lane == 0) part[slot] = v;
    }
    __syncthreads();
}

// dot_block_store for two sums at once: v1 to part[slot1], v2 to
// part[slot2].  hs: 16 doubles.
__device__ __forceinline__ void dot_block_store2(double v1, double v2, double *hs, double *part,
                                                 int slot1, int slot2) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v1 = warp_sum_d(v1);
    v2 = warp_sum_d(v2);
    if (lane == 0) {
        hs[warp] = v1;
        hs[8 + warp] = v2;
    }
    __syncthreads();
    if (warp == 0) {
        v1 = warp_sum8_d(lane < 8 ? hs[lane] : 0.0);
        v2 = warp_sum8_d(lane < 8 ? hs[8 + lane] : 0.0);
        if (lane == 0) {
            part[slot1] = v1;
            part[slot2] = v2;
        }
    }
}

// Launched as a programmatic dependent of the kernel before it: waits for
// that grid before reading its inputs.
template <typename T>
__global__ void __launch_bounds__(256) dots2_partial_kernel(const T *a, const T *b, const T *c,
                                                            int64_t n, double *part) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ double hs[8];
    const int dot = blockIdx.x / kDotChunks, chunk = blockIdx.x % kDotChunks;
    const T *u = dot == 0 ? a : b;
    const int64_t k0 = chunk * n / kDotChunks, k1 = (chunk + 1) * n / kDotChunks;
    double s = 0.0, cc = 0.0;
    for (int64_t k = k0 + threadIdx.x; k < k1; k += 256)
        dot2_step((double)u[k], (double)c[k], s, cc);
    dot_block_store(s + cc, hs, part, blockIdx.x);
}

// Both dot products from their chunk sums, by every thread of a 256-thread
// block: warps 0-1 add dot 0's kDotChunks chunk sums, warps 2-3 dot 1's,
// each warp its 32 in a fixed tree, then thread d adds dot d's two warp
// sums.  dd[0], dd[1] hold the results on return.  hs: 4 doubles.
template <typename T>
__device__ __forceinline__ void dots2_final_block(const double *part, double *hs, T *dd) {
    static_assert(kDotChunks == 64, "two warps per dot product");
    const int t = threadIdx.x, warp = t >> 5;
    if (warp < 4) {
        const double v = warp_sum_d(part[t]);
        if ((t & 31) == 0) hs[warp] = v;
    }
    __syncthreads();
    if (t < 2) dd[t] = (T)(hs[2 * t] + hs[2 * t + 1]);
    __syncthreads();
}

// x = x + beta (s + v1 d0 + v2 d1) + z, d0 = u1 . y and d1 = u2 . y from
// their chunk sums (every block forms them the same way); and, in the same
// pass, the chunk sums of v1 . x and v2 . x for the new x (part_v, laid out
// as dots2_partial_kernel's).  kDotChunks blocks, block k on chunk k, each
// thread on the elements k0 + thread, k0 + thread + 256, ... in order.
// Launched as a programmatic dependent: waits for the grid before it.
template <typename T>
__global__ void __launch_bounds__(256) gemver_x2_kernel(T *x, const T *s, const T *v1,
                                                        const T *v2, const double *part_u,
                                                        const T *z, int64_t n, T beta,
                                                        double *part_v) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ T dd[2];
    __shared__ double hs[16];
    dots2_final_block<T>(part_u, hs, dd);
    const T d0 = dd[0], d1 = dd[1];
    const int chunk = blockIdx.x;
    const int64_t k0 = chunk * n / kDotChunks, k1 = (chunk + 1) * n / kDotChunks;
    double s1 = 0.0, c1 = 0.0, s2 = 0.0, c2 = 0.0;
    for (int64_t i = k0 + threadIdx.x; i < k1; i += 256) {
        const T inner = fma(v2[i], d1, fma(v1[i], d0, s[i]));
        const T xn = fma(beta, inner, x[i]) + z[i];
        x[i] = xn;
        dot2_step((double)v1[i], (double)xn, s1, c1);
        dot2_step((double)v2[i], (double)xn, s2, c2);
    }
    dot_block_store2(s1 + c1, s2 + c2, hs, part_v, chunk, kDotChunks + chunk);
}

// w = w + alpha (t + u1 e0 + u2 e1), e0 = v1 . x and e1 = v2 . x from
// their chunk sums.
template <typename T>
__global__ void __launch_bounds__(256) gemver_w2_kernel(T *w, const T *t, const T *u1, const T *u2,
                                 const double *part, int64_t n, T alpha) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ T dd[2];
    __shared__ double hs[4];
    dots2_final_block<T>(part, hs, dd);
    const T d0 = dd[0], d1 = dd[1];
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const T inner = fma(u2[i], d1, fma(u1[i], d0, t[i]));
        w[i] = fma(alpha, inner, w[i]);
    }
}

// ---- GEMVER's vector steps with the passes' combine folded in -----------
// The columns-only and rows-only passes leave their partial sums in their
// workspace, and these kernels add them (in the combine kernel's order, so
// with its bits) where they are used: GEMVER then runs five kernels instead
// of seven.

// gemver_x2_kernel with s = A^T y from the columns-only pass's partials
// (ps: that pass's parameters; s_direct: the pass wrote s itself).
template <typename T>
__global__ void __launch_bounds__(256) gemver_x3_kernel(const Params ps, int s_direct,
                                                        const double *part_u, T *x, const T *v1,
                                                        const T *v2, const T *z, int64_t n,
                                                        T beta, double *part_v) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ T dd[2];
    __shared__ double hs[16];
    dots2_final_block<T>(part_u, hs, dd);
    const T d0 = dd[0], d1 = dd[1];
    const T *sv = static_cast<const T *>(ps.s);
    const int chunk = blockIdx.x;
    const int64_t k0 = chunk * n / kDotChunks, k1 = (chunk + 1) * n / kDotChunks;
    double s1 = 0.0, c1 = 0.0, s2 = 0.0, c2 = 0.0;
    for (int64_t i = k0 + threadIdx.x; i < k1; i += 256) {
        T si;
        int64_t c_lo = 0, c_hi = 0;
        const int64_t band = i / ps.band_cols;
        if (!s_direct) band_ctas_of(ps, band, c_lo, c_hi);
        if (s_direct || c_lo == c_hi)
            si = sv[i];
        else
            si = s_segment_sum<T>(ps, band, (int)(i - band * ps.band_cols), c_lo, c_hi);
        const T inner = fma(v2[i], d1, fma(v1[i], d0, si));
        const T xn = fma(beta, inner, x[i]) + z[i];
        x[i] = xn;
        dot2_step((double)v1[i], (double)xn, s1, c1);
        dot2_step((double)v2[i], (double)xn, s2, c2);
    }
    dot_block_store2(s1 + c1, s2 + c2, hs, part_v, chunk, kDotChunks + chunk);
}

// w = w + alpha (t + u1 e0 + u2 e1) with t = A x from the rows-only pass's
// band partials, added as the combine kernel adds them: C threads per row,
// thread y adding bands y, y + C, ..., then the C chunk sums in order (pq:
// that pass's parameters; q_direct: the pass wrote t itself).  e0 = v1 . x
// and e1 = v2 . x from their chunk sums.  Blocks of 256 threads over
// 256 / C rows each.  Launched as a programmatic dependent of the pass.
template <typename T>
__global__ void __launch_bounds__(256) gemver_w3_kernel(const Params pq, int q_direct, int C,
                                                        T *w, const T *u1, const T *u2,
                                                        const double *part, int64_t m, T alpha) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ T dd[2];
    __shared__ double hs[4];
    __shared__ T chunk_sum[256];
    dots2_final_block<T>(part, hs, dd);
    const T d0 = dd[0], d1 = dd[1];
    const int R = 256 / C, xr = threadIdx.x % R, y = threadIdx.x / R;
    const int64_t i = (int64_t)blockIdx.x * R + xr;
    const bool valid = i < m;
    T acc = T(0);
    if (valid && !q_direct) {
        const T *base = static_cast<const T *>(pq.q_ws) + i;
        int64_t k = y;
        if (k < pq.bands) {
            acc = base[k * pq.M];
            k += C;
        }
#pragma unroll 4
        for (; k < pq.bands; k += C) acc = acc + base[k * pq.M];
    }
    chunk_sum[threadIdx.x] = acc;
    __syncthreads();
    if (y == 0 && valid) {
        T ti;
        if (q_direct) {
            ti = static_cast<const T *>(pq.q)[i];
        } else {
            ti = chunk_sum[xr];
            for (int yy = 1; yy < C; ++yy) ti = ti + chunk_sum[yy * R + xr];
        }
        const T inner = fma(u2[i], d1, fma(u1[i], d0, ti));
        w[i] = fma(alpha, inner, w[i]);
    }
}

}  // namespace dmv
