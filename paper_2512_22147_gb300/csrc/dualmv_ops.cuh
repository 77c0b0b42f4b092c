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
// blocks per product each take one contiguous chunk (thread k of a block of
// T threads: elements k, k + T, ... of the chunk, in order).  A thread with at most
// kPlainPerThread elements sums them with fp64 FMAs; one with more sums
// them compensated (TwoProduct/TwoSum) and rounds that once.  The block
// adds its threads' sums in a fixed tree of plain fp64 adds, and the kernel
// that uses the products adds the chunk sums in a fixed tree too.  Along
// any path there are at most 80 roundings, so a product errs by at most
// about 80 u sum |a_k c_k| (u = 2^-53, 8.9e-15): each term's error is
// inside the bar, whose denominator holds |u1| (|u1| . |y|) and the like.
// GB300's FP64 pipe is narrow, so the work is spread over many SMs, the
// trees take one add per level (TwoSum trees, eight operations per level,
// cost the x update 11 us of its call at 8192^2), and compensation is kept
// for the long per-thread sums it is needed for.
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

// Elements per thread above which a thread's share of a dot product is
// summed compensated.
constexpr int64_t kPlainPerThread = 64;

// A thread's share of a dot product (see above): plain FMAs or
// compensated, the same for every thread of a block.
struct ThreadDot {
    double s = 0.0, c = 0.0;
    __device__ __forceinline__ void add(double x, double y, bool comp) {
        if (comp)
            dot2_step(x, y, s, c);
        else
            s = fma(x, y, s);
    }
    __device__ __forceinline__ double value() const { return s + c; }
};

// Whether a chunk of `len` elements over `threads` threads takes
// compensated thread sums.
__device__ __forceinline__ bool dot_compensated(int64_t len, int threads = 256) {
    return len > threads * kPlainPerThread;
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

// The block's NW * 32 thread sums in a fixed tree (each warp's, then the
// NW warps' in warp 0); thread 0 writes the block's sum to part[slot].
// hs: NW doubles.
template <int NW>
__device__ __forceinline__ void dot_block_store(double v, double *hs, double *part, int slot) {
    static_assert(NW >= 1 && NW <= 32 && (NW & (NW - 1)) == 0, "a power of two of warps");
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum_d(v);
    if (lane == 0) hs[warp] = v;
    __syncthreads();
    if (warp == 0) {
        v = lane < NW ? hs[lane] : 0.0;
#pragma unroll
        for (int off = NW / 2; off >= 1; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
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

// 2 kDotChunks blocks of kDotThreads threads: block d kDotChunks + k sums
// chunk k of dot product d (a . c, then b . c) into part[d kDotChunks + k].
// Launched as a programmatic dependent of the kernel before it: waits for
// that grid before reading its inputs, and only then lets its own
// dependents launch, so that every grid before it has completed when they
// start (GEMVER's columns pass relies on that; see Params::pdl_late).  Its
// blocks are small (128 threads, under 48 registers each) so that one fits
// on an SM beside a CTA of that pass.
constexpr int kDotThreads = 128;

template <typename T>
__global__ void __launch_bounds__(kDotThreads) dots2_partial_kernel(const T *a, const T *b,
                                                                    const T *c, int64_t n,
                                                                    double *part) {
    pdl_wait();
    pdl_launch_dependents();
    __shared__ double hs[kDotThreads / 32];
    const int dot = blockIdx.x / kDotChunks, chunk = blockIdx.x % kDotChunks;
    const T *u = dot == 0 ? a : b;
    const int64_t k0 = chunk * n / kDotChunks, k1 = (chunk + 1) * n / kDotChunks;
    const bool comp = dot_compensated(k1 - k0, kDotThreads);
    ThreadDot d;
    for (int64_t k = k0 + threadIdx.x; k < k1; k += kDotThreads)
        d.add((double)u[k], (double)c[k], comp);
    dot_block_store<kDotThreads / 32>(d.value(), hs, part, blockIdx.x);
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
    const bool comp = dot_compensated(k1 - k0);
    ThreadDot e1, e2;
    for (int64_t i = k0 + threadIdx.x; i < k1; i += 256) {
        const T inner = fma(v2[i], d1, fma(v1[i], d0, s[i]));
        const T xn = fma(beta, inner, x[i]) + z[i];
        x[i] = xn;
        e1.add((double)v1[i], (double)xn, comp);
        e2.add((double)v2[i], (double)xn, comp);
    }
    dot_block_store2(e1.value(), e2.value(), hs, part_v, chunk, kDotChunks + chunk);
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
// (ps: that pass's parameters; s_direct: the pass wrote s itself).  Each
// thread reads its first element's operands before the block forms d0 and
// d1, and the next element's before it works on the current one, so the
// loads overlap the chunk-sum tree and the arithmetic.
template <typename T>
__global__ void __launch_bounds__(256) gemver_x3_kernel(const Params ps, int s_direct,
                                                        const double *part_u, T *x, const T *v1,
                                                        const T *v2, const T *z, int64_t n,
                                                        T beta, double *part_v) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ T dd[2];
    __shared__ double hs[16];
    const T *sv = static_cast<const T *>(ps.s);
    const int chunk = blockIdx.x;
    const int64_t k0 = chunk * n / kDotChunks, k1 = (chunk + 1) * n / kDotChunks;
    struct Operands {
        T s, v1, v2, x, z;
    };
    // Element i's operands (zeros past the chunk).
    auto load = [&](int64_t i) {
        Operands o{T(0), T(0), T(0), T(0), T(0)};
        if (i < k1) {
            int64_t c_lo = 0, c_hi = 0;
            const int64_t band = i / ps.band_cols;
            if (!s_direct) band_ctas_of(ps, band, c_lo, c_hi);
            if (s_direct || c_lo == c_hi)
                o.s = sv[i];
            else
                o.s = s_segment_sum<T>(ps, band, (int)(i - band * ps.band_cols), c_lo, c_hi);
            o.v1 = v1[i];
            o.v2 = v2[i];
            o.x = x[i];
            o.z = z[i];
        }
        return o;
    };
    int64_t i = k0 + threadIdx.x;
    Operands cur = load(i);
    dots2_final_block<T>(part_u, hs, dd);
    const T d0 = dd[0], d1 = dd[1];
    const bool comp = dot_compensated(k1 - k0);
    ThreadDot e1, e2;
    for (; i < k1; i += 256) {
        const Operands nxt = load(i + 256);
        const T inner = fma(cur.v2, d1, fma(cur.v1, d0, cur.s));
        const T xn = fma(beta, inner, cur.x) + cur.z;
        x[i] = xn;
        e1.add((double)cur.v1, (double)xn, comp);
        e2.add((double)cur.v2, (double)xn, comp);
        cur = nxt;
    }
    dot_block_store2(e1.value(), e2.value(), hs, part_v, chunk, kDotChunks + chunk);
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
    // Row i's own operands, read before the block forms e0 and e1 so that
    // their loads overlap the chunk-sum tree.
    T ti = T(0), u1i = T(0), u2i = T(0), wi = T(0);
    if (y == 0 && valid) {
        u1i = u1[i];
        u2i = u2[i];
        wi = w[i];
        if (q_direct) ti = static_cast<const T *>(pq.q)[i];
    }
    // Its barriers also put every chunk_sum write before the reads below.
    dots2_final_block<T>(part, hs, dd);
    const T d0 = dd[0], d1 = dd[1];
    if (y == 0 && valid) {
        if (!q_direct) {
            ti = chunk_sum[xr];
            for (int yy = 1; yy < C; ++yy) ti = ti + chunk_sum[yy * R + xr];
        }
        const T inner = fma(u2i, d1, fma(u1i, d0, ti));
        w[i] = fma(alpha, inner, wi);
    }
}

}  // namespace dmv
