// Vector kernels of the operations built on the dual product's passes:
// GESUMMV's combination of its two row passes, and GEMVER's updates of x
// and w with the dot products of its factorised rank-2 update.  None of
// them reads A.
#pragma once

#include <cstdint>

namespace dmv {

template <typename T>
__global__ void axpby_kernel(const T *t, T *y, int64_t n, T alpha, T beta) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        y[i] = alpha * t[i] + beta * y[i];
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
// Two dot products per side (a . c and b . c), deterministic and
// compensated: kDotChunks blocks per product each take one contiguous chunk
// (thread k: elements k, k + 256, ... of the chunk, in order), sum it with
// TwoProduct/TwoSum in double, and add their threads' sums in a fixed
// pairwise tree; a second kernel adds the chunks in order.  GB300's FP64
// pipe is narrow, so the work is spread over many SMs.
constexpr int kDotChunks = 64;

__device__ __forceinline__ void two_sum_d(double a, double b, double &s, double &e) {
    s = a + b;
    const double bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

template <typename T>
__global__ void __launch_bounds__(256) dots2_partial_kernel(const T *a, const T *b, const T *c,
                                                            int64_t n, double *part) {
    __shared__ double hs[256], hc[256];
    const int dot = blockIdx.x / kDotChunks, chunk = blockIdx.x % kDotChunks;
    const T *u = dot == 0 ? a : b;
    const int64_t k0 = chunk * n / kDotChunks, k1 = (chunk + 1) * n / kDotChunks;
    double s = 0.0, cc = 0.0;
    for (int64_t k = k0 + threadIdx.x; k < k1; k += 256) {
        const double x = (double)u[k], y = (double)c[k];
        const double p = x * y;
        const double pe = fma(x, y, -p);  // exact rounding error of the product
        double t, e;
        two_sum_d(s, p, t, e);
        s = t;
        cc += e + pe;
    }
    hs[threadIdx.x] = s;
    hc[threadIdx.x] = cc;
    __syncthreads();
    for (int h = 128; h >= 1; h >>= 1) {
        if ((int)threadIdx.x < h) {
            double t, e;
            two_sum_d(hs[threadIdx.x], hs[threadIdx.x + h], t, e);
            hc[threadIdx.x] += hc[threadIdx.x + h] + e;
            hs[threadIdx.x] = t;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        part[2 * blockIdx.x] = hs[0];
        part[2 * blockIdx.x + 1] = hc[0];
    }
}

// Dot product `dot` (0 or 1) from its chunk sums, in chunk order.
template <typename T>
__device__ __forceinline__ T dots2_final(const double *part, int dot) {
    double s = 0.0, cc = 0.0;
    for (int i = 0; i < kDotChunks; ++i) {
        const int blk = dot * kDotChunks + i;
        double t, e;
        two_sum_d(s, part[2 * blk], t, e);
        s = t;
        cc += part[2 * blk + 1] + e;
    }
    return (T)(s + cc);
}

// x = x + beta (s + v1 d0 + v2 d1) + z, d0 = u1 . y and d1 = u2 . y from
// their chunk sums (every block forms them the same way).
template <typename T>
__global__ void gemver_x2_kernel(T *x, const T *s, const T *v1, const T *v2,
                                 const double *part, const T *z, int64_t n, T beta) {
    __shared__ T dd[2];
    if (threadIdx.x < 2) dd[threadIdx.x] = dots2_final<T>(part, threadIdx.x);
    __syncthreads();
    const T d0 = dd[0], d1 = dd[1];
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const T inner = fma(v2[i], d1, fma(v1[i], d0, s[i]));
        x[i] = fma(beta, inner, x[i]) + z[i];
    }
}

// w = w + alpha (t + u1 e0 + u2 e1), e0 = v1 . x and e1 = v2 . x from
// their chunk sums.
template <typename T>
__global__ void gemver_w2_kernel(T *w, const T *t, const T *u1, const T *u2,
                                 const double *part, int64_t n, T alpha) {
    __shared__ T dd[2];
    if (threadIdx.x < 2) dd[threadIdx.x] = dots2_final<T>(part, threadIdx.x);
    __syncthreads();
    const T d0 = dd[0], d1 = dd[1];
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const T inner = fma(u2[i], d1, fma(u1[i], d0, t[i]));
        w[i] = fma(alpha, inner, w[i]);
    }
}

}  // namespace dmv
