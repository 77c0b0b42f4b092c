// Device kernels of the variant tuner: the functional-equivalence check of
// Eq. 4 (a candidate's outputs against the current baseline's) and the
// magnitude sums that scale it.  They are deliberately simple and share no
// code with the streaming kernels whose outputs they check.
#pragma once

#include <cstdint>

namespace dmv {

// den[i] = sum_j |A_ij| |p_j| in double: one warp per row, lanes strided
// over the row.
template <typename T>
__global__ void __launch_bounds__(256) abs_rows_kernel(const T *A, int64_t M, int64_t N,
                                                       int64_t lda, const T *p, double *den) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t i = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); i < M;
         i += warps) {
        const T *row = A + i * lda;
        double acc = 0.0;
        for (int64_t j = lane; j < N; j += 32)
            acc += fabs((double)row[j]) * fabs((double)p[j]);
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
        if (lane == 0) den[i] = acc;
    }
}

// den[j] = sum_i |A_ij| |r_i| in double: one thread per column, rows in
// order (consecutive threads read consecutive columns).
template <typename T>
__global__ void __launch_bounds__(256) abs_cols_kernel(const T *A, int64_t M, int64_t N,
                                                       int64_t lda, const T *r, double *den) {
    const int64_t threads = (int64_t)gridDim.x * blockDim.x;
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < N; j += threads) {
        double acc = 0.0;
        for (int64_t i = 0; i < M; ++i) acc += fabs((double)A[i * lda + j]) * fabs((double)r[i]);
        den[j] = acc;
    }
}

// Largest per-element error of `got` against `base`, folded into *max_bits
// (the bits of a non-negative double, so unsigned order is numeric order).
// With `den`: |got - base| / den, where a zero denominator demands equality.
// Without: exact outputs, any difference counts as infinite.  NaN counts as
// infinite.
template <typename Out>
__global__ void __launch_bounds__(256) fe_max_kernel(const Out *got, const Out *base,
                                                     const double *den, int64_t n,
                                                     unsigned long long *max_bits) {
    const double inf = __longlong_as_double(0x7ff0000000000000ll);
    double worst = 0.0;
    const int64_t threads = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += threads) {
        double e;
        if (den == nullptr) {
            e = got[i] == base[i] ? 0.0 : inf;
        } else {
            const double d = fabs((double)got[i] - (double)base[i]);
            if (!(d == d)) e = inf;
            else if (den[i] > 0.0) e = d / den[i];
            else e = d == 0.0 ? 0.0 : inf;
        }
        worst = e > worst ? e : worst;
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
        const double o = __shfl_xor_sync(0xffffffffu, worst, off);
        worst = o > worst ? o : worst;
    }
    if ((threadIdx.x & 31) == 0 && worst > 0.0)
        atomicMax(max_bits, (unsigned long long)__double_as_longlong(worst));
}

}  // namespace dmv
