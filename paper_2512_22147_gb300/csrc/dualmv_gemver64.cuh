// GEMVER with update_A in fp64 (Table 1): the pass that writes A_hat.
//
// GEMVER needs A_hat = A + u1 v1^T + u2 v2^T twice, as A_hat^T y and as
// A_hat x, and, with update_A, written over A.  The products factorise
// exactly,
//   A_hat^T y = A^T y + v1 (u1 . y) + v2 (u2 . y),
//   A_hat x   = A x   + u1 (v1 . x) + u2 (v2 . x),
// so the columns-only pass and the dot products are those of GEMVER
// without the update, and only the rows pass changes: it reads a, writes
// a_hat = fma(u2_i, v2_j, fma(u1_i, v1_j, a)) in native fp64 (two DFMAs,
// the same rounding as the on-the-fly kernels), and forms t_i = sum_j a_ij x_j
// from the original a in double-float arithmetic on the FP32 pipes (the
// split and error-free products of dualmv_f64e.cuh).  Native fp64 would add
// a third DFMA per element on the narrow FP64 pipe.
//
// Layout: CTA (c, b) takes rows [c M / C, (c + 1) M / C) of column band b
// (kGvBand columns); warp w of it takes rows w, w + 8, ...  Lane l holds
// columns 2 l, 2 l + 1 of each 64-column group (16-byte loads and stores:
// A 16-byte aligned, lda even).  The band's v1, v2 and the split of x sit in
// shared memory.  A lane's 16 products are summed in a pairwise tree (three
// levels over its 8 column pairs, then the pair), the lanes in a
// butterfly: t's band partial has 9 double-float additions above each
// product, so its error stays below (2^-44 + 27 2^-46) of its terms'
// magnitudes, about 4.4e-13.  The band partials go to q_ws[band][row] for
// the w update, which adds them in a fixed order.
//
// Range: as in the streaming kernel, values of a or x outside
// [2^-40, 2^40) (zeros are fine) make the row's partial native fp64 (x: the
// whole band).  The results are the same arithmetic on every call.
#pragma once

#include "dualmv_f64e.cuh"

namespace dmv {

constexpr int kGvBand = 512;              // columns of a CTA's band
constexpr int kGvWarps = 8;
constexpr int kGvVec = kGvBand / 64;      // 16-byte vectors per lane per row
constexpr int kGvTop = kGvVec == 8 ? 3 : 4;  // levels of the lane's pairwise tree
static_assert(kGvVec == 8 || kGvVec == 16, "a band of 512 or 1024 columns");

struct GvParams {
    double *A;             // a read, a_hat written in place
    int64_t lda;           // even; A 16-byte aligned
    const double *u1, *u2;  // length M
    const double *v1, *v2;  // length N
    const double *x;       // length N: the updated x
    double *q_ws;          // [bands][M] band partials of A x (original A)
    int64_t M, N, bands, row_chunks;
};

__global__ void __launch_bounds__(kGvWarps * 32, 2)
gemver_rows_update_f64_kernel(const GvParams prm) {
    pdl_launch_dependents();
    pdl_wait();  // x comes from the kernel before this one
    __shared__ double2 v1s[kGvBand / 2], v2s[kGvBand / 2];
    __shared__ float4 xs[kGvBand / 2];  // (x_hi[c], x_hi[c+1], x_lo[c], x_lo[c+1])
    __shared__ int band_bad;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t N = prm.N, M = prm.M;
    const int64_t band = blockIdx.y;
    const int64_t c0 = band * kGvBand;
    if (threadIdx.x == 0) band_bad = 0;
    __syncthreads();
    bool xbad = false;
    for (int k = threadIdx.x; k < kGvBand / 2; k += kGvWarps * 32) {
        const int64_t c = c0 + 2 * k;
        const bool in0 = c < N, in1 = c + 1 < N;
        v1s[k] = make_double2(in0 ? prm.v1[c] : 0.0, in1 ? prm.v1[c + 1] : 0.0);
        v2s[k] = make_double2(in0 ? prm.v2[c] : 0.0, in1 ? prm.v2[c + 1] : 0.0);
        const double x0 = in0 ? prm.x[c] : 0.0, x1 = in1 ? prm.x[c + 1] : 0.0;
        float h0, l0, h1, l1;
        split_f64(x0, h0, l0);
        split_f64(x1, h1, l1);
        xs[k] = make_float4(h0, h1, l0, l1);
        xbad |= !f64e_in_range(x0) || !f64e_in_range(x1);
    }
    if (xbad) band_bad = 1;  // every writer stores the same value
    __syncthreads();
    const bool native_band = band_bad != 0;

    const int64_t r_lo = (int64_t)blockIdx.x * M / prm.row_chunks;
    const int64_t r_hi = ((int64_t)blockIdx.x + 1) * M / prm.row_chunks;
    for (int64_t i = r_lo + warp; i < r_hi; i += kGvWarps) {
        double *arow = prm.A + i * prm.lda + c0;
        double2 a[kGvVec];
#pragma unroll
        for (int v = 0; v < kGvVec; ++v) {
            const int off = v * 64 + 2 * lane;
            const int64_t c = c0 + off;
            if (c + 1 < N)
                a[v] = *reinterpret_cast<const double2 *>(arow + off);
            else
                a[v] = make_double2(c < N ? arow[off] : 0.0, 0.0);
        }
        const double u1i = prm.u1[i], u2i = prm.u2[i];

        // t's partial from the original a: products as double-float pairs,
        // summed in a pairwise tree over the lane's kGvVec column pairs.
        DF2 stk[5];
        uint32_t spanv[2] = {0u, 0u};
#pragma unroll
        for (int v = 0; v < kGvVec; ++v) {
            float ah0, al0, ah1, al1;
            split_f64(a[v].x, ah0, al0);
            split_f64(a[v].y, ah1, al1);
            spanv[v & 1] = __vimax3_u32(spanv[v & 1], f64e_range_key(a[v].x),
                                        f64e_range_key(a[v].y));
            const float4 xv = xs[v * 32 + lane];
            DF2 cur;
            df_prod2(make_float2(ah0, ah1), make_float2(al0, al1), make_float2(xv.x, xv.y),
                     make_float2(xv.z, xv.w), cur.s, cur.c);
            // Binary counter over v + 1: fold while the low bits of v are set.
            if (v & 1) cur = df_add2(stk[0], cur);
            if ((v & 3) == 3) cur = df_add2(stk[1], cur);
            if ((v & 7) == 7) cur = df_add2(stk[2], cur);
            if ((v & 15) == 15) cur = df_add2(stk[3], cur);  // (16 vectors only)
            const int lvl = (v & 1) == 0 ? 0 : (v & 3) != 3 ? 1 : (v & 7) != 7 ? 2
                          : (v & 15) != 15 ? 3 : 4;
            stk[lvl] = cur;
        }

        // a_hat, written over a.
#pragma unroll
        for (int v = 0; v < kGvVec; ++v) {
            const int off = v * 64 + 2 * lane;
            const int64_t c = c0 + off;
            const double2 w1 = v1s[v * 32 + lane], w2 = v2s[v * 32 + lane];
            double2 h;
            h.x = fma(u2i, w2.x, fma(u1i, w1.x, a[v].x));
            h.y = fma(u2i, w2.y, fma(u1i, w1.y, a[v].y));
            if (c + 1 < N)
                *reinterpret_cast<double2 *>(arow + off) = h;
            else if (c < N)
                arow[off] = h.x;
        }

        const uint32_t span = max(spanv[0], spanv[1]);
        bool native = native_band;
        if (!native && __any_sync(0xffffffffu, span >= kF64eRangeSpan)) {
            // Exact re-check (zeros pass).
            bool bad = false;
#pragma unroll
            for (int v = 0; v < kGvVec; ++v)
                bad |= !f64e_in_range(a[v].x) || !f64e_in_range(a[v].y);
            native = __any_sync(0xffffffffu, bad);
        }
        double part;
        if (!native) {
            DF sum, hi;
            sum.s = stk[kGvTop].s.x;
            sum.c = stk[kGvTop].c.x;
            hi.s = stk[kGvTop].s.y;
            hi.c = stk[kGvTop].c.y;
            DF t[1] = {df_add(sum, hi)};
            warp_rows_reduce_df<1>(t, lane);
            part = df_to_double(t[0]);
        } else {
            double dot = 0.0;
#pragma unroll
            for (int v = 0; v < kGvVec; ++v) {
                const int64_t c = c0 + v * 64 + 2 * lane;
                dot = fma(a[v].x, c < N ? prm.x[c] : 0.0, dot);
                dot = fma(a[v].y, c + 1 < N ? prm.x[c + 1] : 0.0, dot);
            }
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1)
                dot += __shfl_xor_sync(0xffffffffu, dot, off);
            part = dot;
        }
        if (lane == 0) prm.q_ws[band * M + i] = part;
    }
}

}  // namespace dmv
