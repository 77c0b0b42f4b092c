// GEMVER with update_A (Table 1): the pass that writes A_hat.
//
// GEMVER needs A_hat = A + u1 v1^T + u2 v2^T twice, as A_hat^T y and as
// A_hat x, and, with update_A, written over A.  The products factorise
// exactly,
//   A_hat^T y = A^T y + v1 (u1 . y) + v2 (u2 . y),
//   A_hat x   = A x   + u1 (v1 . x) + u2 (v2 . x),
// so the columns-only pass and the dot products are those of GEMVER
// without the update, and only the rows pass changes: one kernel reads a,
// writes a_hat = fma(u2_i, v2_j, fma(u1_i, v1_j, a)) over it (the same
// fused form as the on-the-fly kernels) and forms the band partials of
// t_i = sum_j a_ij x_j from the original a.
//
//   fp64 (gemver_rows_update_f64_kernel): a_hat in native fp64 (two DFMAs);
//   t in double-float arithmetic on the FP32 pipes (the split and
//   error-free products of dualmv_f64e.cuh), where native fp64 would add a
//   third DFMA per element on the narrow FP64 pipe.
//   fp32 (gemver_rows_update_f32_kernel): everything in FP32 FMAs; the pass
//   is one read and one write of A with little arithmetic.
//
// Layout: CTA (c, b) takes rows [c M / C, (c + 1) M / C) of column band b;
// warp w of it takes rows w, w + 8, ...; each lane holds 16 bytes of every
// 32-lane group of vectors (16-byte loads and stores: A 16-byte aligned,
// the row stride a multiple of 16 bytes).  The band's v1, v2 and x (fp64:
// the split of x) sit in shared memory.  Band partials go to q_ws[band][row]
// for the w update, which adds them in a fixed order.
#pragma once

#include "dualmv_f64e.cuh"

namespace dmv {

constexpr int kGvWarps = 8;

template <typename T>
struct GvParams {
    T *A;                // a read, a_hat written in place
    int64_t lda;         // row stride a multiple of 16 bytes; A 16-byte aligned
    const T *u1, *u2;    // length M
    const T *v1, *v2;    // length N
    const T *x;          // length N: the updated x
    T *q_ws;             // [bands][M] band partials of A x (original A)
    int64_t M, N, bands, row_chunks;
};

// ---- fp64 ----------------------------------------------------------------
// Bands of 512 columns; lane l holds columns 2 l, 2 l + 1 of each 64-column
// group.  A lane's 16 products are summed in a pairwise tree (three levels
// over its 8 column pairs, then the pair), the lanes in a butterfly: t's
// band partial has 9 double-float additions above each product, so its
// error stays below (2^-44 + 27 2^-46) of its terms' magnitudes, about
// 4.4e-13.  Range: as in the streaming kernel, values of a or x outside
// [2^-40, 2^40) (zeros are fine) make the row's partial native fp64 (x: the
// whole band).  The results are the same arithmetic on every call.
constexpr int kGvBand = 512;              // columns of a CTA's band
constexpr int kGvVec = kGvBand / 64;      // 16-byte vectors per lane per row
constexpr int kGvTop = kGvVec == 8 ? 3 : 4;  // levels of the lane's pairwise tree
static_assert(kGvVec == 8 || kGvVec == 16, "a band of 512 or 1024 columns");

__global__ void __launch_bounds__(kGvWarps * 32, 2)
gemver_rows_update_f64_kernel(const GvParams<double> prm) {
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

// ---- fp32 ----------------------------------------------------------------
// Bands of 1024 columns; lane l holds columns 4 l .. 4 l + 3 of each
// 128-column group.  A lane's 32 products are summed as four-product groups
// (two FMAs and an add) in a pairwise tree over its 8 groups, the lanes in
// a butterfly; the band partials are added by the w update.
constexpr int kGvBand32 = 1024;
constexpr int kGvVec32 = kGvBand32 / 128;   // float4 per lane per row

// One row of a band: a_hat written over a, and the row's band partial of
// t (kRagged: columns past N are neither read nor written).
template <bool kRagged>
__device__ __forceinline__ void gv_row_f32(const GvParams<float> &prm, int64_t i, int64_t c0,
                                           int lane, const float4 *v1s, const float4 *v2s,
                                           const float4 *xs) {
    const int64_t N = prm.N;
    float *arow = prm.A + i * prm.lda + c0;
    float4 a[kGvVec32];
#pragma unroll
    for (int v = 0; v < kGvVec32; ++v) {
        const int off = v * 128 + 4 * lane;
        const int64_t c = c0 + off;
        if (!kRagged || c + 3 < N) {
            a[v] = *reinterpret_cast<const float4 *>(arow + off);
        } else {
            a[v].x = c < N ? arow[off] : 0.f;
            a[v].y = c + 1 < N ? arow[off + 1] : 0.f;
            a[v].z = c + 2 < N ? arow[off + 2] : 0.f;
            a[v].w = 0.f;
        }
    }
    const float u1i = prm.u1[i], u2i = prm.u2[i];
    // Per vector: its group of t's products, then a_hat written over a.
    float pv[kGvVec32];
#pragma unroll
    for (int v = 0; v < kGvVec32; ++v) {
        const float4 xv = xs[v * 32 + lane];
        const float t0 = fmaf(a[v].x, xv.x, a[v].y * xv.y);
        const float t1 = fmaf(a[v].z, xv.z, a[v].w * xv.w);
        pv[v] = t0 + t1;
        const int off = v * 128 + 4 * lane;
        const int64_t c = c0 + off;
        const float4 w1 = v1s[v * 32 + lane], w2 = v2s[v * 32 + lane];
        float4 h;
        h.x = fmaf(u2i, w2.x, fmaf(u1i, w1.x, a[v].x));
        h.y = fmaf(u2i, w2.y, fmaf(u1i, w1.y, a[v].y));
        h.z = fmaf(u2i, w2.z, fmaf(u1i, w1.z, a[v].z));
        h.w = fmaf(u2i, w2.w, fmaf(u1i, w1.w, a[v].w));
        if (!kRagged || c + 3 < N) {
            *reinterpret_cast<float4 *>(arow + off) = h;
        } else {
            if (c < N) arow[off] = h.x;
            if (c + 1 < N) arow[off + 1] = h.y;
            if (c + 2 < N) arow[off + 2] = h.z;
        }
        // The next vector's shared loads stay after this store: hoisting
        // all of them next to the row's loads would not fit the registers.
        asm volatile("" ::: "memory");
    }
    static_assert(kGvVec32 == 8, "the tree below is written for 8 groups");
    float dot = ((pv[0] + pv[1]) + (pv[2] + pv[3])) + ((pv[4] + pv[5]) + (pv[6] + pv[7]));
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
    if (lane == 0) prm.q_ws[(c0 / kGvBand32) * prm.M + i] = dot;
}

__global__ void __launch_bounds__(kGvWarps * 32, 2)
gemver_rows_update_f32_kernel(const GvParams<float> prm) {
    pdl_launch_dependents();
    pdl_wait();  // x comes from the kernel before this one
    __shared__ float4 v1s[kGvBand32 / 4], v2s[kGvBand32 / 4], xs[kGvBand32 / 4];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t N = prm.N, M = prm.M;
    const int64_t band = blockIdx.y;
    const int64_t c0 = band * kGvBand32;
    for (int k = threadIdx.x; k < kGvBand32 / 4; k += kGvWarps * 32) {
        const int64_t c = c0 + 4 * k;
        float4 a1, a2, ax;
        a1.x = c < N ? prm.v1[c] : 0.f;
        a1.y = c + 1 < N ? prm.v1[c + 1] : 0.f;
        a1.z = c + 2 < N ? prm.v1[c + 2] : 0.f;
        a1.w = c + 3 < N ? prm.v1[c + 3] : 0.f;
        a2.x = c < N ? prm.v2[c] : 0.f;
        a2.y = c + 1 < N ? prm.v2[c + 1] : 0.f;
        a2.z = c + 2 < N ? prm.v2[c + 2] : 0.f;
        a2.w = c + 3 < N ? prm.v2[c + 3] : 0.f;
        ax.x = c < N ? prm.x[c] : 0.f;
        ax.y = c + 1 < N ? prm.x[c + 1] : 0.f;
        ax.z = c + 2 < N ? prm.x[c + 2] : 0.f;
        ax.w = c + 3 < N ? prm.x[c + 3] : 0.f;
        v1s[k] = a1;
        v2s[k] = a2;
        xs[k] = ax;
    }
    __syncthreads();

    const int64_t r_lo = (int64_t)blockIdx.x * M / prm.row_chunks;
    const int64_t r_hi = ((int64_t)blockIdx.x + 1) * M / prm.row_chunks;
    // Every band but a ragged last one takes the unguarded form.
    if (c0 + kGvBand32 <= N) {
        for (int64_t i = r_lo + warp; i < r_hi; i += kGvWarps)
            gv_row_f32<false>(prm, i, c0, lane, v1s, v2s, xs);
    } else {
        for (int64_t i = r_lo + warp; i < r_hi; i += kGvWarps)
            gv_row_f32<true>(prm, i, c0, lane, v1s, v2s, xs);
    }
}

}  // namespace dmv
