// fp64 dual matrix-vector product (BICG, Tables 1-2) on the FP32 pipes.
//
// GB300's FP64 pipe retires about 1.6 DFMA per clock per SM, and float <->
// double conversions run on the same narrow pipe, so two DFMAs per element
// of A cap a native fp64 kernel near a quarter of HBM bandwidth.  This
// kernel streams A exactly like the generic one (same TMA ring, tile
// schedule, workspace layout and combine kernel) but forms both products in
// "double-float" arithmetic: each double is split, with integer bit
// operations only, into an unevaluated sum of two floats, and products and
// sums use error-free FP32 transformations.
//
// Error bound (u = 2^-24, every |a|, |p_j|, |r_i| in [2^-40, 2^40) or 0):
//   split   a = a_hi + a_lo + d: a_hi is a truncated to 24 significant bits,
//           so |a - a_hi| < 2^-23 |a|; a_lo is that remainder rounded to a
//           float, |d| <= u |a - a_hi| < 2^-47 |a|.
//   product a*x ~ p + q, p = fl(a_hi x_hi), q = err(p) + a_hi x_lo +
//           a_lo x_hi (two FMA roundings).  Dropped: a_lo x_lo < 2^-46 |ax|
//           and the split residues d x, a d_x < 2^-46 |ax|; the roundings of
//           q (|q| < 1.25 2^-22 |ax|) add at most 2^-45 |ax|.  In all,
//           |ax - p - q| < 2^-44 |ax|.
//   sum     Knuth's TwoSum on the high parts (exact); the low parts, which
//           hold the products' q and the TwoSum errors (|low| < 1.5 2^-22
//           of the sum of |terms| beneath it), take two roundings per
//           addition: at most 3 2^-46 of those terms' sum |ax| per addition
//           node.  A term of q passes 8 nodes (the lane's 8 columns in a
//           tree, the 32 lanes in a butterfly); a term of s at most 19 (the
//           4 rows of a tile in a chain, then kGroupTiles = 16 tiles in a
//           chain); then fp64 for segments and band partials.
//   So |q_i - q^_i| < (2^-44 + 24 2^-46 + fp64 sums) sum_j |A_ij p_j|
//   ~ 4.1e-13 and |s_j - s^_j| < (2^-44 + 57 2^-46 + fp64 sums)
//   sum_i |A_ij r_i| ~ 8.8e-13 of the sums of magnitudes, inside the 1e-12
//   bar; random data sits near 1e-14.
//   native  NC of each lane's eight columns (default 2; 0 in the packed
//           kernel) take their column sums from native fp64 FMA instead.
//
// Range.  The split and the FP32 arithmetic are exact only while every
// |a|, |p_j|, |r_i| lies in [2^-40, 2^40) or is zero (products then stay
// inside FP32's normal range).  Each element costs about one and a half
// integer ops of range bookkeeping (a key per element, a three-way max per
// pair); a warp whose rows of a tile hold anything else re-checks them
// exactly (zeros are fine) and, if a value really is out of range,
// recomputes those rows with native fp64 FMA.  Results are the same
// arithmetic on every call, so they are deterministic.
#pragma once

#include "dualmv_kernels.cuh"

namespace dmv {

#ifndef DUALMV_F64E_NATIVE_COLS
#define DUALMV_F64E_NATIVE_COLS 2
#endif

// Range key of a double: its high word shifted left by one (the sign bit
// dropped), less the key of 2^-40 (biased exponent 983).  |a| lies in
// [2^-40, 2^40) exactly when the key is below kF64eRangeSpan (2^40 has
// biased exponent 1063); zero and everything out of range give a key at or
// above it.
constexpr uint32_t kF64eRangeLo = 983u << 21;
constexpr uint32_t kF64eRangeSpan = (1063u - 983u) << 21;

__device__ __forceinline__ uint32_t f64e_range_key(double a) {
    return ((uint32_t)__double2hiint(a) << 1) - kF64eRangeLo;
}

struct DF {
    float s;  // high part
    float c;  // low part (sum of everything below s)
};

// Split a double into hi + lo floats without touching the FP64 pipe.
// hi is a truncated to 24 significant bits: sign, exponent and the top 23
// stored mantissa bits.  A float's biased exponent is the double's less
// 896; for double exponents 897..1150 that is the double's low seven
// exponent bits under its top exponent bit (bit 30 of the high word), so
// hi is the two words funnel-shifted left by three places with bits 31 and
// 30 taken from the high word.  lo is the 29 stored bits left over, as an
// integer (shifted up by three) converted to float, so rounded to 24
// significant bits, times 2^(e - 55) with the sign of a (e the exponent of
// a).  |a - hi| < 2^-23 |a| and |a - hi - lo| < 2^-47 |a|.  Zero (either
// sign) gives two zeros; values outside [2^-40, 2^40) give garbage and
// must be caught by the range check.
__device__ __forceinline__ void split_f64(double a, float &hi, float &lo) {
    const uint32_t h = (uint32_t)__double2hiint(a);
    const uint32_t l = (uint32_t)__double2loint(a);
    const uint32_t hi_bits = (h & 0xC0000000u) | (__funnelshift_l(l, h, 3) & 0x3FFFFFFFu);
    hi = __uint_as_float(hi_bits);
    const float scale = __uint_as_float((hi_bits & 0xFF800000u) - (55u << 23));
    lo = __fmul_rn(__uint2float_rn(l << 3), scale);
}

// Exact range test: |a| in [2^-40, 2^40) or a == 0.
__device__ __forceinline__ bool f64e_in_range(double a) {
    const uint32_t h = (uint32_t)__double2hiint(a), l = (uint32_t)__double2loint(a);
    return f64e_range_key(a) < kF64eRangeSpan || ((h << 1) | l) == 0u;
}

__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

// a * x as (p, q), from the splits of a and x (a_lo x_lo dropped): p + q
// is within 2^-44 |a x| of the exact product.
__device__ __forceinline__ void df_prod(float ah, float al, float xh, float xl, float &p,
                                        float &q) {
    p = __fmul_rn(ah, xh);
    q = __fmaf_rn(ah, xh, -p);  // exact rounding error of p
    q = __fmaf_rn(ah, xl, q);
    q = __fmaf_rn(al, xh, q);
}

// acc += (p, q)
__device__ __forceinline__ void df_acc(DF &acc, float p, float q) {
    float s, e;
    two_sum(acc.s, p, s, e);
    acc.s = s;
    acc.c = __fadd_rn(acc.c, __fadd_rn(e, q));
}

__device__ __forceinline__ DF df_add(DF x, DF y) {
    DF r;
    float e;
    two_sum(x.s, y.s, r.s, e);
    r.c = __fadd_rn(__fadd_rn(x.c, y.c), e);
    return r;
}

__device__ __forceinline__ double df_to_double(DF x) {
    return __dadd_rn((double)x.s, (double)x.c);
}

// Reduce-scatter butterfly (as warp_rows_reduce) on double-float values,
// written on the two float components so that every select stays in
// registers.
template <int RPW>
__device__ __forceinline__ void warp_rows_reduce_df(DF (&v)[RPW], int lane) {
    int off = 16;
#pragma unroll
    for (int h = RPW / 2; h >= 1; h /= 2) {
        const bool upper = (lane & off) != 0;
#pragma unroll
        for (int k = 0; k < h; ++k) {
            const float send_s = upper ? v[k].s : v[k + h].s;
            const float send_c = upper ? v[k].c : v[k + h].c;
            DF keep;
            keep.s = upper ? v[k + h].s : v[k].s;
            keep.c = upper ? v[k + h].c : v[k].c;
            DF recv;
            recv.s = __shfl_xor_sync(0xffffffffu, send_s, off);
            recv.c = __shfl_xor_sync(0xffffffffu, send_c, off);
            v[k] = df_add(keep, recv);
        }
        off >>= 1;
    }
#pragma unroll
    for (; off >= 1; off >>= 1) {
        DF recv;
        recv.s = __shfl_xor_sync(0xffffffffu, v[0].s, off);
        recv.c = __shfl_xor_sync(0xffffffffu, v[0].c, off);
        v[0] = df_add(v[0], recv);
    }
}

// ---- packed pairs --------------------------------------------------------
// GB300 issues a packed FP32 add, multiply or FMA on two floats per lane as
// one instruction (the FMA pipe takes two cycles for it).  This kernel is
// bound by instruction issue, not by the FMA pipe, so the double-float
// arithmetic of a lane's two adjacent columns runs as pairs: same
// operations, same roundings, half the instructions.

struct DF2 {
    float2 s;  // high parts of two values
    float2 c;  // low parts
};

__device__ __forceinline__ float2 add2(float2 a, float2 b) { return __fadd2_rn(a, b); }
// a - b, exactly as a scalar subtraction rounds it: b * -1 is exact, the FMA
// rounds once.
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
    return __ffma2_rn(b, make_float2(-1.f, -1.f), a);
}

__device__ __forceinline__ void two_sum2(float2 a, float2 b, float2 &s, float2 &e) {
    s = add2(a, b);
    const float2 bb = sub2(s, a);
    e = add2(sub2(a, sub2(s, bb)), sub2(b, bb));
}

// a * x for two pairs, as df_prod.
__device__ __forceinline__ void df_prod2(float2 ah, float2 al, float2 xh, float2 xl, float2 &p,
                                         float2 &q) {
    p = __fmul2_rn(ah, xh);
    q = __ffma2_rn(ah, xh, make_float2(-p.x, -p.y));  // exact rounding errors of p
    q = __ffma2_rn(ah, xl, q);
    q = __ffma2_rn(al, xh, q);
}

__device__ __forceinline__ void df_acc2(DF2 &acc, float2 p, float2 q) {
    float2 s, e;
    two_sum2(acc.s, p, s, e);
    acc.s = s;
    acc.c = add2(acc.c, add2(e, q));
}

__device__ __forceinline__ DF2 df_add2(DF2 x, DF2 y) {
    DF2 r;
    float2 e;
    two_sum2(x.s, y.s, r.s, e);
    r.c = add2(add2(x.c, y.c), e);
    return r;
}

// Reduce-scatter butterfly without selects, for values a lane computed in a
// permuted row order: slot j of lane l holds row j ^ butterfly_row(l), so at
// every halving level each lane sends slot k + h and keeps slot k (its
// partner, which differs in that level's lane bit, holds the same row in
// slot k + h).  Slot 0 ends with the full sum of row butterfly_row(l), as in
// warp_rows_reduce_df.  The first level adds its pairs of slots as packed
// pairs.
template <int RPW>
__device__ __forceinline__ void warp_rows_reduce_df_perm(DF (&v)[RPW]) {
    int off = 16;
    int h = RPW / 2;
    if constexpr (RPW >= 4) {
        // First level: RPW / 2 sums, as packed pairs.
#pragma unroll
        for (int k = 0; k < RPW / 2; k += 2) {
            DF2 keep, recv;
            keep.s = make_float2(v[k].s, v[k + 1].s);
            keep.c = make_float2(v[k].c, v[k + 1].c);
            recv.s = make_float2(__shfl_xor_sync(0xffffffffu, v[k + RPW / 2].s, off),
                                 __shfl_xor_sync(0xffffffffu, v[k + RPW / 2 + 1].s, off));
            recv.c = make_float2(__shfl_xor_sync(0xffffffffu, v[k + RPW / 2].c, off),
                                 __shfl_xor_sync(0xffffffffu, v[k + RPW / 2 + 1].c, off));
            const DF2 sum = df_add2(keep, recv);
            v[k].s = sum.s.x;
            v[k].c = sum.c.x;
            v[k + 1].s = sum.s.y;
            v[k + 1].c = sum.c.y;
        }
        off >>= 1;
        h /= 2;
    }
#pragma unroll
    for (; h >= 1; h /= 2) {
#pragma unroll
        for (int k = 0; k < h; ++k) {
            DF recv;
            recv.s = __shfl_xor_sync(0xffffffffu, v[k + h].s, off);
            recv.c = __shfl_xor_sync(0xffffffffu, v[k + h].c, off);
            v[k] = df_add(v[k], recv);
        }
        off >>= 1;
    }
#pragma unroll
    for (; off >= 1; off >>= 1) {
        DF recv;
        recv.s = __shfl_xor_sync(0xffffffffu, v[0].s, off);
        recv.c = __shfl_xor_sync(0xffffffffu, v[0].c, off);
        v[0] = df_add(v[0], recv);
    }
}

// Dynamic shared memory of the fp64 kernel: every consumer warp has its own
// ring of STAGES boxes (its RPW rows of a tile), so warps wait only for
// their own rows and drift apart instead of finishing every tile together;
// then the warp scratch for the s flush and one full/empty mbarrier pair
// per (warp, stage).
template <int W, int RPW, int STAGES, int BAND, int NPH = 0>
struct F64eLayout {
    // NPH > 0 (phased maps): per phase, its RPW / NPH rows of the band's box
    // and then their 16 bytes each from the small box, padded to 128 bytes
    // so that every copy's destination stays 128-byte aligned.  kBoxTx is
    // what a warp's copies deliver, kBoxBytes the slot they land in.
    static constexpr int kPhRows = NPH > 0 ? RPW / NPH : RPW;
    static_assert(kPhRows * 16 <= 128, "small boxes of a phase exceed their pad");
    static constexpr int kPhBytes = kPhRows * BAND * (int)sizeof(double) + (NPH > 0 ? 128 : 0);
    static constexpr int kBoxBytes = (NPH > 0 ? NPH : 1) * kPhBytes;
    static constexpr int kBoxTx = RPW * (BAND * (int)sizeof(double) + (NPH > 0 ? 16 : 0));
    static constexpr int kAlign = 1024;
    static constexpr int kRing = W * STAGES * kBoxBytes;
    static constexpr int kScratch = W * BAND * (int)sizeof(double);
    static constexpr int kBars = 2 * W * STAGES * 8;
    static constexpr int kTotal = kAlign + kRing + kScratch + kBars;
};

// ---------------------------------------------------------------- kernel --
//
// W consumer warps x RPW rows per warp per tile; lane l holds columns
// 2l, 2l+1 (+64, +128, +192) of the 256-column band (four double2 vectors).
// kSelf: no producer warp; lane 0 of each consumer warp issues its own
// warp's boxes, refilling a stage as soon as the warp has consumed it.
// kPack: the double-float arithmetic of each lane's two adjacent columns
// runs as packed pairs (no native columns).
// The kernel body, shared by dualmv_stream_f64e_kernel (one tensor map,
// NPH = 0) and dualmv_stream_f64e_phased_kernel (a pair of maps per row
// phase, tmaps[0 .. 2 NPH - 1]; see dualmv_stream_phased_kernel).
template <int W, int RPW, int STAGES, int BAND, bool kBatched3d, int kOut, int NC, bool kSelf,
          bool kPack, int NPH, bool kRev = false>
__device__ __forceinline__ void f64e_body(const CUtensorMap *tmaps, const Params &prm) {
    constexpr bool kQ = (kOut & kOutQ) != 0;  // row sums q = A p
    constexpr bool kS = (kOut & kOutS) != 0;  // column sums s = A^T r
    // kRev: each CTA walks its tile range backwards (as stream_body's).
    static_assert(!kRev || kOut == kOutQ, "backward walk: rows-only passes");
    using T = double;
    using Acc = double;
    using Vec = double2;
    constexpr int VE = 2;
    constexpr int LANE_COLS = BAND / 32;  // columns per lane
    constexpr int VPL = LANE_COLS / VE;   // 16-byte vectors per lane per row
    constexpr int BM = W * RPW;
    constexpr int ROW_BYTES = BAND * (int)sizeof(T);
    using L = F64eLayout<W, RPW, STAGES, BAND, NPH>;
    static_assert(LANE_COLS == 4 || LANE_COLS == 8, "band of 128 or 256 columns");
    constexpr int BOX_BYTES = L::kBoxBytes;
    static_assert(NPH == 0 || (kSelf && !kBatched3d && RPW % NPH == 0 && NPH <= 2),
                  "phased maps: self-loading warps, one problem, whole phase groups");
    // Phased maps: per phase, the band's box (PROWS rows) then the small box.
    constexpr int PH = NPH > 0 ? NPH : 1;
    constexpr int PROWS = RPW / PH;
    constexpr int PH_BYTES = L::kPhBytes;

    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = smem_raw + shared_align_pad<L::kAlign>(smem_raw);
    unsigned char *ring = smem;
    Acc *scratch = reinterpret_cast<Acc *>(smem + L::kRing);
    uint64_t *full_bar = reinterpret_cast<uint64_t *>(smem + L::kRing + L::kScratch);
    uint64_t *empty_bar = full_bar + W * STAGES;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // Tile indices fit 32 bits (the host sends larger launches elsewhere).
    const int S = (int)prm.stripes, NB = (int)prm.bands;
    const int64_t c = blockIdx.x;
    const int t0 = (int)cta_first_tile(c, prm.tiles, prm.grid);
    const int t1 = (int)cta_first_tile(c + 1, prm.tiles, prm.grid);
    const int ntiles = t1 - t0;
    const int g_first = t0 / S;

    if (threadIdx.x == 0) {
        for (int i = 0; i < W * STAGES; ++i) {
            mbar_init(smem_u32(&full_bar[i]), 1);
            mbar_init(smem_u32(&empty_bar[i]), 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    // Launched as a dependent of whatever precedes it on the stream: nothing
    // is read or written before that grid has completed (in late-wait mode,
    // every grid before it has; see Params::pdl_late).  Its dependents may
    // launch only then, so that a late-wait pass may follow it.
    if (!prm.pdl_late) pdl_wait();
    pdl_launch_dependents();

    // ------------------------------------------------------ producer ----
    if (!kSelf && warp == W) {
        if (lane == 0) {
            const uint64_t pol = policy_evict_first();
            bool ok = true;
            int issued = 0;
            int partial_w = 0;
            TileCursor32 cur;
            cur.init(kRev ? t1 - 1 : t0, S, NB);
            int stage = 0;
            uint32_t phase = 0;
            for (int k = 0; k < ntiles; ++k) {
                const int x = (int)(cur.band * BAND), y = (int)(cur.stripe * BM);
                // One box of RPW rows per consumer warp, into that warp's ring.
                for (int w = 0; w < W && ok; ++w) {
                    const int slot = w * STAGES + stage;
                    if (k >= STAGES)
                        ok = mbar_wait_bounded(smem_u32(&empty_bar[slot]), phase ^ 1u);
                    if (!ok) {
                        partial_w = w;  // boxes 0..w-1 of tile k are in flight
                        break;
                    }
                    const uint32_t fb = smem_u32(&full_bar[slot]);
                    mbar_arrive_expect_tx(fb, L::kBoxTx);
                    const uint32_t dst = smem_u32(ring + (size_t)slot * BOX_BYTES);
                    if constexpr (kBatched3d)
                        tma_load_3d(dst, &tmaps[0], x, y + w * RPW, (int)cur.b, fb, pol);
                    else
                        tma_load_2d(dst, &tmaps[0], x, y + w * RPW, fb, pol);
                }
                if (!ok) break;
                issued = k + 1;
                if constexpr (kRev)
                    cur.retreat(S, NB);
                else
                    cur.advance(S, NB);
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            // Every box issued must land before the CTA exits (bounded): the
            // last STAGES whole tiles, and the first partial_w boxes of a
            // tile abandoned half way by a timeout.
            for (int k = issued > STAGES ? issued - STAGES : 0; k <= issued; ++k) {
                const int st = (int)(k % STAGES);
                const int nw = k < issued ? W : partial_w;
                for (int w = 0; w < nw; ++w)
                    mbar_wait_bounded(smem_u32(&full_bar[w * STAGES + st]),
                                      (uint32_t)(k / STAGES) & 1u);
            }
        }
        return;
    }

    // ----------------------------------------------------- consumers ----
    const T *__restrict__ pg = static_cast<const T *>(prm.p);
    const T *__restrict__ rg = static_cast<const T *>(prm.r);
    const int nthreads_c = W * 32;

    // Lane columns LANE_COLS - kNativeCols .. LANE_COLS - 1 sum s in fp64
    // (NC of every 8).
    static_assert(NC >= 0 && NC <= 8, "native columns: 0..8 of every 8");
    static_assert(!kPack || (NC == 0 && VE == 2), "packed pairs: no native columns");
    constexpr int kNativeCols = NC * LANE_COLS / 8;
    constexpr int kFirstNative = LANE_COLS - kNativeCols;
    double snat[kNativeCols > 0 ? kNativeCols : 1];  // fp64 segment sums of s
#pragma unroll
    for (int j = 0; j < kNativeCols; ++j) snat[j] = 0.0;
    float ph[LANE_COLS], pl[LANE_COLS];  // split p of this lane's columns
    float2 ph2[VPL], pl2[VPL];           // the same, as pairs (kPack)
    DF2 grp2[VPL];                       // group sums of s as pairs (kPack)
    bool p_bad = false;                  // some p of this lane out of range
    DF grp[LANE_COLS];                   // group sums of s (double-float)
    // Segment sums of s (fp64) live in this warp's row of the flush scratch;
    // each lane owns its 8 columns there, so no synchronisation is needed
    // until the segment flush.
    Acc *segp = scratch + warp * BAND;
#pragma unroll
    for (int e = 0; e < LANE_COLS; ++e) {
        ph[e] = pl[e] = 0.f;
        grp[e].s = grp[e].c = 0.f;
    }
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
        ph2[v] = pl2[v] = make_float2(0.f, 0.f);
        grp2[v].s = grp2[v].c = make_float2(0.f, 0.f);
    }
#pragma unroll
    for (int v = 0; v < VPL; ++v)
#pragma unroll
        for (int e = 0; e < VE; ++e) segp[lane_col<T>(v, lane, e)] = 0.0;
    int ngrp = 0;
    int seg_start_stripe = 0;
    bool ok = true;

    TileCursor32 cur;
    cur.init(kRev ? t1 - 1 : t0, S, NB);
    T r_next = T(0);
    {
        const int64_t row = cur.stripe * BM + (int64_t)warp * RPW + lane;
        if (kS && lane < RPW && row < prm.M) r_next = rg[cur.b * prm.strideR + row];
    }
    int stage = 0;
    uint32_t phase = 0;

    // Self-loading: lane 0 keeps a second cursor STAGES tiles ahead and
    // refills each stage of this warp's ring right after the warp read it.
    TileCursor32 ld{0, 0, 0, 0};
    int issued = 0;           // boxes this warp issued (lane 0)
    int waited_to = ntiles;   // first tile whose wait was abandoned
    uint64_t pol = 0;
    auto issue = [&](int st) {
        const int slot_i = warp * STAGES + st;
        const uint32_t fb = smem_u32(&full_bar[slot_i]);
        mbar_arrive_expect_tx(fb, L::kBoxTx);
        const uint32_t dst = smem_u32(ring + (size_t)slot_i * BOX_BYTES);
        const int x = (int)(ld.band * BAND), y = (int)(ld.stripe * BM) + warp * RPW;
        if constexpr (NPH > 0) {
#pragma unroll
            for (int ph = 0; ph < NPH; ++ph) {
                const uint32_t d = dst + (uint32_t)(ph * PH_BYTES);
                tma_load_2d(d, &tmaps[2 * ph], x, y / NPH, fb, pol);
                tma_load_2d(d + (uint32_t)(PROWS * ROW_BYTES), &tmaps[2 * ph + 1], x + BAND,
                            y / NPH, fb, pol);
            }
        } else if constexpr (kBatched3d) {
            tma_load_3d(dst, &tmaps[0], x, y, (int)ld.b, fb, pol);
        } else {
            tma_load_2d(dst, &tmaps[0], x, y, fb, pol);
        }
        if constexpr (kRev)
            ld.retreat(S, NB);
        else
            ld.advance(S, NB);
        ++issued;
    };
    if constexpr (kSelf) {
        if (lane == 0) {
            pol = policy_evict_first();
            ld.init(kRev ? t1 - 1 : t0, S, NB);
            for (int st = 0; st < STAGES && st < ntiles; ++st) issue(st);
        }
    }
    // Releases the stage just read: to the producer warp, or (self-loading)
    // by refilling it with the tile STAGES ahead.
    auto release = [&](int slot_r, int k_r) {
        __syncwarp();
        if constexpr (kSelf) {
            if (lane == 0 && ok && k_r + STAGES < ntiles) {
                // The warp's reads of this stage (generic proxy) come before
                // the copy that overwrites it (async proxy).
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                issue((int)(slot_r - warp * STAGES));
            }
        } else {
            if (lane == 0) mbar_arrive(smem_u32(&empty_bar[slot_r]));
        }
    };

    for (int k = 0; k < ntiles; ++k) {
        const int g = cur.g;
        const int stripe = cur.stripe;
        const int band = cur.band;
        const int64_t b = cur.b;
        const int64_t col0 = band * BAND;
        const int64_t row0 = stripe * BM + (int64_t)warp * RPW;
        const T rmine = r_next;
        if constexpr (kRev)
            cur.retreat(S, NB);
        else
            cur.advance(S, NB);
        if (kS && k + 1 < ntiles) {
            const int64_t row = cur.stripe * BM + (int64_t)warp * RPW + lane;
            r_next = (lane < RPW && row < prm.M) ? rg[cur.b * prm.strideR + row] : T(0);
        }

        const bool seg_start = k == 0 || stripe == (kRev ? S - 1 : 0);
        if (seg_start) seg_start_stripe = stripe;
        if (kQ && seg_start) {  // new segment: split this band's p
            const T *pb = pg + b * prm.strideP;
            p_bad = false;
#pragma unroll
            for (int v = 0; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) {
                    const int64_t col = col0 + lane_col<T>(v, lane, e);
                    const T pv = col < prm.N ? pb[col] : T(0);
                    split_f64(pv, ph[v * VE + e], pl[v * VE + e]);
                    p_bad |= !f64e_in_range(pv);
                }
            if constexpr (kPack) {
#pragma unroll
                for (int v = 0; v < VPL; ++v) {
                    ph2[v] = make_float2(ph[v * VE], ph[v * VE + 1]);
                    pl2[v] = make_float2(pl[v * VE], pl[v * VE + 1]);
                }
            }
        }
        // r of this warp's rows, split by its owner lane.
        float rh_mine, rl_mine;
        split_f64(rmine, rh_mine, rl_mine);
        const bool r_bad = kS && !f64e_in_range(rmine);

        const int slot = warp * STAGES + stage;
        if (ok) {
            ok = mbar_wait_bounded(smem_u32(&full_bar[slot]), phase);
            if (!ok) waited_to = k;
        }
        // This warp's RPW rows of the tile.
        const unsigned char *tileb = ring + (size_t)slot * BOX_BYTES;
        // Vector v of row r of the box.  Phased maps: row r is row r / NPH of
        // phase r % NPH, its columns start ph_off doubles into its box row.
        // An offset row is read as two 8-byte halves (the last lane's last
        // upper half: the small box), which costs the shared-memory
        // wavefronts of one aligned 16-byte vector.
        auto rowvec = [&](int r, int v) -> Vec {
            if constexpr (NPH == 0) {
                return reinterpret_cast<const Vec *>(tileb + (size_t)r * ROW_BYTES)[v * 32 + lane];
            } else {
                const int ph = r % NPH, pr = r / NPH;
                const unsigned char *phb = tileb + (size_t)ph * PH_BYTES;
                const unsigned char *rowb = phb + (size_t)pr * ROW_BYTES;
                if ((ph == 0 ? prm.ph_off[0] : prm.ph_off[NPH - 1]) == 0)
                    return reinterpret_cast<const Vec *>(rowb)[v * 32 + lane];
                const double *lo = reinterpret_cast<const double *>(rowb) + 2 * (v * 32 + lane) + 1;
                const double *hi =
                    (v == VPL - 1 && lane == 31)
                        ? reinterpret_cast<const double *>(phb + (size_t)PROWS * ROW_BYTES +
                                                           (size_t)pr * 16)
                        : lo + 1;
                return Vec{*lo, *hi};
            }
        };

        // Fast path: double-float arithmetic with a cheap range bound.
        DF q[RPW];
#pragma unroll
        for (int i = 0; i < RPW; ++i) q[i].s = q[i].c = 0.f;
        DF tacc[LANE_COLS];
        DF2 tacc2[VPL];
        double tnat[kNativeCols > 0 ? kNativeCols : 1];
#pragma unroll
        for (int j = 0; j < kNativeCols; ++j) tnat[j] = 0.0;
        // Max over elements of their range keys.  The packed path keeps one
        // running max per 16-byte column vector: a single chain through all
        // of a tile's elements serialises the warp (89% against 85% of HBM
        // on the 65536 x 4096 workload).
        uint32_t span = 0;
        uint32_t spanv[4] = {0u, 0u, 0u, 0u};
        if constexpr (kPack) {
            // Slot i of this lane is row i ^ perm (see warp_rows_reduce_df_perm).
            const int perm = butterfly_row<RPW>(lane);
#pragma unroll
            for (int i = 0; i < RPW; ++i) {
                const int ri = i ^ perm;
                Vec a[VPL];
#pragma unroll
                for (int v = 0; v < VPL; ++v) a[v] = rowvec(ri, v);
                const float rh = __shfl_sync(0xffffffffu, rh_mine, ri);
                const float rl = __shfl_sync(0xffffffffu, rl_mine, ri);
                const float2 rh2 = make_float2(rh, rh), rl2 = make_float2(rl, rl);
                DF2 qp[VPL];
#pragma unroll
                for (int v = 0; v < VPL; ++v) {
                    float ah0, al0, ah1, al1;
                    split_f64(a[v].x, ah0, al0);
                    split_f64(a[v].y, ah1, al1);
                    spanv[v] = __vimax3_u32(spanv[v], f64e_range_key(a[v].x),
                                            f64e_range_key(a[v].y));
                    const float2 ah = make_float2(ah0, ah1), al = make_float2(al0, al1);
                    if constexpr (kS) {
                        float2 p0, p1;
                        df_prod2(ah, al, rh2, rl2, p0, p1);
                        if (i == 0) {
                            tacc2[v].s = p0;
                            tacc2[v].c = p1;
                        } else {
                            df_acc2(tacc2[v], p0, p1);
                        }
                    }
                    if constexpr (kQ) df_prod2(ah, al, ph2[v], pl2[v], qp[v].s, qp[v].c);
                }
                if constexpr (kQ) {
                    // Pairwise over the lane's 8 columns: the two halves of
                    // each pair separately, then the halves together.
                    const DF2 h = df_add2(df_add2(qp[0], qp[1]), df_add2(qp[2], qp[3]));
                    DF lo, hi;
                    lo.s = h.s.x;
                    lo.c = h.c.x;
                    hi.s = h.s.y;
                    hi.c = h.c.y;
                    q[i] = df_add(lo, hi);
                }
            }
        } else {
#pragma unroll
        for (int i = 0; i < RPW; ++i) {
            Vec a[VPL];
#pragma unroll
            for (int v = 0; v < VPL; ++v) a[v] = rowvec(i, v);
            const float rh = __shfl_sync(0xffffffffu, rh_mine, i);
            const float rl = __shfl_sync(0xffffffffu, rl_mine, i);
            const double rd = __shfl_sync(0xffffffffu, rmine, i);
            // Row products with p, summed pairwise (depth 3, not a chain of 7).
            DF qp[LANE_COLS];
#pragma unroll
            for (int v = 0; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) {
                    const int ce = v * VE + e;
                    float ah, al;
                    split_f64(vget(a[v], e), ah, al);
                    span = max(span, f64e_range_key(vget(a[v], e)));
                    if (!kS) {
                    } else if (ce < kFirstNative) {
                        float p0, p1;
                        df_prod(ah, al, rh, rl, p0, p1);
                        if (i == 0) {
                            tacc[ce].s = p0;
                            tacc[ce].c = p1;
                        } else {
                            df_acc(tacc[ce], p0, p1);
                        }
                    } else {
                        tnat[ce - kFirstNative] =
                            fma(vget(a[v], e), rd, tnat[ce - kFirstNative]);
                    }
                    if constexpr (kQ) df_prod(ah, al, ph[ce], pl[ce], qp[ce].s, qp[ce].c);
                }
            if constexpr (!kQ) {
            } else if constexpr (LANE_COLS == 8)
                q[i] = df_add(df_add(df_add(qp[0], qp[1]), df_add(qp[2], qp[3])),
                              df_add(df_add(qp[4], qp[5]), df_add(qp[6], qp[7])));
            else
                q[i] = df_add(df_add(qp[0], qp[1]), df_add(qp[2], qp[3]));
        }
        }
        if constexpr (kPack) {
            if constexpr (VPL == 4)
                span = max(max(spanv[0], spanv[1]), max(spanv[2], spanv[3]));
            else
                span = max(spanv[0], spanv[1]);
        }
        // Anything suspicious in this warp's rows (zeros included)?
        const bool rows_r_bad = __any_sync(0xffffffffu, lane < RPW && r_bad);
        bool need_fp64 = rows_r_bad || __any_sync(0xffffffffu, kQ && p_bad);
        if (!need_fp64 && __any_sync(0xffffffffu, span >= kF64eRangeSpan)) {
            // Exact re-check: zeros are fine, anything else out of range is not.
            bool bad = false;
#pragma unroll
            for (int i = 0; i < RPW; ++i) {
#pragma unroll
                for (int v = 0; v < VPL; ++v) {
                    const Vec av = rowvec(i, v);
                    bad |= !f64e_in_range(av.x) || !f64e_in_range(av.y);
                }
            }
            need_fp64 = __any_sync(0xffffffffu, bad);
        }

        if (!need_fp64) {
            release(slot, k);
            if constexpr (kQ) {
                if constexpr (kPack)
                    warp_rows_reduce_df_perm<RPW>(q);
                else
                    warp_rows_reduce_df<RPW>(q, lane);
            }
            if (kQ && butterfly_writer<RPW>(lane)) {
                const int64_t row = row0 + butterfly_row<RPW>(lane);
                if (row < prm.M) {
                    const double qv = df_to_double(q[0]);
                    if (prm.bands == 1)
                        static_cast<Acc *>(prm.q)[b * prm.strideQ + row] = qv;
                    else
                        static_cast<Acc *>(prm.q_ws)[(b * prm.bands + band) * prm.M + row] = qv;
                }
            }
            if constexpr (kPack) {
#pragma unroll
                for (int v = 0; v < VPL; ++v) grp2[v] = df_add2(grp2[v], tacc2[v]);
            } else {
#pragma unroll
                for (int e = 0; e < kFirstNative; ++e) grp[e] = df_add(grp[e], tacc[e]);
#pragma unroll
                for (int j = 0; j < kNativeCols; ++j) snat[j] += tnat[j];
            }
        } else {
            // Out-of-range values in these rows: native fp64 for them.
            double pd[LANE_COLS];
            const T *pb = pg + b * prm.strideP;
#pragma unroll
            for (int v = 0; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) {
                    const int64_t col = col0 + lane_col<T>(v, lane, e);
                    pd[v * VE + e] = (kQ && col < prm.N) ? pb[col] : 0.0;
                }
            double qd[RPW];
            double td[LANE_COLS];
#pragma unroll
            for (int e = 0; e < LANE_COLS; ++e) td[e] = 0.0;
#pragma unroll
            for (int i = 0; i < RPW; ++i) {
                const double ri = __shfl_sync(0xffffffffu, rmine, i);
                double dot = 0.0;
#pragma unroll
                for (int v = 0; v < VPL; ++v) {
                    const Vec av = rowvec(i, v);
#pragma unroll
                    for (int e = 0; e < VE; ++e) {
                        const double x = vget(av, e);
                        dot = fma(x, pd[v * VE + e], dot);
                        td[v * VE + e] = fma(x, ri, td[v * VE + e]);
                    }
                }
                qd[i] = dot;
            }
            release(slot, k);
            if constexpr (kQ) warp_rows_reduce<RPW>(qd, lane);
            if (kQ && butterfly_writer<RPW>(lane)) {
                const int64_t row = row0 + butterfly_row<RPW>(lane);
                if (row < prm.M) {
                    if (prm.bands == 1)
                        static_cast<Acc *>(prm.q)[b * prm.strideQ + row] = qd[0];
                    else
                        static_cast<Acc *>(prm.q_ws)[(b * prm.bands + band) * prm.M + row] =
                            qd[0];
                }
            }
#pragma unroll
            for (int v = 0; v < VPL; ++v)
#pragma unroll
                for (int e = 0; e < VE; ++e) segp[lane_col<T>(v, lane, e)] += td[v * VE + e];
        }
        if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
        }

        if constexpr (kS) {
            const bool seg_end = (stripe == S - 1 || k == ntiles - 1);
            if (++ngrp == kGroupTiles || seg_end) {
    #pragma unroll
                for (int v = 0; v < VPL; ++v)
    #pragma unroll
                    for (int e = 0; e < VE; ++e) {
                        const int ce = v * VE + e;
                        if constexpr (kPack) {
                            DF x;
                            x.s = e == 0 ? grp2[v].s.x : grp2[v].s.y;
                            x.c = e == 0 ? grp2[v].c.x : grp2[v].c.y;
                            segp[lane_col<T>(v, lane, e)] += df_to_double(x);
                        } else if (ce < kFirstNative) {
                            segp[lane_col<T>(v, lane, e)] += df_to_double(grp[ce]);
                            grp[ce].s = grp[ce].c = 0.f;
                        }
                    }
                if constexpr (kPack) {
    #pragma unroll
                    for (int v = 0; v < VPL; ++v) grp2[v].s = grp2[v].c = make_float2(0.f, 0.f);
                }
                ngrp = 0;
            }
            if (seg_end) {
    #pragma unroll
                for (int v = 0; v < VPL; ++v)
    #pragma unroll
                    for (int e = 0; e < VE; ++e) {
                        const int ce = v * VE + e;
                        if (ce >= kFirstNative) {
                            segp[lane_col<T>(v, lane, e)] += snat[ce - kFirstNative];
                            snat[ce - kFirstNative] = 0.0;
                        }
                    }
            }

            if (seg_end) {  // segment end: flush s
                named_barrier(1, nthreads_c);
                const bool whole_band = (seg_start_stripe == 0 && stripe == S - 1);
                for (int col = threadIdx.x; col < BAND; col += nthreads_c) {
                    Acc acc = scratch[col];
    #pragma unroll
                    for (int w = 1; w < W; ++w) acc = acc + scratch[w * BAND + col];
                    if (whole_band) {
                        if (col0 + col < prm.N)
                            static_cast<Acc *>(prm.s)[b * prm.strideS + col0 + col] = acc;
                    } else {
                        static_cast<Acc *>(prm.s_ws)[((c * prm.max_seg) + (g - g_first)) *
                                                         BAND + col] = acc;
                    }
                }
                named_barrier(1, nthreads_c);
    #pragma unroll
                for (int v = 0; v < VPL; ++v)
    #pragma unroll
                    for (int e = 0; e < VE; ++e) segp[lane_col<T>(v, lane, e)] = 0.0;
            }
        }
    }
    // Self-loading after an abandoned wait: boxes this warp issued for tiles
    // it never waited for must land before the CTA exits (bounded).
    if constexpr (kSelf) {
        if (lane == 0)
            for (int kk = waited_to; kk < issued; ++kk)
                mbar_wait_bounded(smem_u32(&full_bar[warp * STAGES + (int)(kk % STAGES)]),
                                  (uint32_t)(kk / STAGES) & 1u);
    }
}

template <int W, int RPW, int STAGES, int BAND, bool kBatched3d, int kOut = kOutBoth,
          int NC = DUALMV_F64E_NATIVE_COLS, bool kSelf = false, bool kPack = false,
          bool kRev = false>
__global__ void __launch_bounds__((W + (kSelf ? 0 : 1)) * 32, 1)
dualmv_stream_f64e_kernel(const __grid_constant__ CUtensorMap tmap, const Params prm) {
    f64e_body<W, RPW, STAGES, BAND, kBatched3d, kOut, NC, kSelf, kPack, 0, kRev>(&tmap, prm);
    if (prm.pdl_late) pdl_wait();  // see Params::pdl_late
}

// fp64 rows whose stride or base is not 16-byte aligned (odd lda): the same
// kernel reading through a pair of tensor maps per row phase.
template <int W, int RPW, int STAGES, int NPH>
__global__ void __launch_bounds__(W * 32, 1)
dualmv_stream_f64e_phased_kernel(const __grid_constant__ TmapSet maps, const Params prm) {
    f64e_body<W, RPW, STAGES, 256, false, kOutBoth, 0, true, true, NPH>(maps.m, prm);
    if (prm.pdl_late) pdl_wait();  // see Params::pdl_late
}

}  // namespace dmv
