/*
 * dualmv — fused dual matrix-vector product for NVIDIA GB300 (sm_103a).
 *
 *     q = A * p        (q_i = sum_j A_ij p_j,  i < M)
 *     s = A^T * r      (s_j = sum_i A_ij r_i,  j < N)
 *
 * both from a single pass over A.  This is the BICG kernel that the paper
 * tunes (Table 1 and Table 2, row "BICG", Section 4.2); the paper names it
 * without printing a formula, and the definition above is PolyBench's BiCG
 * sub-kernel.
 *
 * Conventions shared by every entry point below
 * ---------------------------------------------
 * Layout.  A is M x N, row-major, element (i, j) at A[i * lda + j], with
 *   lda >= max(1, N).  Columns N..lda-1 of each row are padding and are never
 *   read.  p has N elements, r has M, q has M, s has N; all are contiguous.
 * Memory.  Every pointer is caller-owned DEVICE memory on the current CUDA
 *   device (cudaSetDevice).  Nothing is copied to or from the host.  Outputs
 *   must not alias inputs or each other (not checked; undefined if they do).
 * Streams.  Each call is asynchronous on `stream` (0 is the legacy default
 *   stream): it enqueues its kernels and returns.  The library takes a
 *   stream-ordered workspace from its own per-device memory pool
 *   (cudaMallocFromPoolAsync) and returns it on the same stream.
 * Results.  Floating-point outputs are deterministic run to run for a given
 *   shape on a given GPU (fixed summation order, no atomics).  Integer
 *   outputs are exact modulo 2^64 in any order, so the int32 path adds its
 *   partial sums into q and s with atomics and takes no workspace.
 * Errors.  Every call returns a dualmv_status and never prints or aborts.
 *   DUALMV_ERR_INVALID_VALUE: M < 0, N < 0, batch < 0, lda < max(1, N), a
 *     NULL pointer whose extent is nonzero, or batch strides that make
 *     outputs of different problems overlap.  Nothing is enqueued.
 *   DUALMV_ERR_ALLOC: the workspace could not be allocated.  Nothing ran.
 *   DUALMV_ERR_LAUNCH: a CUDA call failed; dualmv_last_cuda_error() gives
 *     the cudaError_t value.
 *   Empty problems succeed: when N == 0, q is set to zero; when M == 0, s is
 *   set to zero; when batch == 0 nothing happens.
 *   Faults that happen on the device after the call returned (a bounded wait
 *   that timed out) are reported by dualmv_device_fault().
 * Alignment.  The fast path streams A with the Tensor Memory Accelerator and
 *   needs A 16-byte aligned and lda * sizeof(element) (and, batched,
 *   strideA * sizeof(element)) a multiple of 16 bytes.  Other inputs take a
 *   slower plain-load path with the same results contract; this is not an
 *   error.
 */
#ifndef DUALMV_H
#define DUALMV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum dualmv_status {
    DUALMV_SUCCESS = 0,
    DUALMV_ERR_INVALID_VALUE = 1,
    DUALMV_ERR_ALLOC = 2,
    DUALMV_ERR_LAUNCH = 3,
    DUALMV_ERR_TIMEOUT = 4,
    DUALMV_ERR_UNSUPPORTED = 5,
    DUALMV_ERR_TOO_LARGE = 6
} dualmv_status;

/* Opaque CUDA stream handle (the same pointer as cudaStream_t). */
typedef struct CUstream_st *dualmv_stream_t;

/* ---- single problem ----------------------------------------------------
 * BICG (Table 1 / Table 2): q = A p and s = A^T r from one read of A.
 * f32: float inputs, float accumulation and outputs.
 * f64: double inputs, double accumulation and outputs.
 * i32: int32 inputs, products and sums in 64 bits with wrap-around modulo
 *      2^64, int64 outputs (bit-exact in any summation order). */
dualmv_status dualmv_f32(int64_t M, int64_t N, const float *A, int64_t lda,
                         const float *p, const float *r, float *q, float *s,
                         dualmv_stream_t stream);
dualmv_status dualmv_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                         const double *p, const double *r, double *q,
                         double *s, dualmv_stream_t stream);
dualmv_status dualmv_i32(int64_t M, int64_t N, const int32_t *A, int64_t lda,
                         const int32_t *p, const int32_t *r, int64_t *q,
                         int64_t *s, dualmv_stream_t stream);

/* ---- strided batch -----------------------------------------------------
 * `batch` independent problems of the same shape (BICG, Table 1 / Table 2,
 * applied to each).  Problem b uses A + b*strideA, p + b*strideP,
 * r + b*strideR and writes q + b*strideQ, s + b*strideS (strides in
 * elements).  Input strides may be 0 (the same operand for every problem).
 * When batch > 1, strideQ >= M and strideS >= N are required so that the
 * outputs of different problems do not overlap. */
dualmv_status dualmv_f32_strided_batched(
    int64_t M, int64_t N, const float *A, int64_t lda, int64_t strideA,
    const float *p, int64_t strideP, const float *r, int64_t strideR,
    float *q, int64_t strideQ, float *s, int64_t strideS, int64_t batch,
    dualmv_stream_t stream);
dualmv_status dualmv_f64_strided_batched(
    int64_t M, int64_t N, const double *A, int64_t lda, int64_t strideA,
    const double *p, int64_t strideP, const double *r, int64_t strideR,
    double *q, int64_t strideQ, double *s, int64_t strideS, int64_t batch,
    dualmv_stream_t stream);
dualmv_status dualmv_i32_strided_batched(
    int64_t M, int64_t N, const int32_t *A, int64_t lda, int64_t strideA,
    const int32_t *p, int64_t strideP, const int32_t *r, int64_t strideR,
    int64_t *q, int64_t strideQ, int64_t *s, int64_t strideS, int64_t batch,
    dualmv_stream_t stream);

/* ---- operations built on the same streaming kernels --------------------
 * Three more kernels the paper tunes (Table 1 and Table 2), built from the
 * dual product's streaming kernels run single-sided (rows only or columns
 * only, every pass reading its matrix once), and for ATAX from a cluster
 * form of them that reads A once.
 * Conventions as above (row-major, caller-owned device memory, asynchronous
 * on `stream`, stream-ordered scratch from the library's pool).
 *
 * GESUMMV (Table 1 / Table 2, row "GESUMMV"): with A and B both M x N
 * (leading dimensions lda, ldb >= max(1, N)), x of length N and y of
 * length M:  tmp = A x;  y = B x;  y = alpha * tmp + beta * y.
 * Floating-point sums have a fixed order (deterministic).  y must not
 * overlap A, B or x: the pass over B may start while the pass over A still
 * reads (the two share no buffer).  Errors as for dualmv_f32:
 * DUALMV_ERR_INVALID_VALUE for bad sizes or NULL pointers with nonzero
 * extents; N == 0 sets y to zero. */
dualmv_status dualmv_gesummv_f32(int64_t M, int64_t N, float alpha, const float *A,
                                 int64_t lda, float beta, const float *B, int64_t ldb,
                                 const float *x, float *y, dualmv_stream_t stream);
dualmv_status dualmv_gesummv_f64(int64_t M, int64_t N, double alpha, const double *A,
                                 int64_t lda, double beta, const double *B, int64_t ldb,
                                 const double *x, double *y, dualmv_stream_t stream);

/* ATAX (Table 1, row "ATAX"): with A M x N (lda >= max(1, N)), x of length
 * N and y of length N:  tmp = A x (length M);  y = A^T tmp.  The second
 * product needs all of tmp; see dualmv_atax_set_two_pass below for when A
 * is read once and when twice.  Floating-point sums have a fixed order
 * (deterministic).  M == 0 sets y to zero. */
dualmv_status dualmv_atax_f32(int64_t M, int64_t N, const float *A, int64_t lda,
                              const float *x, float *y, dualmv_stream_t stream);
dualmv_status dualmv_atax_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                              const double *x, double *y, dualmv_stream_t stream);

/* ATAX with one read of A.  A problem whose base is 16-byte aligned, whose
 * row stride lda * sizeof(element) is a multiple of 16 bytes and whose
 * width fits a thread-block cluster of at most 16 CTAs streams A once: the
 * CTAs of a cluster share each 4-row stripe (each CTA a slice of the
 * columns: 16 warps x 256 columns = 4096 for fp32; 8 sub-bands x 256 = 2048
 * for fp64, each sub-band with a warp for its row sums and one for its
 * column sums), exchange the stripe's partial row sums through distributed
 * shared memory, and form A^T tmp from the copy still on chip.  So fp32 takes this
 * path for N <= 65536 and fp64 (in double-float arithmetic on the FP32
 * pipes, native fp64 for stripes with values outside [2^-40, 2^40)) for
 * N <= 32768, when the GPU can place such a cluster.  Other problems read A
 * twice: a rows-only pass (tmp = A x), then a columns-only pass.
 * dualmv_atax_set_two_pass(1) forces the two-pass path for every problem
 * (tests, benchmarks); 0 restores the choice.  Returns the previous setting. */
int dualmv_atax_set_two_pass(int two_pass);

/* Which path the calling thread's last ATAX call with M > 0 and N > 0 took:
 * DUALMV_ATAX_ONE_READ (the cluster kernel) or DUALMV_ATAX_TWO_PASS; -1
 * after an empty problem or an error.  Instrumentation for tests. */
enum { DUALMV_ATAX_TWO_PASS = 0, DUALMV_ATAX_ONE_READ = 1 };
int32_t dualmv_atax_last_path(void);

/* GEMVER (Table 1 / Table 2, row "GEMVER"): with A M x N (lda >= max(1, N)),
 * u1, u2, w, y of length M and v1, v2, x, z of length N:
 *     A_hat = A + u1 v1^T + u2 v2^T
 *     x     = x + beta * A_hat^T y + z        (x is read and written)
 *     w     = w + alpha * A_hat x             (w is read and written)
 * w depends on all of the new x, so A is streamed twice: a columns-only
 * pass (A_hat^T y), then a rows-only pass (A_hat x).  Without update_A
 * (the default use) the rank-2 update is factorised (see
 * dualmv_gemver_set_onthefly): the passes are the plain streaming kernels,
 * in double-float arithmetic on the FP32 pipes for fp64.  With update_A
 * nonzero the rows-only pass also writes A_hat over A (as the PolyBench
 * kernel does), each element read before it is written by the same thread:
 *   - A 16-byte aligned and lda * sizeof(element) a multiple of 16: the
 *     columns-only pass and the x update are those of the factorised form;
 *     one rows pass writes A_hat = fma(u2_i, v2_j, fma(u1_i, v1_j, a)) and
 *     forms A x + u1 (v1 . x) + u2 (v2 . x) from the original A (fp64:
 *     A_hat in native fp64, A x in double-float, native fp64 for rows or
 *     bands with values outside [2^-40, 2^40), zeros excepted);
 *   - otherwise both passes form A_hat element by element as they stream
 *     A (native fp64 arithmetic for fp64).
 * The written A_hat is the same fused form on every path. */
dualmv_status dualmv_gemver_f32(int64_t M, int64_t N, float alpha, float beta, float *A,
                                int64_t lda, int update_A, const float *u1, const float *v1,
                                const float *u2, const float *v2, float *w, float *x,
                                const float *y, const float *z, dualmv_stream_t stream);
dualmv_status dualmv_gemver_f64(int64_t M, int64_t N, double alpha, double beta, double *A,
                                int64_t lda, int update_A, const double *u1, const double *v1,
                                const double *u2, const double *v2, double *w, double *x,
                                const double *y, const double *z, dualmv_stream_t stream);

/* How GEMVER applies the rank-2 update when A is not to be overwritten
 * (update_A == 0).  By default it uses the factorisation
 * A_hat^T y = A^T y + v1 (u1 . y) + v2 (u2 . y) and
 * A_hat x = A x + u1 (v1 . x) + u2 (v2 . x): a columns-only and a rows-only
 * pass of the plain kernels plus four dot products (fp64 sums in a fixed
 * order, compensated per thread when a thread adds more than 64 products;
 * error within about 80 u of the products' magnitudes), with no
 * per-element update.  dualmv_gemver_set_onthefly(1) makes
 * it form A_hat element by element as it streams A, as it always does with
 * update_A (tests, benchmarks).  Returns the previous setting. */
int dualmv_gemver_set_onthefly(int onthefly);

/* Which form the calling thread's last GEMVER call took:
 * DUALMV_GEMVER_FACTORED (update_A == 0 without the on-the-fly setting),
 * DUALMV_GEMVER_UPDATE_SPLIT (update_A, aligned rows: the factorised
 * columns pass and the rows pass that writes A_hat, above) or
 * DUALMV_GEMVER_ONTHEFLY (A_hat formed element by element); -1
 * after an empty problem or an argument error.  Instrumentation for tests. */
enum { DUALMV_GEMVER_FACTORED = 0, DUALMV_GEMVER_ONTHEFLY = 1, DUALMV_GEMVER_UPDATE_SPLIT = 2 };
int32_t dualmv_gemver_last_path(void);

/* ---- single problem without allocation --------------------------------
 * The paper has no counterpart to this entry point; it exists for callers
 * that cannot allocate device memory during the call: code inside a
 * framework that owns every device allocation (a fixed memory budget or an
 * allocator dualmv cannot see), real-time loops that must not enter an
 * allocator, and hot streams that must not gain pool-growing calls.
 *
 * Same operation, arguments and results contract as dualmv_f32, but the
 * scratch that holds partial sums between the two kernels is a fixed
 * device array inside the library (dualmv_f32_noalloc_scratch_bytes(),
 * 8 MiB), held by every GPU that loads the library until the process
 * exits.  The call makes no cudaMalloc, cudaFree or pool allocation.
 * The caller still passes A, p, r, q and s.
 *
 * Limit: the row partials need ceil(N / 256) * M * 4 bytes (none when
 * N <= 256), and the column partials 1 KiB for every CTA and band it
 * touches (usually two): about 0.3 MiB on the TMA path (one CTA per SM,
 * 152 on GB300) and 1.2 MiB on the plain-load path (four per SM), more for
 * very short matrices.  A 16384 x 16384 matrix fits, a 32768 x 16384 one
 * does not.  Larger problems return DUALMV_ERR_TOO_LARGE and enqueue
 * nothing.
 * Set-up: the first call on each device looks up the SM count and the
 * device address of the array (cudaGetSymbolAddress) with that device
 * current; make that first call before any stream capture.
 * Sharing: every call on a device uses the same array, and each call fully
 * rewrites the part it reads, so nothing carries over from one call to the
 * next.  Calls that can overlap on the GPU (different streams without
 * ordering between them) race on the array and give wrong results; order
 * them on one stream or with events. */
dualmv_status dualmv_f32_noalloc(int64_t M, int64_t N, const float *A,
                                 int64_t lda, const float *p, const float *r,
                                 float *q, float *s, dualmv_stream_t stream);

/* Size in bytes of the fixed scratch array used by dualmv_f32_noalloc. */
int64_t dualmv_f32_noalloc_scratch_bytes(void);

/* ---- diagnostics and control ------------------------------------------ */

/* Static English text for a status code ("unknown status" otherwise). */
const char *dualmv_status_string(dualmv_status status);

/* cudaError_t value of the most recent CUDA failure seen by this thread
 * (0 if none).  Reading it does not clear it. */
int dualmv_last_cuda_error(void);

/* Synchronises `stream`, then reads and clears the current device's fault
 * word.  Returns DUALMV_ERR_TIMEOUT if any kernel of this library gave up a
 * bounded wait (a pipeline barrier that never completed) since the last
 * read, DUALMV_ERR_LAUNCH if the synchronisation itself failed, and
 * DUALMV_SUCCESS otherwise.  A kernel that gives up writes no output it has
 * not finished; the outputs of that call are then unspecified. */
dualmv_status dualmv_device_fault(dualmv_stream_t stream);

/* The library's stream-ordered workspace pool on `device` (created by the
 * first call that needs it on that device, or by this call): bytes it holds
 * now, and the high-water mark of bytes in use since the last reset.  With
 * reset_high nonzero the mark is reset to the current use after it is read.
 * Returns DUALMV_ERR_INVALID_VALUE for a bad device or NULL outputs.
 * Diagnostics for tests: a call that takes no workspace leaves the mark at
 * the use it had before the call. */
dualmv_status dualmv_pool_usage(int device, int64_t *reserved_bytes, int64_t *used_high_bytes,
                                int reset_high);

/* Which kernel streams A.  DUALMV_PATH_AUTO (default) uses the TMA pipeline
 * when the alignment rules above hold and the plain-load kernel otherwise;
 * DUALMV_PATH_TMA and DUALMV_PATH_DIRECT force one of them (TMA falls back
 * to plain loads when the alignment rules do not hold).  On the TMA path,
 * fp64 products and sums run in double-float arithmetic on the FP32 pipes
 * (GB300's FP64 pipe is far slower than its HBM), with native fp64 FMA for
 * any rows holding values outside [2^-40, 2^40) (zero excepted);
 * DUALMV_PATH_TMA_NATIVE_F64 makes the TMA path use native fp64 FMA for
 * all of them.  Process-wide; meant for tests and tuning.  Returns the
 * previous setting, or -1 for an unknown value. */
enum {
    DUALMV_PATH_AUTO = 0,
    DUALMV_PATH_TMA = 1,
    DUALMV_PATH_DIRECT = 2,
    DUALMV_PATH_TMA_NATIVE_F64 = 3
};
int dualmv_set_path(int path);

/* Instrumentation for benchmarks: the next dualmv call made by this thread
 * records `start` (a cudaEvent_t) on its stream just before it launches its
 * streaming kernel and `stop` just after, so that the streaming kernel can be
 * timed on the stream it runs on.  The events are used once and forgotten;
 * pass NULL, NULL to cancel.  Calls that launch no streaming kernel (empty
 * problems, invalid arguments) leave the request pending. */
void dualmv_record_kernel_events(void *start, void *stop);

/* Instrumentation for benchmarks, not part of the method: reads `bytes`
 * bytes of device memory at `buf` once with 16-byte loads spread over every
 * SM, and xor-folds them into the device word *out (its value means
 * nothing; it keeps the loads alive).  `buf` must be 16-byte aligned and
 * `bytes` a multiple of 16 (else DUALMV_ERR_INVALID_VALUE, nothing
 * enqueued).  Asynchronous on `stream`.  Timed over a buffer larger than
 * L2, it gives the read-only bandwidth ceiling that the streaming kernels
 * are compared with beside the measured copy bandwidth. */
dualmv_status dualmv_read_probe(const void *buf, int64_t bytes, uint32_t *out,
                                dualmv_stream_t stream);

/* Instrumentation for the failure-detection tests, not part of the method:
 * enqueues on `stream` one warp that waits for an mbarrier phase that
 * nothing completes, through the same bounded waits as the library's
 * kernels (CTA scope if cluster_scope == 0, the cluster kernels' cluster
 * scope otherwise).  After about 2 s the wait gives up: it sets the device
 * fault word, so the next dualmv_device_fault returns DUALMV_ERR_TIMEOUT,
 * and the kernel exits normally, leaving the context usable.  The device
 * int32 *waited receives 0 when the wait ran out, 1 if it returned without
 * running out (which nothing can make it do).  DUALMV_ERR_INVALID_VALUE for
 * a NULL `waited`, nothing enqueued. */
dualmv_status dualmv_selftest_wait_timeout(int cluster_scope, int32_t *waited,
                                          dualmv_stream_t stream);

/* ---- planner (pure host code, no CUDA call) ----------------------------
 * The work decomposition a call would use.  A is cut into column bands of
 * `band_cols` columns and row stripes of `tile_rows` rows; a tile is one
 * stripe of one band of one problem.  Tiles are numbered band-major
 * (problem, band, stripe) and CTA c of `grid` owns the contiguous range
 * [floor(c*tiles/grid), floor((c+1)*tiles/grid)).  A band split between
 * CTAs leaves one column partial per CTA ("segment"); row partials of
 * different bands are combined by a second kernel in ascending band order,
 * column partials in ascending CTA order.  `num_sms` is the SM count to plan
 * for.  Returns DUALMV_ERR_INVALID_VALUE for bad shapes or elem_bytes not
 * in {4, 8}. */
typedef struct dualmv_plan_t {
    int64_t band_cols;      /* columns per band (tile width)              */
    int64_t tile_rows;      /* rows per tile (stripe height)              */
    int64_t bands;          /* column bands per problem                   */
    int64_t stripes;        /* row stripes per problem                    */
    int64_t tiles;          /* batch * bands * stripes                    */
    int64_t grid;           /* CTAs launched (persistent)                 */
    int64_t max_segments;   /* most band segments one CTA can own         */
    int64_t workspace_bytes;/* stream-ordered scratch the call allocates  */
    int64_t smem_bytes;     /* dynamic shared memory per CTA              */
    int64_t threads;        /* threads per CTA                            */
} dualmv_plan_t;

dualmv_status dualmv_plan(int64_t M, int64_t N, int64_t batch,
                          int64_t elem_bytes, int64_t acc_bytes,
                          int64_t num_sms, dualmv_plan_t *out);

/* ---- kernel variants and the variant tuner (Section 3.2, Eq. 3-5) ------
 * The dual product of one unbatched problem on the TMA path can run any of
 * several compiled variants of its streaming kernel, which differ in tile
 * shape (consumer warps x rows per warp), TMA ring depth and, for fp64,
 * arithmetic (double-float on the FP32 pipes, or native fp64 FMA).  Entry 0
 * of each element type's table is the default that untuned calls use.
 * Batched calls, single-sided products (GESUMMV, ATAX, GEMVER) and the
 * plain-load path always use their default kernel.  Untuned calls use
 * entry 0, except int32 problems whose base or row stride is not a multiple
 * of 128 bytes, which use the first DUALMV_KERNEL_WIDE entry: with such
 * rows a 256-column box row straddles a 128-byte line that the next band
 * fetches again, and the wide tiles read W KiB of each row at once. */
enum { DUALMV_DTYPE_F32 = 0, DUALMV_DTYPE_F64 = 1, DUALMV_DTYPE_I32 = 2 };
enum {
    DUALMV_KERNEL_STREAM = 0, /* TMA ring, native arithmetic of the dtype  */
    DUALMV_KERNEL_F64E = 1,   /* TMA ring per warp, double-float fp64      */
    DUALMV_KERNEL_WIDE = 2,   /* int32: tiles of rows_per_warp rows by     */
                              /* warps * 256 columns, one 256-column       */
                              /* sub-band per warp                         */
    DUALMV_KERNEL_PHASED = 3, /* rows whose stride or base is not 16-byte  */
                              /* aligned: TMA through one pair of tensor   */
                              /* maps per row phase (no variants; fp64 in  */
                              /* double-float arithmetic)                  */
    DUALMV_KERNEL_PLAIN = 4,  /* plain global loads (no variants)          */
    DUALMV_KERNEL_CLUSTER = 5 /* small fp32 problems: one cluster of 16    */
                              /* CTAs does the whole call (no variants)   */
};
typedef struct dualmv_variant_t {
    int32_t index;          /* position in its dtype's table              */
    int32_t kernel;         /* DUALMV_KERNEL_*                            */
    int32_t warps;          /* consumer warps per CTA                     */
    int32_t rows_per_warp;  /* rows of a tile per consumer warp           */
    int32_t stages;         /* TMA ring depth                             */
    int32_t band_cols;      /* columns per band                           */
    int32_t tile_rows;      /* warps * rows_per_warp                      */
    int32_t threads;        /* threads per CTA (consumers + producer)     */
    int32_t native_cols;    /* DUALMV_KERNEL_F64E: of each lane's 8       */
                            /* columns, how many sum s with native fp64   */
                            /* FMA (0 for the other kernels)              */
    int32_t producer_warp;  /* 1: a dedicated TMA producer warp feeds the  */
                            /* consumers; 0: each consumer warp issues its */
                            /* own boxes (threads = warps * 32)            */
    int32_t packed;         /* DUALMV_KERNEL_F64E: 1 if the double-float   */
                            /* arithmetic of column pairs runs as packed   */
                            /* FP32x2 instructions                         */
    int32_t batched;        /* 1 if the variant also runs strided batches  */
                            /* (a 3-D tensor-map instance), so that        */
                            /* dualmv_tune_*_strided_batched may choose it */
    int32_t single_sided;   /* 1 if it also runs single-sided passes (q    */
                            /* only, s only: GESUMMV, GEMVER, ATAX's two   */
                            /* passes), so that dualmv_tune_pass_* may     */
                            /* choose it                                   */
    int32_t pad_;           /* zero                                        */
    int64_t smem_bytes;     /* dynamic shared memory per CTA              */
} dualmv_variant_t;

/* Number of variants for `dtype` (DUALMV_DTYPE_*), or -1 for an unknown
 * dtype.  Host only. */
int32_t dualmv_variant_count(int32_t dtype);

/* Description of variant `index` of `dtype`.  DUALMV_ERR_INVALID_VALUE for
 * an unknown dtype, an index out of range or a NULL `out`.  Host only. */
dualmv_status dualmv_variant_info(int32_t dtype, int32_t index, dualmv_variant_t *out);

/* Forces variant `index` for every eligible call of `dtype` in this
 * process (-1 restores the normal choice: a tuned variant for the shape if
 * dualmv_tune_* recorded one, else entry 0).  A strided-batched call runs
 * the forced variant if it has a batched instance, and a single-sided pass
 * (of GESUMMV, GEMVER's columns pass, ATAX's two passes) if it has
 * single-sided instances; else entry 0.  Without a forced or tuned variant,
 * fp64 single-sided passes run entry 1 (8 warps x 4 rows), which their
 * half-size arithmetic suits better than entry 0's 12 warps.  Returns the previous setting, or
 * -2 for an unknown dtype or an index out of range.  Meant for tests. */
int32_t dualmv_set_variant(int32_t dtype, int32_t index);

/* The variant recorded by dualmv_tune_* for this dtype and shape (one
 * problem), or -1. */
int32_t dualmv_tuned_variant(int32_t dtype, int64_t M, int64_t N, int64_t lda);

/* The variant recorded by dualmv_tune_*_strided_batched for this dtype,
 * shape and batch count (batch 1: as dualmv_tuned_variant), or -1. */
int32_t dualmv_tuned_variant_batched(int32_t dtype, int64_t M, int64_t N, int64_t lda,
                                     int64_t batch);

/* The variant recorded by dualmv_tune_pass_* for this dtype, shape and
 * pass (DUALMV_PASS_ROWS or DUALMV_PASS_COLS), or -1. */
int32_t dualmv_tuned_variant_pass(int32_t dtype, int64_t M, int64_t N, int64_t lda,
                                  int32_t pass);

/* Forgets every recorded tuning result. */
void dualmv_tune_clear(void);

/* The variant the calling thread's last dual-product call or single-sided
 * pass launched (one problem or a strided batch): its table index, or -1
 * if that call ran no variant of the table (an empty problem, the phased,
 * plain-load or single-cluster path, an fp32 single-sided pass on its
 * default kernel (entry 0's shape, also walking its tiles backwards),
 * native fp64 by default, or an error).  Untuned fp64 single-sided passes,
 * GEMVER's backward rows pass among them, run entry 1 and report it.
 * Instrumentation for tests and benchmarks. */
int32_t dualmv_last_variant(void);

/* The kind of streaming kernel (DUALMV_KERNEL_*) that the calling thread's
 * last dual product ran (dualmv_f32/f64/i32 and their strided-batched forms,
 * and the passes inside GESUMMV, ATAX and GEMVER), or -1 if it ran none (an
 * empty problem or an error).  PHASED: rows whose stride or base the TMA
 * unit cannot take as one tensor, for one dual product (fp64 unless
 * DUALMV_PATH_TMA_NATIVE_F64 is set); PLAIN: the remaining unaligned cases;
 * CLUSTER: one fp32 dual product of at most 8 MiB with 256 <= N <= 2048
 * (N and lda multiples of 4, A and p 16-byte aligned), under
 * DUALMV_PATH_AUTO and with no variant forced or tuned for it, which one
 * cluster of 16 CTAs computes without workspace or combine kernel.
 * Instrumentation for tests and benchmarks. */
int32_t dualmv_last_kernel(void);

/* Trimmed mean of Eq. 3: the R values sorted, the k smallest and k largest
 * dropped, the rest averaged.  DUALMV_ERR_INVALID_VALUE unless R > 2k,
 * k >= 0 and both pointers are non-NULL.  Host only; `t` is not modified. */
dualmv_status dualmv_trimmed_mean(const double *t, int64_t R, int64_t k, double *out);

typedef struct dualmv_tune_config_t {
    int32_t repeats;     /* R timed calls per candidate (R > 2 * trim)        */
    int32_t trim;        /* k of Eq. 3                                        */
    int32_t max_rounds;  /* D: rounds of candidate generation at most         */
    int32_t candidates;  /* N: candidates per round at most (>= 1)            */
    double min_gain;     /* stop once a round's best candidate is not faster  */
                         /* than the baseline by at least this fraction       */
    int32_t flush_l2;    /* nonzero: write a buffer of twice the L2 size      */
                         /* before every timed call, outside its events       */
} dualmv_tune_config_t;

/* One evaluated candidate, in evaluation order. */
typedef struct dualmv_tune_step_t {
    int32_t index;       /* variant                                           */
    int32_t round;       /* d (0-based)                                       */
    int32_t feasible;    /* passed functional equivalence (Eq. 4)             */
    int32_t pad_;
    double ms;           /* trimmed mean (Eq. 3); 0 if not feasible           */
    double fe;           /* largest per-element error against the baseline   */
} dualmv_tune_step_t;

#define DUALMV_TUNE_MAX_TRACE 64

typedef struct dualmv_tune_result_t {
    int32_t best;        /* index of the chosen variant (the final baseline)  */
    int32_t rounds;      /* rounds run                                        */
    int32_t evaluated;   /* candidates run, the initial baseline excluded     */
    int32_t rejected;    /* candidates that failed functional equivalence     */
    double baseline_ms;  /* trimmed mean of K^(0)                             */
    double best_ms;      /* trimmed mean of the chosen variant                */
    double worst_fe;     /* largest FE error among accepted candidates        */
    int32_t trace_len;   /* entries of `trace` filled (min(evaluated, max))  */
    int32_t initial;     /* index of K^(0), the shape's untuned variant       */
    dualmv_tune_step_t trace[DUALMV_TUNE_MAX_TRACE];
} dualmv_tune_result_t;

/* Tunes the variant for this problem by the loop of Section 3.2:
 *   K^(0) = the variant an untuned call of this shape uses (see above).  In
 *   round d, up to `candidates` variants not tried
 *   before that differ from K^(d) in one property (kernel, warps, rows per
 *   warp, stages or native columns) are run once and checked for functional equivalence
 *   with K^(d) (Eq. 4); each that passes is timed `repeats` times and
 *   scored by the trimmed mean of Eq. 3.  The fastest feasible candidate
 *   (Eq. 5) becomes K^(d+1) if it beats K^(d) by more than `min_gain`;
 *   otherwise, or after `max_rounds` rounds, or when no untried neighbour is
 *   left, the loop stops.
 * Functional equivalence: int32 outputs equal bit for bit; floating-point
 *   outputs within the parity bar |x - x_base| <= tol * sum|A||v| per
 *   element (tol 1e-5 for f32, 1e-12 for f64), the sums |A||p| and |A|^T|r|
 *   computed in double by separate simple kernels.
 * The chosen variant is recorded for (dtype, M, N, lda) and used by later
 *   calls of that shape (see dualmv_tuned_variant), and its outputs are
 *   left in q and s.
 * Synchronous: blocks the calling thread on `stream` while it measures.
 *   Allocates its scratch from the library's pool on `stream`.
 * Errors: DUALMV_ERR_INVALID_VALUE for the dualmv_* argument errors, NULL
 *   `cfg` or `res`, repeats <= 2 * trim, trim < 0, max_rounds < 0,
 *   candidates < 1 or a negative or NaN min_gain (nothing enqueued);
 *   DUALMV_ERR_TIMEOUT if a candidate's kernel gave up a bounded wait;
 *   otherwise as dualmv_*.  Problems off the TMA path (misaligned A,
 *   DUALMV_PATH_DIRECT or DUALMV_PATH_TMA_NATIVE_F64 in force) and empty
 *   problems run the default once and report evaluated = 0. */
dualmv_status dualmv_tune_f32(int64_t M, int64_t N, const float *A, int64_t lda,
                              const float *p, const float *r, float *q, float *s,
                              const dualmv_tune_config_t *cfg,
                              dualmv_tune_result_t *res, dualmv_stream_t stream);
dualmv_status dualmv_tune_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                              const double *p, const double *r, double *q, double *s,
                              const dualmv_tune_config_t *cfg,
                              dualmv_tune_result_t *res, dualmv_stream_t stream);
dualmv_status dualmv_tune_i32(int64_t M, int64_t N, const int32_t *A, int64_t lda,
                              const int32_t *p, const int32_t *r, int64_t *q, int64_t *s,
                              const dualmv_tune_config_t *cfg,
                              dualmv_tune_result_t *res, dualmv_stream_t stream);

/* The same loop for a strided batch (arguments as
 * dualmv_*_strided_batched, then cfg, res, stream).  Candidates are the
 * variants with a batched instance (dualmv_variant_t.batched); K^(0) is
 * entry 0; Eq. 4 compares every problem's outputs; the choice is recorded
 * for (dtype, M, N, lda, batch) and used by later strided-batched calls of
 * that shape (dualmv_tuned_variant_batched).  batch == 1 tunes one problem
 * as dualmv_tune_*.  Blocks until done. */
dualmv_status dualmv_tune_f32_strided_batched(
    int64_t M, int64_t N, const float *A, int64_t lda, int64_t strideA, const float *p,
    int64_t strideP, const float *r, int64_t strideR, float *q, int64_t strideQ, float *s,
    int64_t strideS, int64_t batch, const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
    dualmv_stream_t stream);
dualmv_status dualmv_tune_f64_strided_batched(
    int64_t M, int64_t N, const double *A, int64_t lda, int64_t strideA, const double *p,
    int64_t strideP, const double *r, int64_t strideR, double *q, int64_t strideQ, double *s,
    int64_t strideS, int64_t batch, const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
    dualmv_stream_t stream);
dualmv_status dualmv_tune_i32_strided_batched(
    int64_t M, int64_t N, const int32_t *A, int64_t lda, int64_t strideA, const int32_t *p,
    int64_t strideP, const int32_t *r, int64_t strideR, int64_t *q, int64_t strideQ, int64_t *s,
    int64_t strideS, int64_t batch, const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
    dualmv_stream_t stream);

/* The same loop for one single-sided pass, the building block of GESUMMV
 * (rows: q = A x), GEMVER (its columns pass: s = A^T y) and ATAX's two-pass
 * fallback (both): pass DUALMV_PASS_ROWS computes out = A x (x of length N,
 * out of length M), DUALMV_PASS_COLS out = A^T x (x of length M, out of
 * length N).  Candidates are the variants with single-sided instances
 * (dualmv_variant_t.single_sided: every fp32 shape, the packed
 * self-loading fp64 shapes); K^(0) is the passes' default, entry 0 for
 * fp32 and entry 1 (8 warps x 4 rows) for fp64; Eq. 4 compares `out`.  The
 * choice is recorded for (dtype, M, N, lda, pass) and used by later
 * single-sided passes of that shape that walk their tiles forwards
 * (dualmv_tuned_variant_pass; GEMVER's rows pass, which walks backwards to
 * start on tiles still in L2, runs the passes' default shape).  The chosen
 * variant's
 * result is left in `out`.  DUALMV_ERR_INVALID_VALUE for an unknown pass
 * and the argument errors of dualmv_tune_*; blocks until done. */
enum { DUALMV_PASS_ROWS = 1, DUALMV_PASS_COLS = 2 };
dualmv_status dualmv_tune_pass_f32(int64_t M, int64_t N, const float *A, int64_t lda,
                                   int32_t pass, const float *x, float *out,
                                   const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
                                   dualmv_stream_t stream);
dualmv_status dualmv_tune_pass_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                                   int32_t pass, const double *x, double *out,
                                   const dualmv_tune_config_t *cfg, dualmv_tune_result_t *res,
                                   dualmv_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* DUALMV_H */
