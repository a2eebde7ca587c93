/*
 * tcu_dft.h -- C ABI of the GB300 (sm_103a) batched complex DFT.
 *
 * The operation (arXiv 1908.06649, Sec. 4.5): the DFT of an n-vector x is
 * y = x^T W with the symmetric Fourier matrix W[r][c] = exp(-(2 pi i/n) r c).
 * It is computed with the paper's Cooley-Tukey scheme for the (m, l)-TCU
 * (Sec. 4.5, Theorem 7): with sqrt(m) = r and n = r^k, each of the k stages is
 * one tall-left product of the (batch*n/r) x r data matrix with the r x r DFT
 * matrix F_r (X^T W_sqrt(m)), followed by the element-wise twiddle multiply
 * w_n^{rc} and the transposition that feeds the next stage.  A complex r x r
 * product is done as real arithmetic (Sec. 4.5: four real products and two
 * sums), here as one real (2r x 2r) block operand [[Re, Im], [-Im, Re]] on the
 * tensor cores (tcgen05, kind::tf32, accumulating in tensor memory).
 *
 * Conventions
 *   forward : y_k = sum_j x_j exp(-2 pi i j k / n), unscaled.
 *   inverse : x_j = (1/n) sum_k y_k exp(+2 pi i j k / n) (the paper defines
 *             only the forward transform; this is the numpy/torch
 *             "backward" normalisation).
 *   Output is in natural order.
 *
 * Data layout (all entry points): `batch` transforms of length n, stored
 * contiguously, transform-major, as interleaved complex64 (float re, float
 * im): element j of transform b is at ((float2*)ptr)[b*n + j].  Device
 * pointers must be 16-byte aligned.
 *
 * Threading: plans are independent objects; one plan must not be executed
 * concurrently on two streams (its scratch is shared).  tcu_dft_last_error()
 * is thread-local.
 *
 * Diagnostics (environment, read at each call):
 *   TCU_DFT_DEBUG=1       every exec call synchronises its stream and returns
 *                         the plan's error word (as the *_check calls)
 *                         instead of returning once the launches are queued.
 *   TCU_DFT_FAIL_ALLOC=k  host-side fault injection for tests: the k-th
 *                         device allocation of each plan call (k >= 1) fails
 *                         as if the device were out of memory; the plan call
 *                         then frees what it had and returns NULL with
 *                         ERR_OOM.
 * Each pass's launches sit in an NVTX range ("tcu_dft pass 1", ...; the 2-D
 * calls "tcu_dft2", "tcu_conv2", "tcu_stencil").  The library is also built
 * with every shared-memory, tensor-memory and global index of the pass
 * kernels checked (libtcu_dft_checked.so, -DTCU_DFT_CHECKED): an index out
 * of range skips the access and records ERR_BOUNDS in the plan's error word.
 */
#ifndef TCU_DFT_H
#define TCU_DFT_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct tcu_dft_plan_s *tcu_dft_plan_t;

/* precision: operand type and number of tensor products per stage.
 *   TCU_DFT_TF32    -- one TF32 product, operands rounded to TF32 (~1e-3
 *                      rel. L2)
 *   TCU_DFT_3XTF32  -- hi*hi + lo*hi + hi*lo TF32 split products (fp32-level)
 *   TCU_DFT_BF16    -- one BF16 product (kind::f16; ~1e-2 rel. L2), n = r^k
 *                      only (no mixed radix, no 2-D plans)
 *   TCU_DFT_3XBF16  -- the same three split products in BF16 (~1e-4), n = r^k
 *                      only
 * The BF16 modes are the low-precision variant (Sec. 4.5 cites half-precision
 * tensor-core FFTs): half the products of the TF32 modes per stage. */
enum { TCU_DFT_TF32 = 1, TCU_DFT_3XTF32 = 3, TCU_DFT_BF16 = 4, TCU_DFT_3XBF16 = 5 };

/* direction = sign of the exponent */
enum { TCU_DFT_FORWARD = -1, TCU_DFT_INVERSE = +1 };

/* status codes */
enum {
  TCU_DFT_OK = 0,
  TCU_DFT_ERR_INVALID = 1,     /* bad argument (null, size, alignment, overlap) */
  TCU_DFT_ERR_UNSUPPORTED = 2, /* valid but not supported (radix, n not r^k, n too large) */
  TCU_DFT_ERR_CUDA = 3,        /* a CUDA runtime/driver call failed, or no sm_103 device */
  TCU_DFT_ERR_OOM = 4,         /* device allocation failed */
  TCU_DFT_ERR_TIMEOUT = 5,     /* a device-side wait hit its iteration limit */
  TCU_DFT_ERR_TOO_LARGE = 6,   /* beyond the fixed memory of tcu_dft_exec_noalloc */
  TCU_DFT_ERR_BOUNDS = 7       /* checked build: a kernel index was out of range */
};

/* Build a plan for `batch` forward/inverse DFTs of length n with radix
 * sqrt_m (the TCU side length sqrt(m) of Sec. 3; one of 8, 16, 32) and the
 * given precision.  n must equal sqrt_m^k for some k >= 1 (Theorem 7 assumes
 * all of n, n/sqrt(m), ... are integers).
 * The k stages run in up to three HBM passes of at most two stages each
 * (three for sqrt_m = 8), so n <= 16^6, 32^6 or 8^9.
 * Allocates the device tables (F_r operand images, twiddles) and, when n
 * needs several passes, one scratch buffer of batch*n complex64 values per
 * intermediate (two for three passes); uses the current CUDA device.  This
 * is the only call that allocates.
 * Returns NULL on error and sets tcu_dft_last_error():
 *   ERR_INVALID (n < 1, batch < 1, precision not one of TCU_DFT_TF32,
 *   TCU_DFT_3XTF32, TCU_DFT_BF16, TCU_DFT_3XBF16),
 *   ERR_UNSUPPORTED (sqrt_m not in {8,16,32}, n not a power of sqrt_m, n
 *   beyond three passes, or batch*n > 2^40), ERR_CUDA (no sm_103 device),
 *   ERR_OOM. */
tcu_dft_plan_t tcu_dft_plan(int64_t n, int64_t batch, int32_t sqrt_m,
                            int32_t precision);

/* Plan flags for tcu_dft_plan_ex.  By default a two-pass transform runs as
 * two kernel launches with a full batch*n intermediate in HBM. */
enum {
  TCU_DFT_PLAN_DEFAULT = 0,
  /* Explicitly the default two-launch schedule. */
  TCU_DFT_PLAN_NO_FUSE = 1,
  /* Run both passes in ONE fused launch whose intermediate is a small ring
   * of transforms kept in L2 (HBM then moves each point once in and once
   * out).  Only for two passes of >= 2 stages each; otherwise ignored. */
  TCU_DFT_PLAN_FUSE = 2,
  /* Run both passes in ONE launch on clusters of two CTAs (one per SM):
   * each cluster takes whole transforms, splits each one's pass-1 and
   * pass-2 work between its two CTAs and keeps the transform's
   * intermediate in one of two scratch slots of its own that stay in L2
   * (2 * clusters * n complex64 of scratch instead of batch * n); the
   * passes synchronise through mbarriers of the cluster.  HBM moves each
   * point once in and once out.  For sqrt_m = 16, n = 16^4 in TF32 or
   * 3xTF32; otherwise ignored.  Not with FUSE or NO_FUSE. */
  TCU_DFT_PLAN_ONE_PASS = 4
};

/* tcu_dft_plan with scheduling flags (TCU_DFT_PLAN_*); unknown bits, or
 * FUSE together with NO_FUSE, are rejected with ERR_INVALID.  Same results
 * either way. */
tcu_dft_plan_t tcu_dft_plan_ex(int64_t n, int64_t batch, int32_t sqrt_m,
                               int32_t precision, uint32_t flags);

/* 1 if the plan runs its two passes as one launch (TCU_DFT_PLAN_FUSE or
 * TCU_DFT_PLAN_ONE_PASS), 0 if not, -1 for a
 * NULL plan. */
int tcu_dft_is_fused(tcu_dft_plan_t p);

/* Forward transform: equivalent to tcu_dft_exec_dir(p, in, out,
 * TCU_DFT_FORWARD, stream). */
int tcu_dft_exec(tcu_dft_plan_t p, const void *in, void *out, void *stream);

/* Run the plan on `stream` (a cudaStream_t; NULL = legacy default stream).
 * in, out: device pointers to batch*n complex64 values (caller-owned,
 * 16-byte aligned).  in == out (full overlap) is allowed; partial overlap is
 * rejected with ERR_INVALID.  Asynchronous: no allocation and no host
 * synchronisation.  On an argument error nothing is launched.  Returns OK,
 * ERR_INVALID, or ERR_CUDA if a launch failed. */
int tcu_dft_exec_dir(tcu_dft_plan_t p, const void *in, void *out, int dir,
                     void *stream);

/* Same as tcu_dft_exec_dir, and records `events[i]` (cudaEvent_t handles,
 * caller-created) on `stream` just before pass i and events[npasses] after
 * the last pass, so the caller can time each pass kernel on the stream it
 * runs on.  `events` must hold tcu_dft_num_passes(p) + 1 entries. */
int tcu_dft_exec_timed(tcu_dft_plan_t p, const void *in, void *out, int dir,
                       void *stream, void *const *events);

/* End-to-end variant for host data: copies h_in (host, batch*n complex64;
 * pinned memory makes the copy asynchronous) into the caller-owned device
 * buffer d_work (batch*n complex64, 16-byte aligned), transforms it in place,
 * and copies the result to h_out (host).  All on `stream`; the call returns
 * after enqueuing (synchronise the stream before reading h_out).  Returns
 * OK, ERR_INVALID or ERR_CUDA. */
int tcu_dft_exec_host(tcu_dft_plan_t p, const void *h_in, void *h_out,
                      void *d_work, int dir, void *stream);

/* Synchronise `stream` and report whether any device-side wait of this
 * plan's kernels gave up (ERR_TIMEOUT) or, in the checked build, an index
 * was out of range (ERR_BOUNDS), then clear the flag.  OK otherwise;
 * ERR_CUDA if the synchronisation itself failed. */
int tcu_dft_check(tcu_dft_plan_t p, void *stream);

/* Free the plan's device memory (cudaFree synchronises the device).
 * Destroying NULL is a no-op returning OK. */
int tcu_dft_destroy(tcu_dft_plan_t p);

/* The pass grouping tcu_dft_plan would choose for n and sqrt_m, without
 * creating a plan or touching the GPU: returns the number of HBM passes (0
 * if n is not supported) and writes the stages of each pass to stages[0 ..
 * passes) (caller array of 3; the q-point pass of a mixed-radix n counts
 * as one stage). */
int tcu_dft_plan_passes(int64_t n, int32_t sqrt_m, int32_t *stages);

/* Plan introspection: number of HBM passes, and stages in pass i (0-based);
 * -1 for a NULL plan or an index out of range. */
int tcu_dft_num_passes(tcu_dft_plan_t p);
int tcu_dft_pass_stages(tcu_dft_plan_t p, int i);

/* Transform without allocating: for callers that may not allocate device
 * memory at all -- code running where memory belongs to someone else (a
 * framework's pool, a caching allocator, an embedding application) or where
 * a cudaMalloc would stall the device and break a latency budget.  The paper
 * has no counterpart; it is a service of this library.
 *
 * Same transform and arguments as tcu_dft_plan + tcu_dft_exec_dir, without
 * a plan: in, out are caller-owned device buffers of batch*n complex64
 * (16-byte aligned, in == out allowed), dir is TCU_DFT_FORWARD or
 * TCU_DFT_INVERSE, stream a cudaStream_t.  Every buffer it uses besides in
 * and out is a fixed array inside the library (the two-pass intermediate:
 * 4 Mi complex64 = 32 MiB; twiddle and F_r tables for n <= 2^18), present on
 * every GPU that loads the library until the process exits.  It never calls
 * cudaMalloc or cudaFree.
 *
 * Limits: n a power of sqrt_m that needs at most two passes (sqrt_m 16:
 * n <= 16^4; 8: n <= 8^4; 32: n <= 32^3) and n <= 2^18; when n needs two
 * passes, batch*n <= 2^22.  Larger requests return TCU_DFT_ERR_TOO_LARGE
 * with nothing launched; other argument errors ERR_INVALID / ERR_UNSUPPORTED
 * as tcu_dft_plan would.
 *
 * Argument errors (including a misaligned or partially overlapping buffer)
 * are found before any CUDA call.
 *
 * The first call on a device resolves the device addresses of those arrays
 * (with that device current) and fills the tables; make that first call
 * before any stream capture.  A later call with another n or sqrt_m refills
 * the tables from host memory, stream-ordered on `stream`: such a call must
 * not be captured either, and returns ERR_INVALID with nothing enqueued if
 * `stream` is capturing.  All calls share the arrays, which keep the last
 * call's contents: calls whose work overlaps on the GPU (other streams, other
 * host threads) race with each other.  Asynchronous like tcu_dft_exec_dir: a
 * device-side wait timeout is not reported by default; with TCU_DFT_DEBUG=1
 * in the environment the call synchronises `stream` and returns it
 * (ERR_TIMEOUT), as tcu_dft_check does for plans. */
int tcu_dft_exec_noalloc(int64_t n, int64_t batch, int32_t sqrt_m, int32_t precision,
                         const void *in, void *out, int dir, void *stream);

/* ---------------------------------------------------------------- 2-D
 * 2-D DFT and circular 2-D convolution (Sec. 4.6: a 2-D DFT is a 1-D DFT of
 * every row and of every column; Lemma 1 reduces stencils to batched
 * convolutions computed through it).  Arrays are row-major n1 x n2
 * complex64, batch-major (x[(b n1 + i) n2 + j]), 16-byte aligned, caller
 * owned.  n1 and n2 are powers of sqrt_m of at most one warpgroup pass each
 * (sqrt_m^2 for 16 and 32, 8^3 for 8) with n1 * n2 >= 128 sqrt_m.  Forward
 * unscaled; inverse with the conjugate exponent and 1/(n1 n2).
 * tcu_dft2_plan allocates its tables and one batch-size scratch array and
 * returns NULL with tcu_dft_last_error() set on error (ERR_INVALID,
 * ERR_UNSUPPORTED, ERR_CUDA, ERR_OOM).  The exec calls are asynchronous on
 * `stream`, allocate nothing, allow in == out and reject partial overlap
 * (ERR_INVALID) before launching. */
typedef struct tcu_dft2_plan_s *tcu_dft2_plan_t;
tcu_dft2_plan_t tcu_dft2_plan(int64_t n1, int64_t n2, int64_t batch, int32_t sqrt_m,
                              int32_t precision);
int tcu_dft2_exec(tcu_dft2_plan_t p, const void *in, void *out, int dir, void *stream);
/* out = IDFT2(DFT2(in) * spectrum) for every array of the batch: the
 * circular convolution of each array with the one n1 x n2 array whose 2-D
 * DFT is `spectrum` (device, n1*n2 complex64, e.g. from tcu_dft2_exec on a
 * batch-1 plan).  Three passes: columns; rows transformed, multiplied by
 * the spectrum and transformed back on chip; inverse columns. */
int tcu_conv2_exec(tcu_dft2_plan_t p, const void *in, const void *spectrum, void *out,
                   void *stream);
int tcu_dft2_check(tcu_dft2_plan_t p, void *stream);  /* as tcu_dft_check */
int tcu_dft2_destroy(tcu_dft2_plan_t p);                /* NULL: no-op, OK */

/* ------------------------------------------------------------- stencils
 * Linear (n, k)-stencil of Sec. 4.6 on a side x side row-major fp32 grid A
 * (device, caller owned): A_k[i][j] = sum over |a|, |b| <= k of
 * W[k+a][k+b] A[i+a][j+b], W the weight matrix of k sweeps of the 3 x 3
 * update w3x3[(a+1)*3 + (b+1)] (a, b in {-1, 0, 1}); cells outside the grid
 * are 0 at time 0 and the sweeps act on the free plane.
 * tcu_stencil_weights: W ((2k+1)^2 fp32, device) as the coefficients of
 *   P(x,y)^k (Lemma 2): P on an Nw x Nw grid, 2-D DFT, pointwise k-th power,
 *   inverse 2-D DFT, Nw the smallest power of sqrt_m >= 2k + 1.
 * tcu_stencil_exec: Lemma 1 -- output blocks of B x B points, B = N - 2k,
 *   N the smallest power of sqrt_m >= 3k (tcu_stencil_tiles): the (B + 2k) x
 *   (B + 2k) input
 *   window of every block (Lemma 1's 3k x 3k tile A'_{r,c} when B = k),
 *   zero-padded to N x N, convolved with the flipped, padded W as ONE batch,
 *   the B x B centres written to A_k (device, side^2 fp32; A_k == A
 *   allowed).  The result is the same for every B <= N - 2k; the largest
 *   makes the fewest tiles.
 * Needs N, Nw within one warpgroup pass (k <= 85 for sqrt_m 16, 170 for 8,
 * 341 for 32); else ERR_UNSUPPORTED.  Any side >= 1 (the last blocks of a
 * row or column are cut).  The plan allocates ceil(side/B)^2 N^2 complex64
 * of tiles plus tables; the calls are asynchronous on `stream` and allocate
 * nothing.  w3x3 is a host array. */
typedef struct tcu_stencil_plan_s *tcu_stencil_plan_t;
tcu_stencil_plan_t tcu_stencil_plan(int64_t side, int32_t steps, int32_t sqrt_m,
                                    int32_t precision);
int tcu_stencil_weights(tcu_stencil_plan_t p, const float *w3x3, float *W, void *stream);
int tcu_stencil_exec(tcu_stencil_plan_t p, const float *w3x3, const float *A, float *Ak,
                     void *stream);
int tcu_stencil_check(tcu_stencil_plan_t p, void *stream);
/* The tiling tcu_stencil_plan would choose, without a plan or a GPU: the
 * number of tiles ceil(side / B)^2 (0 if the arguments are unsupported), the
 * tile side N (the smallest power of sqrt_m with N >= 3k and N^2 >=
 * 128 sqrt_m, one warpgroup pass per axis) and the output block side
 * B = N - 2k, written to *tile and *block (either may be NULL). */
int64_t tcu_stencil_tiles(int64_t side, int32_t steps, int32_t sqrt_m, int64_t *tile,
                          int64_t *block);
int tcu_stencil_destroy(tcu_stencil_plan_t p);

/* Failure-detection self-test (not a transform): runs a fused plan's
 * schedule with its work queue started past work that then never runs, so
 * that the dependency waits of the items it claims cannot be satisfied.
 * Every such wait gives up after its limit (2 s of the global timer); the
 * kernel records TCU_DFT_ERR_TIMEOUT in the plan's error word, waits
 * (bounded) for its own copies in flight, frees its tensor memory and
 * returns, leaving the context usable: tcu_dft_check then reports
 * TCU_DFT_ERR_TIMEOUT and clears the word, and the plan transforms normally
 * afterwards.  No fault, trap or unbounded wait is involved.  `out` receives
 * partial data.  Needs a fused plan (TCU_DFT_PLAN_FUSE) with at least
 * lag + 2 chunks of transforms (batch >= 48 for n = 16^4); ERR_INVALID
 * otherwise.  Asynchronous on `stream`. */
int tcu_dft_exec_stalled(tcu_dft_plan_t p, const void *in, void *out, void *stream);

/* Status of the last plan call (tcu_dft_plan*, tcu_dft2_plan,
 * tcu_stencil_plan) on this thread. */
int tcu_dft_last_error(void);

/* Static, human-readable name of a status code. */
const char *tcu_dft_strerror(int status);

#ifdef __cplusplus
}
#endif
#endif /* TCU_DFT_H */
