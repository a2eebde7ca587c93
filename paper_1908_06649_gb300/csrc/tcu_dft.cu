// tcu_dft.cu -- batched complex DFT on GB300 (sm_103a) tensor cores.
//
// The method (arXiv 1908.06649, Sec. 4.5, Theorem 7): with r = sqrt(m) and
// n = r^k, the Cooley-Tukey recursion arranges x as an r x (n/r) row-major
// matrix, replaces every column by its length-r DFT with ONE tall-left tensor
// product X^T * W_r, multiplies entry (k1, c) by the twiddle w_n^{k1 c},
// transposes, and recurses on the rows; the result is read out column-major
// (digit-reversed).  Here every stage is exactly that product: the rows of the
// (batch * n / r) x r data matrix times F_r, on tcgen05 tensor cores.
//
// Complex arithmetic (Sec. 4.5: a complex product is four real products and
// two sums) is one real GEMM on interleaved (re, im) data: a data row
// [a0, b0, a1, b1, ...] times the real 2r x 2r block operand
//     Bf[2j][2c] = Re w,  Bf[2j][2c+1] = Im w,
//     Bf[2j+1][2c] = -Im w, Bf[2j+1][2c+1] = Re w,   w = w_r^{jc},
// gives [Re y0, Im y0, Re y1, ...].
//
// Precision: kind::tf32.  TF32 mode rounds both operands to TF32 (rna).  3xTF32
// mode splits each fp32 value v = hi + lo with hi = rna_tf32(v), lo =
// rna_tf32(v - hi) and accumulates lo*Bhi + hi*Blo + hi*Bhi in fp32 (TMEM).
//
// Kernel structure (one launch per HBM pass; a pass holds s <= 4 stages):
//   load    : the tile's G sub-transforms of length L = r^s, HBM -> SMEM
//             (coalesced; the order follows whichever of the two strides is 1)
//   stage t : rows of the current digit, SMEM -> registers -> hi/lo split ->
//             tcgen05.st into TMEM (the A operand lives in tensor memory);
//             one thread issues tcgen05.mma (A: TMEM, B: F_r image in SMEM,
//             D: TMEM); epilogue tcgen05.ld, twiddle w_L^{k_t c_t}, write back
//             to SMEM in place (in-place decimation in frequency).
//   store   : natural-order output (digit reversal on the SMEM read), optional
//             inter-pass twiddle w_n^{b k} and 1/n scale, coalesced to HBM.
// SMEM addresses are XOR-swizzled (low digit ^= next digit) so that the
// strided row reads of every stage are bank-conflict free.
//
// Every device wait (mbarrier) is bounded: on expiry the kernel records
// TCU_DFT_ERR_TIMEOUT in the plan's error word, skips the rest of its work,
// frees its tensor memory and returns.

#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cmath>
#include <vector>

#include "../../include/tcu_dft.h"

#if defined(__CUDA_ARCH__) && (__CUDA_ARCH__ < 1000)
#error "tcu_dft targets sm_103a (tcgen05); compile with -gencode arch=compute_103a,code=sm_103a"
#endif

namespace {

constexpr int kThreads = 128;               // 4 warps: one per TMEM lane quarter
constexpr unsigned long long kWaitNs = 2000000000ull;  // 2 s bound per wait

// ------------------------------------------------------------------ PTX glue
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ float tf32_rna(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return __uint_as_float(r);
}

__device__ __forceinline__ void mbar_init(uint32_t addr, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(addr), "r"(count)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.b32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(addr), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: true on success, false if the limit expired.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t addr, uint32_t parity) {
  if (mbar_try_wait(addr, parity)) return true;
  const unsigned long long t0 = global_ns();
  while (true) {
    if (mbar_try_wait(addr, parity)) return true;
    if (global_ns() - t0 > kWaitNs) return false;
  }
}

__device__ __forceinline__ void fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t slot_addr, uint32_t ncols) {
  asm volatile(
      "tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
          slot_addr),
      "r"(ncols)
      : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::
                   : "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr),
               "r"(ncols)
               : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem desc], kind::tf32, cta_group::1
__device__ __forceinline__ void mma_tf32_ts(uint32_t d, uint32_t a, uint64_t bdesc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
      "r"(a), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t mbar_addr) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 "
      "[%0];" ::"r"(mbar_addr)
      : "memory");
}

// 32 lanes x 16 consecutive 32-bit columns, one lane per thread.  The wait
// is inside the same asm statement so that no use of the destination
// registers can be scheduled before the load has completed.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float *v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, "
      "[%16];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
        "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
        "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float *v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::
          "r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])),
      "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
      "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
      "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])),
      "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])),
      "r"(__float_as_uint(v[14])), "r"(__float_as_uint(v[15]))
      : "memory");
}

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor, no swizzle, K-major canonical layout:
// core matrices of 8 rows x 16 bytes; LBO = byte step between core matrices
// along K, SBO = byte step between 8-row groups along M/N.
__device__ __forceinline__ uint64_t smem_desc_noswz(uint32_t addr, uint32_t lbo,
                                                    uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version for tcgen05
  return d;                // base offset 0, swizzle mode 0 (none)
}

// Instruction descriptor for kind::tf32: D fp32, A/B tf32, both K-major.
__host__ __device__ constexpr uint32_t idesc_tf32(int M, int N) {
  return (1u << 4)                 // D format: F32
         | (2u << 7)               // A format: TF32
         | (2u << 10)              // B format: TF32
         | ((uint32_t)(N >> 3) << 17)
         | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ float2 cmul(float2 a, float2 b) {
  return make_float2(fmaf(a.x, b.x, -a.y * b.y), fmaf(a.x, b.y, a.y * b.x));
}

// ------------------------------------------------------------ pass kernel
struct PassArgs {
  const float2 *in;
  float2 *out;
  const float *bimg;   // B images for this direction: hi then lo (16 r^2 B each)
  const float2 *twL;   // w_L^e, e in [0, L)
  const float2 *twA;   // inter-pass twiddle, high part: w_N^{i 2^h}
  const float2 *twB;   // inter-pass twiddle, low part:  w_N^{j}
  int *err;
  long long U;         // sub-transforms in the pass
  long long Uper;      // sub-transforms per transform
  long long n;         // transform length
  long long in_vstride, in_stride, out_vstride, out_stride;
  int s;               // stages in this pass
  int log2L;           // log2(r^s)
  int log2G;           // log2(sub-transforms per tile)
  int tw_log2N;        // inter-pass twiddle period log2 (0: none)
  int tw_h;            // low-part bits of the two-level twiddle
  float scale;         // output scale (1 or 1/n)
};

template <int R>
struct Cfg {
  static constexpr int LOG2R = (R == 8) ? 3 : (R == 16) ? 4 : 5;
  static constexpr int TILE_PTS = (R == 8) ? 4096 : 8192;   // points per tile
  static constexpr int ROWS = TILE_PTS / R;                 // data rows per tile
  static constexpr int NGROUPS = ROWS / 128;                // M=128 groups
  static constexpr int Q = (2 * R > 32) ? 2 * R : 32;       // TMEM cols per region
  static constexpr int GCOLS = 3 * Q;                       // A_hi | A_lo | D
  static constexpr int TMEM_COLS = 512;
  static constexpr int IMG_BYTES = 16 * R * R;              // one B image
  static constexpr int LBO = 128;                           // K-adjacent core mats
  static constexpr int SBO = 64 * R;                        // 8-row groups
  static constexpr int KSTEPS = 2 * R / 8;                  // K=8 per tf32 MMA
  static constexpr size_t SMEM_BYTES =
      2 * IMG_BYTES + (size_t)TILE_PTS * 8 + 64;
  static_assert(NGROUPS * GCOLS <= TMEM_COLS, "TMEM budget");
};

template <int R>
__device__ __forceinline__ int swz(int p) {
  return p ^ ((p >> Cfg<R>::LOG2R) & (R - 1));
}

template <int R, int PREC>
__global__ void __launch_bounds__(kThreads, 1) dft_pass_kernel(const PassArgs a) {
  using C = Cfg<R>;
  constexpr int LOG2R = C::LOG2R;
  extern __shared__ __align__(1024) unsigned char smem[];
  float *img = reinterpret_cast<float *>(smem);                 // hi | lo
  float2 *S = reinterpret_cast<float2 *>(smem + 2 * C::IMG_BYTES);
  uint64_t *mbar = reinterpret_cast<uint64_t *>(smem + 2 * C::IMG_BYTES +
                                                (size_t)C::TILE_PTS * 8);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mbar + 1);

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int L = 1 << a.log2L;
  const int G = 1 << a.log2G;
  const long long tile = blockIdx.x;
  const long long u0 = tile << a.log2G;
  const long long rem = a.U - u0;
  const int Gt = rem < G ? (int)rem : G;

  // ---- set-up: B images to SMEM, mbarrier, TMEM
  {
    const float4 *src = reinterpret_cast<const float4 *>(a.bimg);
    float4 *dst = reinterpret_cast<float4 *>(img);
    const int n4 = (PREC == 3 ? 2 : 1) * C::IMG_BYTES / 16;
    for (int i = tid; i < n4; i += kThreads) dst[i] = __ldg(src + i);
  }
  if (tid == 0) {
    mbar_init(smem_u32(mbar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (warp == 0) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);

  // ---- load the tile (zero-fill beyond the last sub-transform)
  const int total = G << a.log2L;
  for (int idx = tid; idx < total; idx += kThreads) {
    int ul, e;
    if (a.in_stride == 1) {
      ul = idx >> a.log2L;
      e = idx & (L - 1);
    } else {
      e = idx >> a.log2G;
      ul = idx & (G - 1);
    }
    float2 v = make_float2(0.f, 0.f);
    if (ul < Gt) {
      const long long u = u0 + ul;
      const long long beta = u / a.Uper;
      const long long vv = u - beta * a.Uper;
      v = __ldg(a.in + beta * a.n + vv * a.in_vstride + (long long)e * a.in_stride);
    }
    S[swz<R>((ul << a.log2L) + e)] = v;
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tbase = *tmem_slot;
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  const int log2rows = a.log2L - LOG2R;  // log2(rows per sub-transform)
  bool failed = false;

  for (int t = 1; t <= a.s && !failed; ++t) {
    const int shift_lo = LOG2R * (a.s - t);
    // ---- build the rows of stage t and move them into TMEM (A operand)
#pragma unroll 1
    for (int g = 0; g < C::NGROUPS; ++g) {
      const int rho = g * 128 + warp * 32 + lane;
      const int ul = rho >> log2rows;
      const int q = rho & ((1 << log2rows) - 1);
      const int hi = q >> shift_lo;
      const int lo = q & ((1 << shift_lo) - 1);
      const int base = (ul << a.log2L) + (hi << (shift_lo + LOG2R)) + lo;
      float vh[2 * R], vl[2 * R];
#pragma unroll
      for (int j = 0; j < R; ++j) {
        const float2 v = S[swz<R>(base + (j << shift_lo))];
        const float hx = tf32_rna(v.x), hy = tf32_rna(v.y);
        vh[2 * j] = hx;
        vh[2 * j + 1] = hy;
        vl[2 * j] = tf32_rna(v.x - hx);
        vl[2 * j + 1] = tf32_rna(v.y - hy);
      }
      const uint32_t col = tbase + lane_base + g * C::GCOLS;
#pragma unroll
      for (int c = 0; c < 2 * R; c += 16) tmem_st16(col + c, vh + c);
      if (PREC == 3) {
#pragma unroll
        for (int c = 0; c < 2 * R; c += 16) tmem_st16(col + C::Q + c, vl + c);
      }
    }
    tmem_wait_st();
    fence_before_sync();
    __syncthreads();

    // ---- one thread issues the stage GEMMs: D = A * Bf  (tall-left x F_r)
    if (tid == 0) {
      fence_after_sync();
      constexpr uint32_t idesc = idesc_tf32(128, 2 * R);
      const uint32_t ihi = smem_u32(img);
      const uint32_t ilo = ihi + C::IMG_BYTES;
#pragma unroll 1
      for (int g = 0; g < C::NGROUPS; ++g) {
        const uint32_t ahi = tbase + g * C::GCOLS;
        const uint32_t alo = ahi + C::Q;
        const uint32_t d = ahi + 2 * C::Q;
        uint32_t acc = 0;
        if (PREC == 3) {
#pragma unroll
          for (int kk = 0; kk < C::KSTEPS; ++kk) {
            mma_tf32_ts(d, alo + 8 * kk,
                        smem_desc_noswz(ihi + kk * 2 * C::LBO, C::LBO, C::SBO),
                        idesc, acc);
            acc = 1;
          }
#pragma unroll
          for (int kk = 0; kk < C::KSTEPS; ++kk)
            mma_tf32_ts(d, ahi + 8 * kk,
                        smem_desc_noswz(ilo + kk * 2 * C::LBO, C::LBO, C::SBO),
                        idesc, 1);
        }
#pragma unroll
        for (int kk = 0; kk < C::KSTEPS; ++kk) {
          mma_tf32_ts(d, ahi + 8 * kk,
                      smem_desc_noswz(ihi + kk * 2 * C::LBO, C::LBO, C::SBO),
                      idesc, acc);
          acc = 1;
        }
      }
      mma_commit(smem_u32(mbar));
    }
    const bool ok = mbar_wait_bounded(smem_u32(mbar), (uint32_t)((t - 1) & 1));
    failed = __syncthreads_or(!ok) != 0;
    if (failed) break;
    fence_after_sync();

    // ---- epilogue: TMEM -> registers, twiddle, in-place write to SMEM
#pragma unroll 1
    for (int g = 0; g < C::NGROUPS; ++g) {
      const int rho = g * 128 + warp * 32 + lane;
      const int ul = rho >> log2rows;
      const int q = rho & ((1 << log2rows) - 1);
      const int hi = q >> shift_lo;
      const int lo = q & ((1 << shift_lo) - 1);
      const int base = (ul << a.log2L) + (hi << (shift_lo + LOG2R)) + lo;
      float d[2 * R];
      const uint32_t col = tbase + lane_base + g * C::GCOLS + 2 * C::Q;
#pragma unroll
      for (int c = 0; c < 2 * R; c += 16) tmem_ld16(col + c, d + c);
      tmem_wait_ld();
      // twiddle w_{L_t}^{k_t c_t} = w_L^{k_t * lo * r^(t-1)}
      const int estep = lo << (LOG2R * (t - 1));
#pragma unroll
      for (int j = 0; j < R; ++j) {
        float2 y = make_float2(d[2 * j], d[2 * j + 1]);
        if (t < a.s) y = cmul(y, __ldg(a.twL + ((j * estep) & (L - 1))));
        S[swz<R>(base + (j << shift_lo))] = y;
      }
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
  }

  // ---- store: natural order, inter-pass twiddle, scale
  if (!failed) {
    const long long Nmask = (1ll << a.tw_log2N) - 1;
    const long long hmask = (1ll << a.tw_h) - 1;
    for (int idx = tid; idx < total; idx += kThreads) {
      int ul, k;
      if (a.out_stride == 1) {
        ul = idx >> a.log2L;
        k = idx & (L - 1);
      } else {
        k = idx >> a.log2G;
        ul = idx & (G - 1);
      }
      if (ul >= Gt) continue;
      int rev = 0, kk = k;
      for (int t = 0; t < a.s; ++t) {
        rev = (rev << LOG2R) | (kk & (R - 1));
        kk >>= LOG2R;
      }
      float2 v = S[swz<R>((ul << a.log2L) + rev)];
      const long long u = u0 + ul;
      const long long beta = u / a.Uper;
      const long long vv = u - beta * a.Uper;
      if (a.tw_log2N) {
        const long long e = (vv * (long long)k) & Nmask;
        const float2 w = cmul(__ldg(a.twA + (e >> a.tw_h)), __ldg(a.twB + (e & hmask)));
        v = cmul(v, w);
      }
      v.x *= a.scale;
      v.y *= a.scale;
      a.out[beta * a.n + vv * a.out_vstride + (long long)k * a.out_stride] = v;
    }
  } else if (tid == 0) {
    atomicExch(a.err, TCU_DFT_ERR_TIMEOUT);
  }

  // ---- teardown
  fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    fence_after_sync();
    tmem_dealloc(tbase, C::TMEM_COLS);
  }
}

// ------------------------------------------------------------ group kernel
// Persistent kernel for passes of L = r^S <= 128 r points per sub-transform.
// A CTA holds NWG independent warpgroups.  A warpgroup owns one TMEM slot
// (A_hi | A_lo | D for 128 rows), one SMEM transpose buffer and one mbarrier,
// and walks a strided list of work items; an item is GG = 128 r / L
// consecutive sub-transforms, i.e. exactly 128 data rows per stage, so every
// stage of an item is one M=128 tcgen05 product and the transposes between
// stages stay inside the warpgroup.  Stage-1 rows are loaded from global
// memory straight into registers (the row-to-lane map makes the loads
// coalesced), the next item's rows are prefetched while the current item's
// products run, and the last stage's rows are stored straight from registers.

enum RowMode { kQF = 0, kUF = 1, kRQF = 2 };

struct GroupArgs {
  const float2 *in;
  float2 *out;
  const float *bimg;   // hi | lo B images of F_r for this direction
  const float2 *twL;   // w_L^e, e in [0, L)
  const float2 *twA;   // inter-pass twiddle, high part: w_N^{i 2^h}
  const float2 *twB;   // inter-pass twiddle, low part:  w_N^{j}
  int *err;
  long long U;         // sub-transforms in the pass
  long long n;         // transform length
  long long in_vstride, in_stride, out_vstride, out_stride;
  int log2Uper;        // log2(sub-transforms per transform)
  int tw_log2N;        // inter-pass twiddle period log2 (0: none)
  int tw_h;            // low-part bits of the two-level twiddle
  int mode_first, mode_mid, mode_last;  // RowMode of the first/middle/last stage
  unsigned long long swz_tab;           // 16 nibbles: SMEM swizzle per (ul & 15)
  float scale;         // output scale (1 or 1/n)
};

template <int R, int S>
struct GCfg {
  static constexpr int LOG2R = (R == 8) ? 3 : (R == 16) ? 4 : 5;
  static constexpr int NWG = (R == 32) ? 2 : 4;
  static constexpr int THREADS = 128 * NWG;
  static constexpr int GPTS = 128 * R;               // points per item
  static constexpr int LOG2GPTS = 7 + LOG2R;
  static constexpr int LOG2L = LOG2R * S;
  static constexpr int L = 1 << LOG2L;
  static constexpr int LOG2RPS = LOG2L - LOG2R;      // rows per sub-transform
  static constexpr int LOG2GG = LOG2GPTS - LOG2L;    // sub-transforms per item
  static constexpr int GG = 1 << LOG2GG;
  static constexpr int Q = (2 * R > 32) ? 2 * R : 32;
  static constexpr int GCOLS = 3 * Q;
  static constexpr int IMG_BYTES = 16 * R * R;
  static constexpr int LBO = 128, SBO = 64 * R, KSTEPS = 2 * R / 8;
  static constexpr size_t OFF_TW = 2 * IMG_BYTES;
  static constexpr size_t OFF_BUF = OFF_TW + (size_t)L * 8;
  static constexpr size_t OFF_BAR =
      OFF_BUF + (S > 1 ? (size_t)NWG * GPTS * 8 : 0);
  static constexpr size_t SMEM_BYTES = OFF_BAR + 8 * NWG + 16;
  static_assert(LOG2GG >= 0, "sub-transform longer than one item");
  static_assert(NWG * GCOLS <= 512, "TMEM budget");
};

// bar.sync on a named barrier that also ORs a predicate across the threads
__device__ __forceinline__ bool named_bar_or(int id, int count, bool v) {
  uint32_t out;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.or.pred p, %2, %3, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(out)
      : "r"((uint32_t)v), "r"(id), "r"(count)
      : "memory");
  return out != 0;
}

template <int R, int S>
__device__ __forceinline__ void row_of(int mode, int rho, int &ul, int &q) {
  using C = GCfg<R, S>;
  if (mode == kUF) {
    ul = rho & (C::GG - 1);
    q = rho >> C::LOG2GG;
  } else {
    ul = rho >> C::LOG2RPS;
    q = rho & ((1 << C::LOG2RPS) - 1);
    if (mode == kRQF) {  // digit-reversed q over S-1 digits
      int rq = 0, v = q;
#pragma unroll
      for (int i = 0; i < S - 1; ++i) {
        rq = (rq << C::LOG2R) | (v & (R - 1));
        v >>= C::LOG2R;
      }
      q = rq;
    }
  }
}

__device__ __forceinline__ int gswz(int p, uint32_t tabv) {
  return p ^ (int)((tabv ^ (uint32_t)(p >> 4)) & 15u);
}

// Split a complex row into TF32 hi / lo parts and store them as the A
// operand rows of this thread's TMEM lane.
template <int R, int PREC>
__device__ __forceinline__ void split_store(const float2 *x, uint32_t col_hi,
                                            uint32_t col_lo) {
#pragma unroll
  for (int c = 0; c < R; c += 8) {
    float vh[16], vl[16];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float hx = tf32_rna(x[c + j].x), hy = tf32_rna(x[c + j].y);
      vh[2 * j] = hx;
      vh[2 * j + 1] = hy;
      if (PREC == 3) {
        vl[2 * j] = tf32_rna(x[c + j].x - hx);
        vl[2 * j + 1] = tf32_rna(x[c + j].y - hy);
      }
    }
    tmem_st16(col_hi + 2 * c, vh);
    if (PREC == 3) tmem_st16(col_lo + 2 * c, vl);
  }
}

template <int R, int PREC>
__device__ __forceinline__ void issue_stage_mma(uint32_t slot, uint32_t img_addr) {
  constexpr int Q = (2 * R > 32) ? 2 * R : 32;
  constexpr int IMG = 16 * R * R, LBO = 128, SBO = 64 * R, KSTEPS = 2 * R / 8;
  constexpr uint32_t idesc = idesc_tf32(128, 2 * R);
  const uint32_t ahi = slot, alo = slot + Q, d = slot + 2 * Q;
  const uint32_t ihi = img_addr, ilo = img_addr + IMG;
  uint32_t acc = 0;
  if (PREC == 3) {
#pragma unroll
    for (int kk = 0; kk < KSTEPS; ++kk) {
      mma_tf32_ts(d, alo + 8 * kk, smem_desc_noswz(ihi + kk * 2 * LBO, LBO, SBO),
                  idesc, acc);
      acc = 1;
    }
#pragma unroll
    for (int kk = 0; kk < KSTEPS; ++kk)
      mma_tf32_ts(d, ahi + 8 * kk, smem_desc_noswz(ilo + kk * 2 * LBO, LBO, SBO),
                  idesc, 1);
  }
#pragma unroll
  for (int kk = 0; kk < KSTEPS; ++kk) {
    mma_tf32_ts(d, ahi + 8 * kk, smem_desc_noswz(ihi + kk * 2 * LBO, LBO, SBO),
                idesc, acc);
    acc = 1;
  }
}

template <int R, int S>
__device__ __forceinline__ void load_row(const GroupArgs &a, long long item,
                                         long long nitems, int ul, int q,
                                         float2 *x) {
  using C = GCfg<R, S>;
  const long long u = (item << C::LOG2GG) + ul;
  if (item < nitems && u < a.U) {
    const long long beta = u >> a.log2Uper;
    const long long vv = u & ((1ll << a.log2Uper) - 1);
    const float2 *src = a.in + beta * a.n + vv * a.in_vstride + (long long)q * a.in_stride;
    const long long js = a.in_stride << (C::LOG2R * (S - 1));
#pragma unroll
    for (int j = 0; j < R; ++j) x[j] = __ldg(src + j * js);
  } else {
#pragma unroll
    for (int j = 0; j < R; ++j) x[j] = make_float2(0.f, 0.f);
  }
}

template <int R, int PREC, int S>
__global__ void __launch_bounds__(GCfg<R, S>::THREADS, 1)
    dft_group_kernel(const GroupArgs a) {
  using C = GCfg<R, S>;
  constexpr int LOG2R = C::LOG2R;
  extern __shared__ __align__(1024) unsigned char smem[];
  float *img = reinterpret_cast<float *>(smem);
  float2 *tw = reinterpret_cast<float2 *>(smem + C::OFF_TW);
  uint64_t *mbar = reinterpret_cast<uint64_t *>(smem + C::OFF_BAR);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mbar + C::NWG);

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int wg = warp >> 2, wq = warp & 3;
  const int rho = wq * 32 + lane;
  float2 *buf = reinterpret_cast<float2 *>(smem + C::OFF_BUF) + wg * C::GPTS;

  // ---- set-up
  {
    const float4 *src = reinterpret_cast<const float4 *>(a.bimg);
    float4 *dst = reinterpret_cast<float4 *>(img);
    const int n4 = (PREC == 3 ? 2 : 1) * C::IMG_BYTES / 16;
    for (int i = tid; i < n4; i += C::THREADS) dst[i] = __ldg(src + i);
    if (S > 1)
      for (int i = tid; i < C::L; i += C::THREADS) tw[i] = __ldg(a.twL + i);
  }
  if (tid == 0) {
    for (int w = 0; w < C::NWG; ++w) mbar_init(smem_u32(mbar + w), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (warp == 0) tmem_alloc(smem_u32(tmem_slot), 512);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tbase = *tmem_slot;
  const uint32_t slot = tbase + wg * C::GCOLS;
  const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
  const uint32_t img_addr = smem_u32(img);
  const uint32_t bar_addr = smem_u32(mbar + wg);
  const int bar_id = 1 + wg;

  const long long nitems = (a.U + C::GG - 1) >> C::LOG2GG;
  const long long istride = (long long)gridDim.x * C::NWG;
  long long item = (long long)blockIdx.x * C::NWG + wg;
  uint32_t phase = 0;
  bool fail = false;

  int ul1, q1;
  row_of<R, S>(a.mode_first, rho, ul1, q1);
  float2 x[R];
  load_row<R, S>(a, item, nitems, ul1, q1, x);

  while (item < nitems) {
    // ---- stage 1 operand
    split_store<R, PREC>(x, slot + lane_off, slot + C::Q + lane_off);
    tmem_wait_st();
    fence_before_sync();
    if (named_bar_or(bar_id, 128, fail)) break;
    if (rho == 0) {
      fence_after_sync();
      issue_stage_mma<R, PREC>(slot, img_addr);
      mma_commit(bar_addr);
    }
    const long long next = item + istride;
    load_row<R, S>(a, next, nitems, ul1, q1, x);  // prefetch
    if (!mbar_wait_bounded(bar_addr, phase)) fail = true;
    phase ^= 1;
    fence_after_sync();

#pragma unroll 1
    for (int t = 1; t <= S; ++t) {
      if (t < S) {
        // epilogue of stage t, 8 outputs at a time: TMEM -> registers,
        // twiddle w_{L_t}^{k_t c_t} = w_L^{k_t * lo * r^(t-1)}, transposed
        // write to the SMEM buffer
        const int mode = (t == 1) ? a.mode_first : a.mode_mid;
        int ul, q;
        row_of<R, S>(mode, rho, ul, q);
        const int shift_lo = LOG2R * (S - t);
        const int hi = q >> shift_lo, lo = q & ((1 << shift_lo) - 1);
        const int base = (ul << C::LOG2L) + (hi << (shift_lo + LOG2R)) + lo;
        const uint32_t tabv = (uint32_t)(a.swz_tab >> (4 * (ul & 15))) & 15u;
        const int estep = lo << (LOG2R * (t - 1));
#pragma unroll
        for (int c = 0; c < R; c += 8) {
          float d[16];
          tmem_ld16(slot + 2 * C::Q + lane_off + 2 * c, d);
#pragma unroll
          for (int jj = 0; jj < 8; ++jj) {
            const int j = c + jj;
            const float2 y = cmul(make_float2(d[2 * jj], d[2 * jj + 1]),
                                  tw[(j * estep) & (C::L - 1)]);
            buf[gswz(base + (j << shift_lo), tabv)] = y;
          }
        }
        fence_before_sync();
        named_bar_or(bar_id, 128, false);
        // rows of stage t+1, 8 elements at a time: SMEM -> split -> TMEM
        const int mode2 = (t + 1 == S) ? a.mode_last : a.mode_mid;
        row_of<R, S>(mode2, rho, ul, q);
        const int shift2 = LOG2R * (S - t - 1);
        const int hi2 = q >> shift2, lo2 = q & ((1 << shift2) - 1);
        const int base2 = (ul << C::LOG2L) + (hi2 << (shift2 + LOG2R)) + lo2;
        const uint32_t tabv2 = (uint32_t)(a.swz_tab >> (4 * (ul & 15))) & 15u;
#pragma unroll
        for (int c = 0; c < R; c += 8) {
          float2 row[8];
#pragma unroll
          for (int jj = 0; jj < 8; ++jj)
            row[jj] = buf[gswz(base2 + ((c + jj) << shift2), tabv2)];
          split_store<8, PREC>(row, slot + lane_off + 2 * c, slot + C::Q + lane_off + 2 * c);
        }
        tmem_wait_st();
        fence_before_sync();
        if (named_bar_or(bar_id, 128, fail)) {
          fail = true;
          break;
        }
        if (rho == 0) {
          fence_after_sync();
          issue_stage_mma<R, PREC>(slot, img_addr);
          mma_commit(bar_addr);
        }
        if (!mbar_wait_bounded(bar_addr, phase)) fail = true;
        phase ^= 1;
        fence_after_sync();
      } else {
        // last stage: natural-order output straight from registers
        float d[2 * R];
#pragma unroll
        for (int c = 0; c < 2 * R; c += 16) tmem_ld16(slot + 2 * C::Q + lane_off + c, d + c);
        int ul, q;
        row_of<R, S>(a.mode_last, rho, ul, q);
        const long long u = (item << C::LOG2GG) + ul;
        if (u < a.U) {
          int klow = 0, v = q;
#pragma unroll
          for (int i = 0; i < S - 1; ++i) {
            klow = (klow << LOG2R) | (v & (R - 1));
            v >>= LOG2R;
          }
          const long long beta = u >> a.log2Uper;
          const long long vv = u & ((1ll << a.log2Uper) - 1);
          float2 *dst = a.out + beta * a.n + vv * a.out_vstride + klow * a.out_stride;
          const long long jstep = a.out_stride << (LOG2R * (S - 1));
          // twiddle exponent (vv * k) mod 2^tw_log2N, tw_log2N <= 32: exact in
          // wrap-around 32-bit arithmetic
          const uint32_t Nmask = (uint32_t)((1ull << a.tw_log2N) - 1);
          const uint32_t hmask = (1u << a.tw_h) - 1;
          const uint32_t e0 = (uint32_t)vv * (uint32_t)klow;
          const uint32_t estep = (uint32_t)vv << (LOG2R * (S - 1));
#pragma unroll
          for (int j = 0; j < R; ++j) {
            float2 y = make_float2(d[2 * j], d[2 * j + 1]);
            if (a.tw_log2N) {
              const uint32_t e = (e0 + (uint32_t)j * estep) & Nmask;
              y = cmul(y, cmul(__ldg(a.twA + (e >> a.tw_h)), __ldg(a.twB + (e & hmask))));
            }
            y.x *= a.scale;
            y.y *= a.scale;
            dst[j * jstep] = y;
          }
        }
      }
    }
    // a failed wait is acted on at the next barrier, where the flag is
    // reduced over the warpgroup so that every thread leaves together
    item = next;
  }
  if (fail && rho == 0) atomicExch(a.err, TCU_DFT_ERR_TIMEOUT);

  // ---- teardown
  fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    fence_after_sync();
    tmem_dealloc(tbase, 512);
  }
}

// ------------------------------------------------------------------ host side
enum PassKind { kTilePass = 0, kGroupPass = 1 };

struct PassPlan {
  int kind;        // kTilePass or kGroupPass
  int s;
  int log2L;
  int log2G;       // tile kernel: sub-transforms per tile
  long long U, Uper;
  int log2Uper;
  long long in_vstride, in_stride, out_vstride, out_stride;
  int tw_log2N, tw_h;
  int modes[3];    // group kernel: row map of first / middle / last stage
  unsigned long long swz_tab;
  bool last;
  float2 *twL[2];  // [dir index] w_L^e
};

thread_local int g_last_error = TCU_DFT_OK;

int ilog2(long long v) {
  int l = 0;
  while ((1ll << l) < v) ++l;
  return l;
}

}  // namespace

struct tcu_dft_plan_s {
  long long n, batch;
  int r, log2r, k, precision;
  int npasses;
  int num_sms;
  PassPlan pass[2];
  float *bimg[2];      // [dir index] hi | lo images
  float2 *twA[2], *twB[2];
  float2 *scratch;
  int *err;
  int device;
};

namespace {

int dir_index(int dir) { return dir == TCU_DFT_INVERSE ? 1 : 0; }

// Round an fp32 value to TF32 (10 explicit mantissa bits), nearest, ties away
// from zero -- the same rule as PTX cvt.rna.tf32.f32.
float host_tf32_rna(float x) {
  uint32_t b;
  memcpy(&b, &x, 4);
  if ((b & 0x7F800000u) != 0x7F800000u) b = (b + 0x1000u) & 0xFFFFE000u;
  float r;
  memcpy(&r, &b, 4);
  return r;
}

// B operand images (hi, lo) of the real 2r x 2r block form of F_r for one
// direction, in the canonical no-swizzle K-major layout the MMA reads.
void build_images(int r, int sign, std::vector<float> &out) {
  const int K = 2 * r, N = 2 * r;
  const int lbo = 128, sbo = 64 * r;
  const size_t img_floats = (size_t)16 * r * r / 4;
  out.assign(2 * img_floats, 0.f);
  for (int kr = 0; kr < K; ++kr) {
    for (int nc = 0; nc < N; ++nc) {
      const int j = kr >> 1, a = kr & 1, c = nc >> 1, b = nc & 1;
      const long long m = ((long long)j * c) % r;
      const double ang = (double)sign * 2.0 * M_PI * (double)m / (double)r;
      const double re = cos(ang), im = sin(ang);
      double v;
      if (a == 0)
        v = (b == 0) ? re : im;
      else
        v = (b == 0) ? -im : re;
      const float hi = host_tf32_rna((float)v);
      const float lo = host_tf32_rna((float)(v - (double)hi));
      const size_t off =
          ((size_t)(nc >> 3) * sbo + (size_t)(kr >> 2) * lbo + (nc & 7) * 16 +
           (kr & 3) * 4) / 4;
      out[off] = hi;
      out[img_floats + off] = lo;
    }
  }
}

std::vector<float2> twiddle_table(long long period, long long count, long long step,
                                  int sign) {
  std::vector<float2> t((size_t)count);
  for (long long e = 0; e < count; ++e) {
    const long long m = (e * step) % period;
    const double ang = (double)sign * 2.0 * M_PI * (double)m / (double)period;
    t[(size_t)e] = make_float2((float)cos(ang), (float)sin(ang));
  }
  return t;
}

// Largest stage count per pass: tile kernel (a sub-transform fills at most one
// SMEM tile) and group kernel (a sub-transform fits 128 rows).
int max_tile_stages(int r) { return r == 8 ? 4 : (r == 16 ? 3 : 2); }
int max_group_stages(int r) { return r == 8 ? 3 : 2; }

int stage_mode(const int modes[3], int t, int S) {
  return t == 1 ? modes[0] : (t == S ? modes[2] : modes[1]);
}

// Shared-memory wavefronts per warp-wide 8-byte access of the group kernel's
// transposes (1.0 = conflict free), for swizzle table `tab`:
// phys(P) = P ^ ((tab[ul & 15] ^ (P >> 4)) & 15).
double swizzle_cost(int r, int S, const int modes[3], unsigned long long tab) {
  const int log2r = ilog2(r);
  const int L = 1 << (log2r * S);
  const int rps = L / r, gg = 128 * r / L;
  long long waves = 0, accesses = 0;
  for (int t = 1; t < S; ++t) {
    for (int side = 0; side < 2; ++side) {  // epilogue write of t, read of t+1
      const int tt = t + side;
      const int mode = stage_mode(modes, tt, S);
      const int sl = log2r * (S - tt);
      for (int w = 0; w < 4; ++w)
        for (int j = 0; j < r; ++j)
          for (int h = 0; h < 2; ++h) {
            int seen = 0;  // bitmask of the 16 eight-byte bank slots
            int count = 0;
            for (int l = 16 * h; l < 16 * h + 16; ++l) {
              const int rho = 32 * w + l;
              int ul, q;
              if (mode == kUF) {
                ul = rho % gg;
                q = rho / gg;
              } else {
                ul = rho / rps;
                q = rho % rps;
                if (mode == kRQF) {
                  int rq = 0, v = q;
                  for (int i = 0; i < S - 1; ++i) {
                    rq = rq * r + v % r;
                    v /= r;
                  }
                  q = rq;
                }
              }
              const int hi = q >> sl, lo = q & ((1 << sl) - 1);
              const int P = ul * L + (hi << (sl + log2r)) + (j << sl) + lo;
              const unsigned tv = (unsigned)(tab >> (4 * (ul & 15))) & 15u;
              const int ph = P ^ (int)((tv ^ (unsigned)(P >> 4)) & 15u);
              const int slot = ph & 15;
              if (!(seen & (1 << slot))) {
                seen |= 1 << slot;
                ++count;
              }
            }
            waves += (16 + count - 1) / count;
            ++accesses;
          }
    }
  }
  return accesses ? (double)waves / (double)accesses : 1.0;
}

unsigned long long choose_swizzle(int r, int S, const int modes[3]) {
  std::vector<unsigned long long> cands;
  for (int c = 0; c < 4; ++c) {
    unsigned long long t = 0;
    for (int u = 0; u < 16; ++u) t |= (unsigned long long)((u << c) & 15) << (4 * u);
    cands.push_back(t);
  }
  for (int c = 1; c < 4; ++c) {
    unsigned long long t = 0;
    for (int u = 0; u < 16; ++u) t |= (unsigned long long)((u ^ (u << c)) & 15) << (4 * u);
    cands.push_back(t);
  }
  cands.push_back(0ull);
  cands.push_back(0x7fe70d6c0000a378ull);  // found by an offline search
  unsigned long long best = cands[0];
  double bc = 1e30;
  for (unsigned long long t : cands) {
    const double c = swizzle_cost(r, S, modes, t);
    if (c < bc - 1e-9) {
      bc = c;
      best = t;
    }
  }
  return best;
}

template <typename T>
int upload(T **dst, const std::vector<T> &src) {
  if (cudaMalloc((void **)dst, src.size() * sizeof(T)) != cudaSuccess) {
    cudaGetLastError();
    *dst = nullptr;
    return TCU_DFT_ERR_OOM;
  }
  if (cudaMemcpy(*dst, src.data(), src.size() * sizeof(T), cudaMemcpyHostToDevice) !=
      cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  return TCU_DFT_OK;
}

void free_plan(tcu_dft_plan_s *p) {
  if (!p) return;
  for (int d = 0; d < 2; ++d) {
    cudaFree(p->bimg[d]);
    cudaFree(p->twA[d]);
    cudaFree(p->twB[d]);
    for (int i = 0; i < p->npasses; ++i) cudaFree(p->pass[i].twL[d]);
  }
  cudaFree(p->scratch);
  cudaFree(p->err);
  delete p;
}

template <int R>
size_t smem_bytes() {
  // one CTA per SM: the kernel allocates all 512 TMEM columns
  size_t b = Cfg<R>::SMEM_BYTES;
  return b < 120 * 1024 ? 120 * 1024 : b;
}

template <int R, int PREC>
cudaError_t launch_pass(const PassArgs &a, long long grid, cudaStream_t st) {
  const size_t sm = smem_bytes<R>();
  cudaError_t e = cudaFuncSetAttribute(dft_pass_kernel<R, PREC>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sm);
  if (e != cudaSuccess) return e;
  dft_pass_kernel<R, PREC><<<(unsigned)grid, kThreads, sm, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_dispatch(int r, int prec, const PassArgs &a, long long grid,
                            cudaStream_t st) {
  if (r == 8) return prec == 3 ? launch_pass<8, 3>(a, grid, st) : launch_pass<8, 1>(a, grid, st);
  if (r == 16)
    return prec == 3 ? launch_pass<16, 3>(a, grid, st) : launch_pass<16, 1>(a, grid, st);
  return prec == 3 ? launch_pass<32, 3>(a, grid, st) : launch_pass<32, 1>(a, grid, st);
}

template <int R, int PREC, int S>
cudaError_t launch_group(const GroupArgs &a, int num_sms, cudaStream_t st) {
  using C = GCfg<R, S>;
  const size_t sm = C::SMEM_BYTES;
  cudaError_t e = cudaFuncSetAttribute(dft_group_kernel<R, PREC, S>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sm);
  if (e != cudaSuccess) return e;
  const long long nitems = (a.U + C::GG - 1) >> C::LOG2GG;
  long long grid = (nitems + C::NWG - 1) / C::NWG;
  if (grid > num_sms) grid = num_sms;
  dft_group_kernel<R, PREC, S><<<(unsigned)grid, C::THREADS, sm, st>>>(a);
  return cudaGetLastError();
}

template <int R, int PREC>
cudaError_t launch_group_s(int s, const GroupArgs &a, int num_sms, cudaStream_t st) {
  if (s == 1) return launch_group<R, PREC, 1>(a, num_sms, st);
  if (s == 2) return launch_group<R, PREC, 2>(a, num_sms, st);
  if constexpr (R == 8) {
    if (s == 3) return launch_group<R, PREC, 3>(a, num_sms, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_group_dispatch(int r, int prec, int s, const GroupArgs &a,
                                  int num_sms, cudaStream_t st) {
  if (r == 8)
    return prec == 3 ? launch_group_s<8, 3>(s, a, num_sms, st)
                     : launch_group_s<8, 1>(s, a, num_sms, st);
  if (r == 16)
    return prec == 3 ? launch_group_s<16, 3>(s, a, num_sms, st)
                     : launch_group_s<16, 1>(s, a, num_sms, st);
  return prec == 3 ? launch_group_s<32, 3>(s, a, num_sms, st)
                   : launch_group_s<32, 1>(s, a, num_sms, st);
}

int tile_points(int r) { return r == 8 ? 4096 : 8192; }

bool overlaps(const void *a, const void *b, size_t bytes) {
  const char *x = (const char *)a, *y = (const char *)b;
  return x < y + bytes && y < x + bytes;
}

}  // namespace

extern "C" {

const char *tcu_dft_strerror(int status) {
  switch (status) {
    case TCU_DFT_OK: return "ok";
    case TCU_DFT_ERR_INVALID: return "invalid argument";
    case TCU_DFT_ERR_UNSUPPORTED: return "unsupported size or radix";
    case TCU_DFT_ERR_CUDA: return "CUDA error";
    case TCU_DFT_ERR_OOM: return "device allocation failed";
    case TCU_DFT_ERR_TIMEOUT: return "device wait timed out";
    default: return "unknown status";
  }
}

int tcu_dft_last_error(void) { return g_last_error; }

tcu_dft_plan_t tcu_dft_plan(int64_t n, int64_t batch, int32_t sqrt_m,
                            int32_t precision) {
  g_last_error = TCU_DFT_OK;
  if (n < 1 || batch < 1 || (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32)) {
    g_last_error = TCU_DFT_ERR_INVALID;
    return nullptr;
  }
  if (sqrt_m != 8 && sqrt_m != 16 && sqrt_m != 32) {
    g_last_error = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  const int r = sqrt_m, log2r = ilog2(r);
  int k = 0;
  long long m = 1;
  while (m < n) {
    m *= r;
    ++k;
  }
  if (m != n || k < 1) {
    g_last_error = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  // Pass grouping: prefer the group kernel (sub-transforms of <= 128 rows),
  // fall back to the tile kernel for longer sub-transforms.
  const int sg = max_group_stages(r), stl = max_tile_stages(r);
  int stages[2] = {0, 0}, kinds[2] = {kGroupPass, kGroupPass}, npasses;
  if (k <= sg) {
    npasses = 1;
    stages[0] = k;
  } else if (k <= 2 * sg) {
    npasses = 2;
    stages[0] = (k + 1) / 2;
    stages[1] = k - stages[0];
  } else if (k <= stl + sg) {
    npasses = 2;
    stages[0] = k - sg;
    kinds[0] = kTilePass;
    stages[1] = sg;
  } else if (k <= 2 * stl) {
    npasses = 2;
    stages[0] = (k + 1) / 2;
    stages[1] = k - stages[0];
    kinds[0] = kinds[1] = kTilePass;
  } else {
    g_last_error = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  if ((long long)batch * n > (1ll << 40)) {
    g_last_error = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  int dev = 0;
  cudaDeviceProp prop;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaGetDeviceProperties(&prop, dev) != cudaSuccess || prop.major != 10 ||
      prop.minor != 3) {
    cudaGetLastError();
    g_last_error = TCU_DFT_ERR_CUDA;
    return nullptr;
  }

  tcu_dft_plan_s *p = new tcu_dft_plan_s();
  memset(p, 0, sizeof(*p));
  p->n = n;
  p->batch = batch;
  p->r = r;
  p->log2r = log2r;
  p->k = k;
  p->precision = precision;
  p->npasses = npasses;
  p->device = dev;
  p->num_sms = prop.multiProcessorCount;
  const int log2n = ilog2(n);
  int rc = TCU_DFT_OK;
  for (int pi = 0; pi < npasses && rc == TCU_DFT_OK; ++pi) {
    PassPlan &pp = p->pass[pi];
    pp.kind = kinds[pi];
    pp.s = stages[pi];
    pp.log2L = log2r * pp.s;
    pp.log2G = ilog2(tile_points(r)) - pp.log2L;
    pp.last = (pi == npasses - 1);
    const long long L = 1ll << pp.log2L;
    if (npasses == 1) {
      pp.U = batch;
      pp.Uper = 1;
      pp.in_vstride = n;
      pp.in_stride = 1;
      pp.out_vstride = n;
      pp.out_stride = 1;
      pp.tw_log2N = 0;
    } else if (pi == 0) {
      const long long n2 = n / L;  // four-step: x[n2 a + b], DFT over a
      pp.U = batch * n2;
      pp.Uper = n2;
      pp.in_vstride = 1;
      pp.in_stride = n2;
      pp.out_vstride = 1;
      pp.out_stride = n2;
      pp.tw_log2N = log2n;       // w_n^{b k1}
      pp.tw_h = (log2n + 1) / 2;
    } else {
      const long long n1 = n / L;  // rows k1 of the four-step, DFT over b
      pp.U = batch * n1;
      pp.Uper = n1;
      pp.in_vstride = L;
      pp.in_stride = 1;
      pp.out_vstride = 1;
      pp.out_stride = n1;
      pp.tw_log2N = 0;
    }
    pp.log2Uper = ilog2(pp.Uper);
    pp.modes[0] = pp.in_stride == 1 ? kQF : kUF;
    pp.modes[1] = kUF;
    pp.modes[2] = pp.out_stride == 1 ? kRQF : kUF;
    pp.swz_tab = choose_swizzle(r, pp.s, pp.modes);
    for (int d = 0; d < 2 && rc == TCU_DFT_OK; ++d) {
      const int sign = d == 0 ? -1 : 1;
      rc = upload(&pp.twL[d], twiddle_table(L, L, 1, sign));
    }
  }
  for (int d = 0; d < 2 && rc == TCU_DFT_OK; ++d) {
    const int sign = d == 0 ? -1 : 1;
    std::vector<float> img;
    build_images(r, sign, img);
    rc = upload(&p->bimg[d], img);
    if (rc == TCU_DFT_OK && npasses == 2) {
      const int h = p->pass[0].tw_h;
      rc = upload(&p->twA[d], twiddle_table(n, n >> h, 1ll << h, sign));
      if (rc == TCU_DFT_OK) rc = upload(&p->twB[d], twiddle_table(n, 1ll << h, 1, sign));
    }
  }
  if (rc == TCU_DFT_OK) {
    if (cudaMalloc((void **)&p->err, sizeof(int)) != cudaSuccess ||
        cudaMemset(p->err, 0, sizeof(int)) != cudaSuccess) {
      cudaGetLastError();
      rc = TCU_DFT_ERR_OOM;
    }
  }
  if (rc == TCU_DFT_OK && npasses == 2) {
    if (cudaMalloc((void **)&p->scratch, (size_t)batch * n * sizeof(float2)) !=
        cudaSuccess) {
      cudaGetLastError();
      rc = TCU_DFT_ERR_OOM;
    }
  }
  if (rc != TCU_DFT_OK) {
    free_plan(p);
    g_last_error = rc;
    return nullptr;
  }
  return p;
}

static int exec_impl(tcu_dft_plan_t p, const void *in, void *out, int dir,
                     void *stream, void *const *events) {
  if (!p || !in || !out || (dir != TCU_DFT_FORWARD && dir != TCU_DFT_INVERSE))
    return TCU_DFT_ERR_INVALID;
  if (((uintptr_t)in & 15) || ((uintptr_t)out & 15)) return TCU_DFT_ERR_INVALID;
  const size_t bytes = (size_t)p->batch * p->n * sizeof(float2);
  if (in != out && overlaps(in, out, bytes)) return TCU_DFT_ERR_INVALID;
  cudaStream_t st = (cudaStream_t)stream;
  const int di = dir_index(dir);
  for (int pi = 0; pi < p->npasses; ++pi) {
    const PassPlan &pp = p->pass[pi];
    if (pp.kind == kGroupPass) {
      GroupArgs g;
      memset(&g, 0, sizeof(g));
      g.in = (pi == 0) ? (const float2 *)in : p->scratch;
      g.out = pp.last ? (float2 *)out : p->scratch;
      g.bimg = p->bimg[di];
      g.twL = pp.twL[di];
      g.twA = p->twA[di];
      g.twB = p->twB[di];
      g.err = p->err;
      g.U = pp.U;
      g.n = p->n;
      g.in_vstride = pp.in_vstride;
      g.in_stride = pp.in_stride;
      g.out_vstride = pp.out_vstride;
      g.out_stride = pp.out_stride;
      g.log2Uper = pp.log2Uper;
      g.tw_log2N = pp.tw_log2N;
      g.tw_h = pp.tw_h;
      g.mode_first = pp.modes[0];
      g.mode_mid = pp.modes[1];
      g.mode_last = pp.modes[2];
      g.swz_tab = pp.swz_tab;
      g.scale = (pp.last && dir == TCU_DFT_INVERSE) ? (float)(1.0 / (double)p->n) : 1.0f;
      if (events && cudaEventRecord((cudaEvent_t)events[pi], st) != cudaSuccess)
        return TCU_DFT_ERR_CUDA;
      if (launch_group_dispatch(p->r, p->precision, pp.s, g, p->num_sms, st) !=
          cudaSuccess)
        return TCU_DFT_ERR_CUDA;
      continue;
    }
    PassArgs a;
    memset(&a, 0, sizeof(a));
    a.in = (pi == 0) ? (const float2 *)in : p->scratch;
    a.out = pp.last ? (float2 *)out : p->scratch;
    a.bimg = p->bimg[di];
    a.twL = pp.twL[di];
    a.twA = p->twA[di];
    a.twB = p->twB[di];
    a.err = p->err;
    a.U = pp.U;
    a.Uper = pp.Uper;
    a.n = p->n;
    a.in_vstride = pp.in_vstride;
    a.in_stride = pp.in_stride;
    a.out_vstride = pp.out_vstride;
    a.out_stride = pp.out_stride;
    a.s = pp.s;
    a.log2L = pp.log2L;
    a.log2G = pp.log2G;
    a.tw_log2N = pp.tw_log2N;
    a.tw_h = pp.tw_h;
    a.scale = (pp.last && dir == TCU_DFT_INVERSE) ? (float)(1.0 / (double)p->n) : 1.0f;
    const long long grid = (pp.U + (1ll << pp.log2G) - 1) >> pp.log2G;
    if (events && cudaEventRecord((cudaEvent_t)events[pi], st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    if (launch_dispatch(p->r, p->precision, a, grid, st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
  }
  if (events && cudaEventRecord((cudaEvent_t)events[p->npasses], st) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  return TCU_DFT_OK;
}

int tcu_dft_exec_dir(tcu_dft_plan_t p, const void *in, void *out, int dir,
                     void *stream) {
  return exec_impl(p, in, out, dir, stream, nullptr);
}

int tcu_dft_exec_timed(tcu_dft_plan_t p, const void *in, void *out, int dir,
                       void *stream, void *const *events) {
  if (!events) return TCU_DFT_ERR_INVALID;
  for (int i = 0; p && i <= p->npasses; ++i)
    if (!events[i]) return TCU_DFT_ERR_INVALID;
  return exec_impl(p, in, out, dir, stream, events);
}

int tcu_dft_exec(tcu_dft_plan_t p, const void *in, void *out, void *stream) {
  return tcu_dft_exec_dir(p, in, out, TCU_DFT_FORWARD, stream);
}

int tcu_dft_exec_host(tcu_dft_plan_t p, const void *h_in, void *h_out, void *d_work,
                      int dir, void *stream) {
  if (!p || !h_in || !h_out || !d_work) return TCU_DFT_ERR_INVALID;
  if ((uintptr_t)d_work & 15) return TCU_DFT_ERR_INVALID;
  const size_t bytes = (size_t)p->batch * p->n * sizeof(float2);
  cudaStream_t st = (cudaStream_t)stream;
  if (cudaMemcpyAsync(d_work, h_in, bytes, cudaMemcpyHostToDevice, st) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  const int rc = tcu_dft_exec_dir(p, d_work, d_work, dir, stream);
  if (rc != TCU_DFT_OK) return rc;
  if (cudaMemcpyAsync(h_out, d_work, bytes, cudaMemcpyDeviceToHost, st) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  return TCU_DFT_OK;
}

int tcu_dft_check(tcu_dft_plan_t p, void *stream) {
  if (!p) return TCU_DFT_ERR_INVALID;
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return TCU_DFT_ERR_CUDA;
  int flag = 0;
  if (cudaMemcpy(&flag, p->err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  if (flag) {
    cudaMemset(p->err, 0, sizeof(int));
    return TCU_DFT_ERR_TIMEOUT;
  }
  return TCU_DFT_OK;
}

int tcu_dft_destroy(tcu_dft_plan_t p) {
  free_plan(p);
  return TCU_DFT_OK;
}

int tcu_dft_num_passes(tcu_dft_plan_t p) { return p ? p->npasses : -1; }

int tcu_dft_pass_stages(tcu_dft_plan_t p, int i) {
  if (!p || i < 0 || i >= p->npasses) return -1;
  return p->pass[i].s;
}

}  // extern "C"
