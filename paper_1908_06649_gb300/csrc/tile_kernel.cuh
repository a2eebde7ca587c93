// tile_kernel.cuh -- the general pass kernel: one CTA transforms a tile of
// G sub-transforms of length L = r^s (s <= 4) held whole in shared memory.
// Used for sub-transforms longer than 128 data rows (L > 128 r), which the
// warpgroup kernel cannot hold.
#pragma once
#include "tcgen05.cuh"

namespace tcu {

constexpr int kThreads = 128;  // 4 warps: one per TMEM lane quarter

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
__global__ void __launch_bounds__(kThreads, 1) dft_tile_kernel(const PassArgs a) {
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

}  // namespace tcu
