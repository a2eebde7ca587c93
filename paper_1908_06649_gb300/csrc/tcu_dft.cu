// tcu_dft.cu -- batched complex DFT on GB300 (sm_103a) tensor cores: plan,
// tables, pass scheduling and the C ABI declared in include/tcu_dft.h.
//
// The method (arXiv 1908.06649, Sec. 4.5, Theorem 7): with r = sqrt(m) and
// n = r^k, the Cooley-Tukey recursion arranges x as an r x (n/r) row-major
// matrix, replaces every column by its length-r DFT with ONE tall-left tensor
// product X^T * W_r, multiplies entry (k1, c) by the twiddle w_n^{k1 c},
// transposes, and recurses on the rows; the result is read out column-major.
// Here every stage is exactly that product: the rows of the
// (batch * n / r) x r data matrix times F_r, on tcgen05 tensor cores.
//
// Complex arithmetic (Sec. 4.5: a complex product is four real products and
// two sums) is one real GEMM on interleaved (re, im) data: a data row
// [a0, b0, a1, b1, ...] times the real 2r x 2r block operand
//     Bf[2j][2c] = Re w,  Bf[2j][2c+1] = Im w,
//     Bf[2j+1][2c] = -Im w, Bf[2j+1][2c+1] = Re w,   w = w_r^{jc},
// gives [Re y0, Im y0, Re y1, ...].
//
// Passes.  The k stages are grouped into at most two HBM passes (the
// four-step split n = n1 * n2): pass 1 transforms the n2 stride-n2
// subsequences of length n1 and multiplies by w_n^{b k1}; pass 2 transforms
// the n1 contiguous rows of length n2 and writes y[k1 + n1 k2].  A pass whose
// sub-transforms fit 128 data rows runs on the warpgroup kernel
// (group_kernel.cuh); longer ones on the tile kernel (tile_kernel.cuh).  Two
// warpgroup passes of >= 2 stages each run fused in one launch with an
// L2-resident intermediate.

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cmath>
#include <mutex>
#include <vector>

#include "../../include/tcu_dft.h"
#include "launch.h"

#if defined(__CUDA_ARCH__) && (__CUDA_ARCH__ < 1000)
#error "tcu_dft targets sm_103a (tcgen05); compile with -gencode arch=compute_103a,code=sm_103a"
#endif

using namespace tcu;

namespace {

enum PassKind { kTilePass = 0, kGroupPass = 1 };

struct PassPlan {
  int kind;        // kTilePass or kGroupPass
  int s;
  int log2L;
  int log2G;       // tile kernel: sub-transforms per tile
  long long U, Uper;
  int log2Uper;
  long long in_vstride, in_stride, out_vstride, out_stride;
  int tw_log2N, tw_h;  // tile kernel: inter-pass twiddle, two-level table
  int modes[3];        // group kernel: row map of first / middle / last stage
  unsigned long long swz_tab;
  bool last;
  float2 *twL[2];      // tile kernel: w_L^e          [dir index]
  float2 *tw_stage[2]; // group kernel: [t][j][lo]    [dir index]
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
  float *bimg[2];          // [dir index] hi | lo images
  float2 *twA[2], *twB[2]; // tile kernel pass 1: two-level w_n^e
  float2 *tw_out[2];       // group kernel pass 1: w_n^{b k} as [k][b]
  CUtensorMap tw_map[2];   // TMA map of tw_out[d]
  float2 *scratch;         // intermediate (full size, or the fused ring)
  // fused two-pass schedule
  bool fused;
  int log2C, nchunks, lag, ring_chunks;
  int items1_per_tf, log2_items_per_chunk;
  int *counters;
  size_t counter_bytes;
  int *err;
  int device;
};

namespace {

int dir_index(int dir) { return dir == TCU_DFT_INVERSE ? 1 : 0; }

// cuTensorMapEncodeTiled from the driver, through the runtime (no -lcuda).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
    else
      cudaGetLastError();
  }
  return fn;
}

// TMA map of a [depth][rows][cols] array of complex64 (cols contiguous, row
// pitch cols, plane pitch plane_elems), seen as fp32 pairs; boxes of
// box_cols complex x box_rows rows x 1 plane.
bool encode_map(CUtensorMap *m, const void *base, long long cols, long long rows,
                long long depth, long long plane_elems, int box_cols, int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint64_t dims[3] = {(cuuint64_t)(2 * cols), (cuuint64_t)rows, (cuuint64_t)depth};
  const cuuint64_t strides[2] = {(cuuint64_t)(cols * 8), (cuuint64_t)(plane_elems * 8)};
  const cuuint32_t box[3] = {(cuuint32_t)(2 * box_cols), (cuuint32_t)box_rows, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void *>(base), dims,
             strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

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

// exp(sign * 2 pi i * m / period) with m reduced mod period, fp64 -> fp32
float2 root(long long m, long long period, int sign) {
  m %= period;
  const double ang = (double)sign * 2.0 * M_PI * (double)m / (double)period;
  return make_float2((float)cos(ang), (float)sin(ang));
}

// B operand images of the real 2r x 2r block form of F_r for one direction,
// in the canonical no-swizzle K-major layout the MMA reads: hi, lo, and the
// same two scaled by 2^-log2n (exact: a power of two) for the inverse's last
// stage, which folds the 1/n normalisation into the product.
void build_images(int r, int sign, int log2n, std::vector<float> &out) {
  const int K = 2 * r, N = 2 * r;
  const int lbo = 128, sbo = 64 * r;
  const size_t img_floats = (size_t)16 * r * r / 4;
  const float sc = ldexpf(1.0f, -log2n);
  out.assign(4 * img_floats, 0.f);
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
      out[2 * img_floats + off] = hi * sc;
      out[3 * img_floats + off] = lo * sc;
    }
  }
}

std::vector<float2> twiddle_table(long long period, long long count, long long step,
                                  int sign) {
  std::vector<float2> t((size_t)count);
  for (long long e = 0; e < count; ++e) t[(size_t)e] = root(e * step, period, sign);
  return t;
}

// Stage twiddles of a warpgroup pass: for t = 1 .. s-1 a block [j][lo],
// j < r, lo < r^(s-t), holding w_L^{j * lo * r^(t-1)}.
std::vector<float2> stage_twiddles(int r, int s, int sign) {
  long long L = 1;
  for (int i = 0; i < s; ++i) L *= r;
  std::vector<float2> t;
  long long rt = 1;  // r^(t-1)
  for (int st = 1; st < s; ++st) {
    const long long rows = L / (r * rt);  // r^(s-t)
    for (int j = 0; j < r; ++j)
      for (long long lo = 0; lo < rows; ++lo) t.push_back(root(j * lo * rt, L, sign));
    rt *= r;
  }
  if (t.empty()) t.push_back(make_float2(1.f, 0.f));
  return t;
}

// Largest stage count per pass: tile kernel (a sub-transform fills at most one
// SMEM tile) and warpgroup kernel (a sub-transform fits 128 rows).
int max_tile_stages(int r) { return r == 8 ? 4 : (r == 16 ? 3 : 2); }
int max_group_stages(int r) { return r == 8 ? 3 : 2; }

// Two warpgroup passes of k stages: the strided first pass takes the smaller
// half -- its sub-transforms are shorter, so an item spans more adjacent
// columns and its TMA boxes have wider rows.
void split_two_passes(int k, int stages[2]) {
  stages[0] = k / 2;
  stages[1] = k - stages[0];
}

int stage_mode(const int modes[3], int t, int S) {
  return t == 1 ? modes[0] : (t == S ? modes[2] : modes[1]);
}

// Shared-memory wavefronts per warp-wide 8-byte access of the warpgroup
// kernel's transposes (1.0 = conflict free), for swizzle table `tab`:
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
            int seen = 0, count = 0;
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
    cudaFree(p->tw_out[d]);
    for (int i = 0; i < 2; ++i) {
      cudaFree(p->pass[i].twL[d]);
      cudaFree(p->pass[i].tw_stage[d]);
    }
  }
  cudaFree(p->scratch);
  cudaFree(p->counters);
  cudaFree(p->err);
  delete p;
}

int tile_points(int r) { return r == 8 ? 4096 : 8192; }

// ---------------------------------------------------------------- launches
cudaError_t tile_dispatch(int r, int prec, const PassArgs &a, long long grid,
                          cudaStream_t st) {
  if (r == 8) return launch_tile_r8(prec, a, grid, st);
  if (r == 16) return launch_tile_r16(prec, a, grid, st);
  return launch_tile_r32(prec, a, grid, st);
}

cudaError_t pass_dispatch(int r, int prec, int s, int so, int role, const GArgs &a,
                          int num_sms, cudaStream_t st) {
  if (r == 8) return launch_pass_r8(prec, s, so, role, a, num_sms, st);
  if (r == 16) return launch_pass_r16(prec, s, so, role, a, num_sms, st);
  return launch_pass_r32(prec, s, so, role, a, num_sms, st);
}

cudaError_t fused_dispatch(int r, int prec, int s1, int s2, const GArgs &a, int num_sms,
                           cudaStream_t st) {
  if (r == 8) return launch_fused_r8(prec, s1, s2, a, num_sms, st);
  if (r == 16) return launch_fused_r16(prec, s1, s2, a, num_sms, st);
  return launch_fused_r32(prec, s1, s2, a, num_sms, st);
}

bool overlaps(const void *a, const void *b, size_t bytes) {
  const char *x = (const char *)a, *y = (const char *)b;
  return x < y + bytes && y < x + bytes;
}

// Warpgroup-kernel description of pass `pi` between buffers `in` and `out`.
PRun group_pass(const tcu_dft_plan_s *p, int pi, int di, const float2 *in, float2 *out,
                long long in_bmask, long long out_bmask, bool inverse) {
  const PassPlan &pp = p->pass[pi];
  PRun g;
  memset(&g, 0, sizeof(g));
  g.in = in;
  g.out = out;
  g.in_bmask = in_bmask;
  g.out_bmask = out_bmask;
  g.U = pp.U;
  g.tw_out = (pi == 0 && p->npasses == 2) ? p->tw_out[di] : nullptr;
  g.tw_stage = pp.tw_stage[di];
  g.swz_tab = pp.swz_tab;
  // the inverse's last stage uses the F images scaled by 1/n
  g.last_img = (pp.last && inverse) ? 2 * 16 * p->r * p->r : 0;
  return g;
}

int pass_role(const tcu_dft_plan_s *p, int pi) {
  return p->npasses == 1 ? kSingle : (pi == 0 ? kFirst : kSecond);
}

int other_stages(const tcu_dft_plan_s *p, int pi) {
  return p->npasses == 1 ? 0 : p->pass[1 - pi].s;
}

// TMA maps of a first (strided) warpgroup pass: its input x[b][a][v] and
// its inter-pass twiddles.
bool first_pass_maps(const tcu_dft_plan_s *p, int di, const void *in, GArgs *g) {
  const PassPlan &p1 = p->pass[0];
  const long long n1 = 1ll << p1.log2L, n2 = p->n / n1;
  const long long gg1 = (128ll * p->r) >> p1.log2L;
  const int box_rows = n1 < 256 ? (int)n1 : 256;
  if (!encode_map(&g->tm_in, in, n2, n1, p->batch, p->n, (int)gg1, box_rows)) return false;
  g->tm_tw = p->tw_map[di];
  return true;
}

// ------------------------------------------- fixed memory of exec_noalloc
// tcu_dft_exec_noalloc keeps everything besides the caller's buffers in
// these file-scope arrays.  In host code their names are only stand-ins:
// kernels get the device addresses resolved by cudaGetSymbolAddress.
constexpr long long kNaMaxPoints = 1ll << 22;      // two-pass intermediate
constexpr long long kNaMaxN = 1ll << 18;           // longest transform
constexpr int kNaImgFloats = 4 * 16 * 32 * 32 / 4;  // 4 F_r images, r <= 32
constexpr int kNaStageTw = 1024;                    // stage twiddles of a pass
static __device__ __align__(256) float2 g_na_scratch[kNaMaxPoints];
static __device__ __align__(256) float g_na_img[2][kNaImgFloats];
static __device__ __align__(256) float2 g_na_tw_stage[2][2][kNaStageTw];
static __device__ __align__(256) float2 g_na_tw_out[2][kNaMaxN];
static __device__ __align__(256) int g_na_err;

struct NaDevice {
  bool ready;  // device addresses resolved
  int num_sms;
  float2 *scratch;
  float *img;
  float2 *tw_stage;
  float2 *tw_out;
  int *err;
  long long n;  // tables currently held (0: none)
  int r;
  CUtensorMap tw_map[2];
};

std::mutex g_na_mutex;
NaDevice g_na_dev[64];

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
    case TCU_DFT_ERR_TOO_LARGE:
      return "size exceeds the fixed memory of tcu_dft_exec_noalloc";
    default: return "unknown status";
  }
}

int tcu_dft_last_error(void) { return g_last_error; }

tcu_dft_plan_t tcu_dft_plan(int64_t n, int64_t batch, int32_t sqrt_m,
                            int32_t precision) {
  return tcu_dft_plan_ex(n, batch, sqrt_m, precision, TCU_DFT_PLAN_DEFAULT);
}

tcu_dft_plan_t tcu_dft_plan_ex(int64_t n, int64_t batch, int32_t sqrt_m,
                               int32_t precision, uint32_t flags) {
  g_last_error = TCU_DFT_OK;
  if (n < 1 || batch < 1 || (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32) ||
      (flags & ~(uint32_t)(TCU_DFT_PLAN_NO_FUSE | TCU_DFT_PLAN_FUSE)) ||
      ((flags & TCU_DFT_PLAN_NO_FUSE) && (flags & TCU_DFT_PLAN_FUSE))) {
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
  // Pass grouping: prefer the warpgroup kernel (sub-transforms of <= 128
  // rows), fall back to the tile kernel for longer sub-transforms.
  const int sg = max_group_stages(r), stl = max_tile_stages(r);
  int stages[2] = {0, 0}, kinds[2] = {kGroupPass, kGroupPass}, npasses;
  if (k <= sg) {
    npasses = 1;
    stages[0] = k;
  } else if (k <= 2 * sg) {
    npasses = 2;
    split_two_passes(k, stages);
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
      if (pp.kind == kTilePass)
        rc = upload(&pp.twL[d], twiddle_table(L, L, 1, sign));
      else
        rc = upload(&pp.tw_stage[d], stage_twiddles(r, pp.s, sign));
    }
  }
  for (int d = 0; d < 2 && rc == TCU_DFT_OK; ++d) {
    const int sign = d == 0 ? -1 : 1;
    std::vector<float> img;
    build_images(r, sign, log2n, img);
    rc = upload(&p->bimg[d], img);
    if (rc == TCU_DFT_OK && npasses == 2) {
      if (p->pass[0].kind == kTilePass) {
        const int h = p->pass[0].tw_h;
        rc = upload(&p->twA[d], twiddle_table(n, n >> h, 1ll << h, sign));
        if (rc == TCU_DFT_OK) rc = upload(&p->twB[d], twiddle_table(n, 1ll << h, 1, sign));
      } else {
        // [k1][b] = w_n^{b k1}, b < n2, k1 < n1
        const long long n1 = 1ll << p->pass[0].log2L, n2 = n / n1;
        std::vector<float2> t((size_t)n);
        for (long long k1 = 0; k1 < n1; ++k1)
          for (long long b = 0; b < n2; ++b) t[(size_t)(k1 * n2 + b)] = root(b * k1, n, sign);
        rc = upload(&p->tw_out[d], t);
        const long long gg1 = (128ll * r) >> p->pass[0].log2L;
        const int box_rows = n1 < 256 ? (int)n1 : 256;
        if (rc == TCU_DFT_OK &&
            !encode_map(&p->tw_map[d], p->tw_out[d], n2, n1, 1, n, (int)gg1, box_rows))
          rc = TCU_DFT_ERR_CUDA;
      }
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
    const PassPlan &p1 = p->pass[0], &p2 = p->pass[1];
    p->fused = p1.kind == kGroupPass && p2.kind == kGroupPass && p1.s >= 2 && p2.s >= 2 &&
               (flags & TCU_DFT_PLAN_FUSE);
    long long scratch_tf = batch;
    if (p->fused) {
      // chunks of C transforms (a power of two dividing the batch, <= 8);
      // pass 2 trails pass 1 by `lag` chunks; the ring holds 8 chunks and
      // transform b's intermediate sits at ring slot b & (8 C - 1)
      int log2C = 0;
      while (log2C < 3 && (batch % (2ll << log2C)) == 0) ++log2C;
      p->log2C = log2C;
      p->nchunks = (int)(batch >> log2C);
      p->lag = p->nchunks < 4 ? p->nchunks : 4;
      p->ring_chunks = 8;
      const long long n1 = 1ll << p1.log2L, n2 = 1ll << p2.log2L;
      const long long gg1 = (128ll * r) >> p1.log2L, gg2 = (128ll * r) >> p2.log2L;
      p->items1_per_tf = (int)(n2 / gg1);
      // every item is 128 r points, so both passes have n C / (128 r) per chunk
      if ((n2 / gg1) != (n1 / gg2)) rc = TCU_DFT_ERR_UNSUPPORTED;
      p->log2_items_per_chunk = ilog2(n2 / gg1) + log2C;
      scratch_tf = (long long)p->ring_chunks << log2C;
      p->counter_bytes = (size_t)(1 + batch + p->nchunks) * sizeof(int);
      if (cudaMalloc((void **)&p->counters, p->counter_bytes) != cudaSuccess) {
        cudaGetLastError();
        rc = TCU_DFT_ERR_OOM;
      }
    }
    if (rc == TCU_DFT_OK &&
        cudaMalloc((void **)&p->scratch, (size_t)scratch_tf * n * sizeof(float2)) !=
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
  const float scale_last =
      dir == TCU_DFT_INVERSE ? (float)(1.0 / (double)p->n) : 1.0f;

  const bool inverse = dir == TCU_DFT_INVERSE;
  if (p->fused) {
    GArgs g;
    memset(&g, 0, sizeof(g));
    const long long ring_mask = ((long long)p->ring_chunks << p->log2C) - 1;
    g.p[0] = group_pass(p, 0, di, (const float2 *)in, p->scratch, -1, ring_mask, inverse);
    g.p[1] = group_pass(p, 1, di, p->scratch, (float2 *)out, ring_mask, -1, inverse);
    if (!first_pass_maps(p, di, in, &g)) return TCU_DFT_ERR_CUDA;
    g.bimg = p->bimg[di];
    g.err = p->err;
    g.counters = p->counters;
    g.batch = p->batch;
    g.nchunks = p->nchunks;
    g.lag = p->lag;
    g.ring_chunks = p->ring_chunks;
    g.items1_per_tf = p->items1_per_tf;
    g.log2_items_per_chunk = p->log2_items_per_chunk;
    if (cudaMemsetAsync(p->counters, 0, p->counter_bytes, st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    if (events && cudaEventRecord((cudaEvent_t)events[0], st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    if (fused_dispatch(p->r, p->precision, p->pass[0].s, p->pass[1].s, g, p->num_sms,
                       st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    // one fused launch covers both passes: events[1] == events[2]
    if (events && (cudaEventRecord((cudaEvent_t)events[1], st) != cudaSuccess ||
                   cudaEventRecord((cudaEvent_t)events[2], st) != cudaSuccess))
      return TCU_DFT_ERR_CUDA;
    return TCU_DFT_OK;
  }

  for (int pi = 0; pi < p->npasses; ++pi) {
    const PassPlan &pp = p->pass[pi];
    const float2 *src = (pi == 0) ? (const float2 *)in : p->scratch;
    float2 *dst = pp.last ? (float2 *)out : p->scratch;
    const float scale = pp.last ? scale_last : 1.0f;
    if (events && cudaEventRecord((cudaEvent_t)events[pi], st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    if (pp.kind == kGroupPass) {
      GArgs g;
      memset(&g, 0, sizeof(g));
      g.p[0] = group_pass(p, pi, di, src, dst, -1, -1, inverse);
      if (pass_role(p, pi) == kFirst && !first_pass_maps(p, di, src, &g))
        return TCU_DFT_ERR_CUDA;
      g.bimg = p->bimg[di];
      g.err = p->err;
      if (pass_dispatch(p->r, p->precision, pp.s, other_stages(p, pi), pass_role(p, pi), g,
                        p->num_sms, st) != cudaSuccess)
        return TCU_DFT_ERR_CUDA;
      continue;
    }
    PassArgs a;
    memset(&a, 0, sizeof(a));
    a.in = src;
    a.out = dst;
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
    a.scale = scale;
    const long long grid = (pp.U + (1ll << pp.log2G) - 1) >> pp.log2G;
    if (tile_dispatch(p->r, p->precision, a, grid, st) != cudaSuccess)
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

int tcu_dft_is_fused(tcu_dft_plan_t p) { return p ? (p->fused ? 1 : 0) : -1; }

int tcu_dft_pass_stages(tcu_dft_plan_t p, int i) {
  if (!p || i < 0 || i >= p->npasses) return -1;
  return p->pass[i].s;
}

int tcu_dft_exec_noalloc(int64_t n, int64_t batch, int32_t sqrt_m, int32_t precision,
                         const void *in, void *out, int dir, void *stream) {
  // ---- arguments (no CUDA call before they are known to be good)
  if (n < 1 || batch < 1 || (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32) ||
      !in || !out || (dir != TCU_DFT_FORWARD && dir != TCU_DFT_INVERSE))
    return TCU_DFT_ERR_INVALID;
  if (sqrt_m != 8 && sqrt_m != 16 && sqrt_m != 32) return TCU_DFT_ERR_UNSUPPORTED;
  const int r = sqrt_m, log2r = ilog2(r);
  int k = 0;
  long long m = 1;
  while (m < n) {
    m *= r;
    ++k;
  }
  if (m != n) return TCU_DFT_ERR_UNSUPPORTED;
  const int sg = max_group_stages(r);
  if (k > 2 * sg || n > kNaMaxN) return TCU_DFT_ERR_TOO_LARGE;
  const int npasses = k <= sg ? 1 : 2;
  if (npasses == 2 && batch * n > kNaMaxPoints) return TCU_DFT_ERR_TOO_LARGE;
  int stages[2] = {k, 0};
  if (npasses == 2) split_two_passes(k, stages);
  const int log2n = ilog2(n);
  cudaStream_t st = (cudaStream_t)stream;

  std::lock_guard<std::mutex> lock(g_na_mutex);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return TCU_DFT_ERR_CUDA;
  }
  NaDevice &D = g_na_dev[dev];
  if (!D.ready) {
    // once per device, with it current: where the fixed arrays live
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess || prop.major != 10 ||
        prop.minor != 3 ||
        cudaGetSymbolAddress((void **)&D.scratch, g_na_scratch) != cudaSuccess ||
        cudaGetSymbolAddress((void **)&D.img, g_na_img) != cudaSuccess ||
        cudaGetSymbolAddress((void **)&D.tw_stage, g_na_tw_stage) != cudaSuccess ||
        cudaGetSymbolAddress((void **)&D.tw_out, g_na_tw_out) != cudaSuccess ||
        cudaGetSymbolAddress((void **)&D.err, g_na_err) != cudaSuccess) {
      cudaGetLastError();
      return TCU_DFT_ERR_CUDA;
    }
    D.num_sms = prop.multiProcessorCount;
    D.n = 0;
    D.ready = true;
  }

  // ---- the plan, on the stack, pointing into the fixed arrays
  tcu_dft_plan_s p;
  memset(&p, 0, sizeof(p));
  p.n = n;
  p.batch = batch;
  p.r = r;
  p.log2r = log2r;
  p.k = k;
  p.precision = precision;
  p.npasses = npasses;
  p.num_sms = D.num_sms;
  p.device = dev;
  p.fused = false;
  p.scratch = D.scratch;
  p.err = D.err;
  for (int d = 0; d < 2; ++d) {
    p.bimg[d] = D.img + (size_t)d * kNaImgFloats;
    p.tw_out[d] = D.tw_out + (size_t)d * kNaMaxN;
  }
  for (int pi = 0; pi < npasses; ++pi) {
    PassPlan &pp = p.pass[pi];
    pp.kind = kGroupPass;
    pp.s = stages[pi];
    pp.log2L = log2r * pp.s;
    pp.last = (pi == npasses - 1);
    const long long L = 1ll << pp.log2L;
    if (npasses == 1) {
      pp.U = batch;
      pp.Uper = 1;
      pp.in_vstride = n;
      pp.in_stride = 1;
      pp.out_vstride = n;
      pp.out_stride = 1;
    } else if (pi == 0) {
      pp.U = batch * (n / L);
      pp.Uper = n / L;
      pp.in_vstride = 1;
      pp.in_stride = n / L;
      pp.out_vstride = 1;
      pp.out_stride = n / L;
    } else {
      pp.U = batch * (n / L);
      pp.Uper = n / L;
      pp.in_vstride = L;
      pp.in_stride = 1;
      pp.out_vstride = 1;
      pp.out_stride = n / L;
    }
    pp.log2Uper = ilog2(pp.Uper);
    pp.modes[0] = pp.in_stride == 1 ? kQF : kUF;
    pp.modes[1] = kUF;
    pp.modes[2] = pp.out_stride == 1 ? kRQF : kUF;
    pp.swz_tab = choose_swizzle(r, pp.s, pp.modes);
    for (int d = 0; d < 2; ++d)
      pp.tw_stage[d] = D.tw_stage + ((size_t)d * 2 + pi) * kNaStageTw;
  }

  // ---- tables for this (n, r), refilled only when they change
  if (D.n != n || D.r != r) {
    D.n = 0;
    for (int d = 0; d < 2; ++d) {
      const int sign = d == 0 ? -1 : 1;
      std::vector<float> img;
      build_images(r, sign, log2n, img);
      if (cudaMemcpyAsync(p.bimg[d], img.data(), img.size() * sizeof(float),
                          cudaMemcpyHostToDevice, st) != cudaSuccess)
        return TCU_DFT_ERR_CUDA;
      for (int pi = 0; pi < npasses; ++pi) {
        const std::vector<float2> t = stage_twiddles(r, p.pass[pi].s, sign);
        if (cudaMemcpyAsync(p.pass[pi].tw_stage[d], t.data(), t.size() * sizeof(float2),
                            cudaMemcpyHostToDevice, st) != cudaSuccess)
          return TCU_DFT_ERR_CUDA;
      }
      if (npasses == 2) {
        const long long n1 = 1ll << p.pass[0].log2L, n2 = n / n1;
        std::vector<float2> t((size_t)n);
        for (long long k1 = 0; k1 < n1; ++k1)
          for (long long b = 0; b < n2; ++b) t[(size_t)(k1 * n2 + b)] = root(b * k1, n, sign);
        if (cudaMemcpyAsync(p.tw_out[d], t.data(), t.size() * sizeof(float2),
                            cudaMemcpyHostToDevice, st) != cudaSuccess)
          return TCU_DFT_ERR_CUDA;
        const long long gg1 = (128ll * r) >> p.pass[0].log2L;
        if (!encode_map(&D.tw_map[d], p.tw_out[d], n2, n1, 1, n, (int)gg1,
                        n1 < 256 ? (int)n1 : 256))
          return TCU_DFT_ERR_CUDA;
      }
    }
    D.n = n;
    D.r = r;
  }
  for (int d = 0; d < 2; ++d) p.tw_map[d] = D.tw_map[d];

  // the timeout word must start at zero; then the ordinary two-launch path
  if (cudaMemsetAsync(D.err, 0, sizeof(int), st) != cudaSuccess) return TCU_DFT_ERR_CUDA;
  return exec_impl(&p, in, out, dir, stream, nullptr);
}

}  // extern "C"
