// host_tables.cu -- host-side tables of a plan: the F_r operand images,
// stage and inter-pass twiddles (fp64 -> fp32 / bf16), the SMEM swizzle
// chosen by a bank-conflict cost model, and the TMA tensor maps.
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

#include "host_plan.h"

using namespace tcu;
using namespace tcu::host;

namespace tcu {
namespace host {

int ilog2(long long v) {
  int l = 0;
  while ((1ll << l) < v) ++l;
  return l;
}

int dir_index(int dir) { return dir == TCU_DFT_INVERSE ? 1 : 0; }

namespace {
thread_local int g_alloc_seq = 0, g_alloc_fail_at = 0;
}  // namespace

void arm_alloc_faults() {
  const char *v = getenv("TCU_DFT_FAIL_ALLOC");
  g_alloc_fail_at = v ? atoi(v) : 0;
  g_alloc_seq = 0;
}

cudaError_t dev_malloc(void **ptr, size_t bytes) {
  if (g_alloc_fail_at > 0 && ++g_alloc_seq == g_alloc_fail_at) {
    *ptr = nullptr;
    return cudaErrorMemoryAllocation;
  }
  return cudaMalloc(ptr, bytes);
}

bool debug_exec() {
  const char *v = getenv("TCU_DFT_DEBUG");
  return v && v[0] == '1';
}

int word_status(int flag) {
  if (flag == 0) return TCU_DFT_OK;
  return flag == TCU_DFT_ERR_BOUNDS ? TCU_DFT_ERR_BOUNDS : TCU_DFT_ERR_TIMEOUT;
}

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

// Round an fp32 value to bf16 (8 significant bits), nearest-even; the bits.
uint16_t host_bf16_rne(float x) {
  uint32_t b;
  memcpy(&b, &x, 4);
  if ((b & 0x7F800000u) != 0x7F800000u) b += 0x7FFFu + ((b >> 16) & 1u);
  return (uint16_t)(b >> 16);
}

float host_bf16_value(uint16_t h) {
  const uint32_t b = (uint32_t)h << 16;
  float r;
  memcpy(&r, &b, 4);
  return r;
}

bool prec_bf16(int precision) { return precision == TCU_DFT_BF16 || precision == TCU_DFT_3XBF16; }

// B operand images of the real 2r x 2r block form of F_r for one direction,
// in the canonical no-swizzle K-major layout the MMA reads: hi, lo, and the
// same two scaled by 2^-log2n (exact: a power of two) for the inverse's last
// stage, which folds the 1/n normalisation into the product.  Core matrices
// are 8 rows x 16 bytes: 4 fp32 (TF32 modes) or 8 bf16 (BF16 modes) of K;
// the four images sit at multiples of their size (16 r^2 or 8 r^2 bytes) in
// a buffer of 64 r^2 bytes.
void build_images(int r, int sign, long long n, int precision, std::vector<float> &out) {
  const int K = 2 * r, N = 2 * r;
  const bool bf = prec_bf16(precision);
  const size_t lbo = 128, sbo = (bf ? 32 : 64) * (size_t)r, esz = bf ? 2 : 4;
  const size_t img_bytes = (bf ? 8 : 16) * (size_t)r * r;
  // n a power of two: the scaled copies are hi, lo times 2^-log2 n (exact);
  // otherwise hi and lo of the fp64 value F / n, rounded separately
  const bool pow2 = (n & (n - 1)) == 0;
  const float sc = pow2 ? ldexpf(1.0f, -ilog2(n)) : 0.f;
  out.assign((size_t)16 * r * r, 0.f);  // 64 r^2 bytes
  unsigned char *bytes = reinterpret_cast<unsigned char *>(out.data());
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
      const int per = bf ? 8 : 4;  // K elements per core-matrix row
      const size_t off = (size_t)(nc >> 3) * sbo + (size_t)(kr / per) * lbo + (nc & 7) * 16 +
                         (size_t)(kr % per) * esz;
      if (bf) {
        const uint16_t hi = host_bf16_rne((float)v);
        const uint16_t lo = host_bf16_rne((float)(v - (double)host_bf16_value(hi)));
        const uint16_t vals[4] = {hi, lo, host_bf16_rne(host_bf16_value(hi) * sc),
                                  host_bf16_rne(host_bf16_value(lo) * sc)};
        for (int i = 0; i < 4; ++i) memcpy(bytes + i * img_bytes + off, &vals[i], 2);
      } else {
        const float hi = host_tf32_rna((float)v);
        const float lo = host_tf32_rna((float)(v - (double)hi));
        const double vs = v / (double)n;
        const float his = pow2 ? hi * sc : host_tf32_rna((float)vs);
        const float los = pow2 ? lo * sc : host_tf32_rna((float)(vs - (double)his));
        const float vals[4] = {hi, lo, his, los};
        for (int i = 0; i < 4; ++i) memcpy(bytes + i * img_bytes + off, &vals[i], 4);
      }
    }
  }
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

int stage_mode(const int modes[3], int t, int S) {
  return t == 1 ? modes[0] : (t == S ? modes[2] : modes[1]);
}

// Shared-memory wavefronts per warp-wide 8-byte access of the warpgroup
// kernel's transposes (1.0 = conflict free), for swizzle table `tab`:
// phys(P) = P ^ ((tab[ul & 15] ^ (P >> 4)) & 15), and for sub-transforms
// longer than 256 points also ^ ((P >> 8) & 15) (gswz in group_kernel.cuh).
double swizzle_cost(int r, int S, const int modes[3], unsigned long long tab, int team) {
  const int log2r = ilog2(r);
  const int L = 1 << (log2r * S);
  const int rps = L / r, gg = 128 * team * r / L;
  long long waves = 0, accesses = 0;
  for (int t = 1; t < S; ++t) {
    for (int side = 0; side < 2; ++side) {  // epilogue write of t, read of t+1
      const int tt = t + side;
      const int mode = stage_mode(modes, tt, S);
      const int sl = log2r * (S - tt);
      for (int w = 0; w < 4 * team; ++w)
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
              unsigned hsw = tv ^ (unsigned)(P >> 4);
              if (log2r * S > 8) hsw ^= (unsigned)(P >> 8);
              const int ph = P ^ (int)(hsw & 15u);
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

unsigned long long choose_swizzle(int r, int S, const int modes[3], int team) {
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
    const double c = swizzle_cost(r, S, modes, t, team);
    if (c < bc - 1e-9) {
      bc = c;
      best = t;
    }
  }
  return best;
}

// Inter-pass twiddles of a strided pass: w_M^{k v}, k < L, v < n2, M = L n2;
// A[k][vl] for vl < min(n2, 256) and, if n2 > 256, B[vh][k] = w_M^{k vh 256}.
void pass_twiddles(long long L, long long n2, int sign, std::vector<float2> &A,
                   std::vector<float2> &B) {
  const long long M = L * n2, VL = n2 > 256 ? 256 : n2;
  A.resize((size_t)(L * VL));
  for (long long k = 0; k < L; ++k)
    for (long long vl = 0; vl < VL; ++vl) A[(size_t)(k * VL + vl)] = root(k * vl, M, sign);
  B.clear();
  if (n2 > VL) {
    B.resize((size_t)((n2 / VL) * L));
    for (long long vh = 0; vh < n2 / VL; ++vh)
      for (long long k = 0; k < L; ++k)
        B[(size_t)(vh * L + k)] = root(k * vh * VL, M, sign);
  }
}

// TMA map of table A of a strided pass (boxes of GG columns x L rows).
bool twiddle_map(CUtensorMap *m, const float2 *A, int r, const PassPlan &pp) {
  const long long L = 1ll << pp.log2L, n2 = 1ll << pp.lo;
  const long long VL = n2 > 256 ? 256 : n2;
  const long long gg = (128ll * pp.tw * r) >> pp.log2L;
  return encode_map(m, A, VL, L, 1, L * VL, (int)gg, L < 256 ? (int)L : 256);
}

// TMA map of a strided pass's input: sequences of M = L n2 points, batch *
// r^sp of them, seen as [sequence][row a][column v].
bool input_map(CUtensorMap *m, const void *in, const tcu_dft_plan_s *p, const PassPlan &pp,
               long long batch) {
  const long long L = 1ll << pp.log2L, n2 = 1ll << pp.lo, pre = 1ll << pp.lp;
  const long long gg = (128ll * pp.tw * p->r) >> pp.log2L;
  return encode_map(m, in, n2, L, batch * pre, L * n2, (int)gg, L < 256 ? (int)L : 256);
}

bool overlaps(const void *a, const void *b, size_t bytes) {
  const char *x = (const char *)a, *y = (const char *)b;
  return x < y + bytes && y < x + bytes;
}

}  // namespace host
}  // namespace tcu
