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
// Passes.  The k stages are grouped into at most three HBM passes of at most
// two stages (three for r = 8) -- the four-step split n = n1 * n2 applied
// recursively, so that every pass's sub-transforms fit one warpgroup item of
// 128 data rows (group_kernel.cuh).  Pass p splits each length-M_p sequence
// left by the passes before it (M_1 = n) into L_p rows of n2_p = M_p / L_p
// columns: it transforms the strided columns, multiplies by w_{M_p}^{k v}
// and stores row k of sequence q as row (k, q) of the next pass's input,
// transform-major with k above q; the last pass transforms contiguous rows
// and writes y[q + k * n / L] in natural order.  A two-pass transform may
// instead run fused in one launch with an L2-resident intermediate.

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

constexpr int kMaxPasses = 3;
constexpr int kHostChunks = 16;  // pipeline depth of the host-buffer path

struct PassPlan {
  int s;            // stages
  int role;         // kSingle, kFirst (strided) or kSecond (last of several)
  int so;           // kFirst: stages after this pass; kSecond: stages before
  int sp;           // kFirst: stages before this pass
  int lo;           // log2: columns of a strided pass / points before the last
  int lp;           // log2: prefix sequences per transform of a strided pass
  int log2L;        // sub-transform length L = r^s
  long long U;      // sub-transforms in the pass
  int modes[3];     // row map of the first / middle / last stage
  unsigned long long swz_tab;
  bool last;
  float2 *tw_stage[2];   // stage twiddles [t][j][lo]          [dir index]
  // kFirst: w_M^{k v}, M = r^(s + so): A [k][vl], B [vh][k] (v = vh 256 + vl,
  // B only when n2 = r^so exceeds 256)
  float2 *tw_a[2], *tw_b[2];
  CUtensorMap tw_map[2];  // TMA map of tw_a[d]
  // mixed radix: q > 0 marks the CUDA-core q-point first pass (roots of the
  // direction); `mixed` a tensor-core pass of a mixed-radix transform
  int q;
  RootsQ roots[2];
  bool mixed;
  int tw;           // warpgroups per item (teams for the 3-stage radix-8 passes)
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
  PassPlan pass[kMaxPasses];
  float *bimg[2];          // [dir index] hi | lo | scaled hi | scaled lo images
  float2 *scratch[2];      // intermediates (or the fused ring in scratch[0])
  // fused two-pass schedule
  bool fused;
  int log2C, nchunks, lag, ring_chunks;
  int items1_per_tf, log2_items_per_chunk;
  int *counters;
  size_t counter_bytes;
  int *err;
  int device;
  // host-buffer path: copy streams and per-chunk events (created by the plan)
  cudaStream_t copy_in, copy_out;
  cudaEvent_t ev_start, ev_in[kHostChunks], ev_done[kHostChunks], ev_out[kHostChunks];
  bool has_copy_streams;
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
void build_images(int r, int sign, int log2n, int precision, std::vector<float> &out) {
  const int K = 2 * r, N = 2 * r;
  const bool bf = prec_bf16(precision);
  const size_t lbo = 128, sbo = (bf ? 32 : 64) * (size_t)r, esz = bf ? 2 : 4;
  const size_t img_bytes = (bf ? 8 : 16) * (size_t)r * r;
  const float sc = ldexpf(1.0f, -log2n);
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
        const float vals[4] = {hi, lo, hi * sc, lo * sc};
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
// phys(P) = P ^ ((tab[ul & 15] ^ (P >> 4)) & 15).
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

// Stages per pass.  Passes hold at most two stages (three for r = 8, whose
// 3-stage sub-transforms of 512 points still fit a 128-row item); up to
// three passes; the earlier passes take the smaller shares, so the strided
// passes have shorter sub-transforms, more adjacent columns per item and
// wider TMA rows.  Returns the number of passes, 0 if n is too long.
int plan_stages(int r, int k, int st[kMaxPasses]) {
  const int sg = r == 8 ? 3 : 2;
  if (k <= sg || (r == 16 && k == 3)) {
    // 16^3 in one pass on items of two warpgroups (one 4096-point transform)
    st[0] = k;
    return 1;
  }
  if (r == 8 && k <= 6) {
    // two passes of 2 + 3 or 3 + 3: the 3-stage passes run on teams of
    // warpgroups (team_size), whose items span 8 adjacent columns
    st[0] = k / 2;
    st[1] = k - st[0];
    return 2;
  }
  int P = (k + 1) / 2;
  if (P > kMaxPasses) P = kMaxPasses;
  const int base = k / P, extra = k % P;
  for (int i = 0; i < P; ++i) {
    st[i] = base + (i >= P - extra ? 1 : 0);
    if (st[i] > sg) return 0;
  }
  return P;
}

// Mixed radix n = q r^k (q < r a power of two; the base case of the
// recursion is a DFT of size q < sqrt(m)): a CUDA-core q-point first pass,
// then the r^k-point transforms of its q rows in one or two tensor-core
// passes (stage split as plan_stages).  Instantiated: k = 2..4 for r = 8
// and 16, k = 2..3 for r = 32.  Returns the number of passes (0: not such
// an n) and fills the passes.
int plan_mixed(int r, long long n, long long batch, PassPlan pass[kMaxPasses]) {
  const int log2r = ilog2(r);
  if (n < 1 || (n & (n - 1))) return 0;
  const int log2n = ilog2(n), k = log2n / log2r, lq = log2n - k * log2r;
  const int kmax = r == 32 ? 3 : 4;
  if (lq == 0 || k < 2 || k > kmax) return 0;
  int st[kMaxPasses] = {0, 0, 0};
  const int tc = k <= (r == 8 ? 3 : 2) ? 1 : 2;
  if (tc == 1) st[0] = k;
  else {
    st[0] = k / 2;
    st[1] = k - st[0];
  }
  PassPlan &p0 = pass[0];
  p0.q = 1 << lq;
  p0.s = 1;
  p0.role = kFirst;
  p0.log2L = lq;
  p0.lo = k * log2r;
  p0.lp = 0;
  p0.U = batch * (n >> lq);
  for (int d = 0; d < 2; ++d)
    for (int m = 0; m < 16; ++m) p0.roots[d].w[m] = root(m, p0.q, d == 0 ? -1 : 1);
  for (int i = 0; i < tc; ++i) {
    PassPlan &pp = pass[1 + i];
    pp.mixed = true;
    pp.s = st[i];
    pp.log2L = log2r * pp.s;
    pp.last = (i == tc - 1);
    if (pp.last) {
      pp.role = kSecond;
      pp.lo = lq + (i ? log2r * st[0] : 0);
      pp.lp = 0;
    } else {
      pp.role = kFirst;
      pp.lo = log2r * st[1];
      pp.lp = lq;
    }
    pp.U = batch * (n >> pp.log2L);
    pp.modes[0] = pp.role == kFirst ? kUF : kQF;
    pp.modes[1] = kUF;
    pp.modes[2] = kUF;
    pp.tw = 1;
    pp.swz_tab = choose_swizzle(r, pp.s, pp.modes, 1);
  }
  return 1 + tc;
}

// Warpgroups per item of pass pp: 4 for the 3-stage radix-8 passes of
// two-pass transforms (an item of 512 rows holds 8 sub-transforms of 512
// points, so the strided side moves 64-byte runs), else 1.
int team_size(int r, int npasses, const PassPlan &pp) {
  if (r == 16 && npasses == 1 && pp.s == 3) return 2;
  return (r == 8 && npasses == 2 && pp.s == 3 && pp.role != kCols) ? 4 : 1;
}

// Role, neighbouring stage counts, size and row maps of pass `pi`.
void pass_geometry(PassPlan &pp, int pi, int P, const int st[kMaxPasses], int k, int r,
                   long long n, long long batch) {
  int before = 0;
  for (int i = 0; i < pi; ++i) before += st[i];
  pp.s = st[pi];
  pp.log2L = ilog2(r) * pp.s;
  pp.last = (pi == P - 1);
  if (P == 1) {
    pp.role = kSingle;
    pp.so = pp.sp = 0;
  } else if (pp.last) {
    pp.role = kSecond;
    pp.so = before;
    pp.sp = 0;
  } else {
    pp.role = kFirst;
    pp.so = k - before - pp.s;
    pp.sp = before;
  }
  pp.lo = ilog2(r) * pp.so;
  pp.lp = ilog2(r) * pp.sp;
  pp.U = batch * (n >> pp.log2L);
  pp.modes[0] = pp.role == kFirst ? kUF : kQF;
  pp.modes[1] = kUF;
  pp.modes[2] = pp.role == kSingle ? kRQF : kUF;
  pp.tw = team_size(r, P, pp);
  pp.swz_tab = choose_swizzle(r, pp.s, pp.modes, pp.tw);
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

void free_plan(tcu_dft_plan_s *p) {
  if (!p) return;
  if (p->has_copy_streams) {
    // null handles (creation failed part-way) are skipped
    if (p->copy_in) cudaStreamSynchronize(p->copy_in), cudaStreamDestroy(p->copy_in);
    if (p->copy_out) cudaStreamSynchronize(p->copy_out), cudaStreamDestroy(p->copy_out);
    if (p->ev_start) cudaEventDestroy(p->ev_start);
    for (int i = 0; i < kHostChunks; ++i) {
      if (p->ev_in[i]) cudaEventDestroy(p->ev_in[i]);
      if (p->ev_done[i]) cudaEventDestroy(p->ev_done[i]);
      if (p->ev_out[i]) cudaEventDestroy(p->ev_out[i]);
    }
  }
  for (int d = 0; d < 2; ++d) {
    cudaFree(p->bimg[d]);
    for (int i = 0; i < kMaxPasses; ++i) {
      cudaFree(p->pass[i].tw_stage[d]);
      cudaFree(p->pass[i].tw_a[d]);
      cudaFree(p->pass[i].tw_b[d]);
    }
    cudaFree(p->scratch[d]);
  }
  cudaFree(p->counters);
  cudaFree(p->err);
  delete p;
}

// ---------------------------------------------------------------- launches
cudaError_t pass_dispatch(int r, int prec, const PassPlan &pp, const GArgs &a, int num_sms,
                          cudaStream_t st, bool team_plan = false) {
  if (pp.mixed) {
    if (r == 8) return launch_pass_mixed_r8(prec, pp.s, pp.lo, pp.role, pp.lp, a, num_sms, st);
    if (r == 16) return launch_pass_mixed_r16(prec, pp.s, pp.lo, pp.role, pp.lp, a, num_sms, st);
    return launch_pass_mixed_r32(prec, pp.s, pp.lo, pp.role, pp.lp, a, num_sms, st);
  }
  if (prec_bf16(prec))
    return launch_pass_bf16_r16(prec, pp.s, pp.lo, pp.role, pp.lp, pp.tw, a, num_sms, st);
  if (r == 8 && team_plan)
    return launch_team_r8(prec, pp.s, pp.lo, pp.role, pp.lp, pp.tw, a, num_sms, st);
  if (r == 16 && pp.tw > 1)
    return launch_team_r16(prec, pp.s, pp.lo, pp.role, pp.lp, pp.tw, a, num_sms, st);
  if (r == 8) return launch_pass_r8(prec, pp.s, pp.lo, pp.role, pp.lp, a, num_sms, st);
  if (r == 16) return launch_pass_r16(prec, pp.s, pp.lo, pp.role, pp.lp, a, num_sms, st);
  return launch_pass_r32(prec, pp.s, pp.lo, pp.role, pp.lp, a, num_sms, st);
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
                long long in_bmask, long long out_bmask, bool inverse, long long batch) {
  const PassPlan &pp = p->pass[pi];
  PRun g;
  memset(&g, 0, sizeof(g));
  g.in = in;
  g.out = out;
  g.in_bmask = in_bmask;
  g.out_bmask = out_bmask;
  g.U = batch * (p->n >> pp.log2L);
  g.tw_out = pp.tw_a[di];
  g.tw_b = pp.tw_b[di];
  g.tw_stage = pp.tw_stage[di];
  g.swz_tab = pp.swz_tab;
  // the inverse's last stage uses the F images scaled by 1/n
  g.last_img = (pp.last && inverse) ? 2 * (prec_bf16(p->precision) ? 8 : 16) * p->r * p->r : 0;
  return g;
}

// Tables of a plan for one direction d: F images, stage twiddles and the
// inter-pass twiddles, as host vectors (uploaded by the caller).
struct DirTables {
  std::vector<float> img;
  std::vector<float2> stage[kMaxPasses], A[kMaxPasses], B[kMaxPasses];
};

void dir_tables(const tcu_dft_plan_s *p, int d, DirTables &t) {
  const int sign = d == 0 ? -1 : 1;
  build_images(p->r, sign, ilog2(p->n), p->precision, t.img);
  for (int pi = 0; pi < p->npasses; ++pi) {
    const PassPlan &pp = p->pass[pi];
    t.stage[pi] = stage_twiddles(p->r, pp.q ? 1 : pp.s, sign);
    if (pp.role == kFirst) pass_twiddles(1ll << pp.log2L, 1ll << pp.lo, sign, t.A[pi], t.B[pi]);
  }
}

// ------------------------------------------- fixed memory of exec_noalloc
// tcu_dft_exec_noalloc keeps everything besides the caller's buffers in
// these file-scope arrays.  In host code their names are only stand-ins:
// kernels get the device addresses resolved by cudaGetSymbolAddress.
constexpr long long kNaMaxPoints = 1ll << 22;      // two-pass intermediate
constexpr long long kNaMaxN = 1ll << 18;           // longest transform
constexpr int kNaImgFloats = 4 * 16 * 32 * 32 / 4;  // 4 F_r images, r <= 32
constexpr int kNaStageTw = 4608;  // stage twiddles of a pass (16^3 + 16^2 = 4352 for 3 stages)
static __device__ __align__(256) float2 g_na_scratch[kNaMaxPoints];
static __device__ __align__(256) float g_na_img[2][kNaImgFloats];
static __device__ __align__(256) float2 g_na_tw_stage[2][2][kNaStageTw];
static __device__ __align__(256) float2 g_na_tw_out[2][kNaMaxN];  // A, then B
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
  if (n < 1 || batch < 1 ||
      (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32 && !prec_bf16(precision)) ||
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
  int st[kMaxPasses] = {0, 0, 0};
  PassPlan mixed[kMaxPasses];
  memset(mixed, 0, sizeof(mixed));
  const bool is_mixed = m != n;
  const int npasses = is_mixed ? plan_mixed(r, n, batch, mixed)
                               : (k >= 1 ? plan_stages(r, k, st) : 0);
  // the BF16 modes are instantiated for radix 16, r^k sizes
  if (npasses == 0 || (long long)batch * n > (1ll << 40) ||
      (prec_bf16(precision) && (r != 16 || is_mixed))) {
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
  if (is_mixed)
    for (int pi = 0; pi < npasses; ++pi) p->pass[pi] = mixed[pi];
  else
    for (int pi = 0; pi < npasses; ++pi) pass_geometry(p->pass[pi], pi, npasses, st, k, r, n, batch);
  int rc = TCU_DFT_OK;
  for (int d = 0; d < 2 && rc == TCU_DFT_OK; ++d) {
    DirTables t;
    dir_tables(p, d, t);
    rc = upload(&p->bimg[d], t.img);
    for (int pi = 0; pi < npasses && rc == TCU_DFT_OK; ++pi) {
      PassPlan &pp = p->pass[pi];
      rc = upload(&pp.tw_stage[d], t.stage[pi]);
      if (rc == TCU_DFT_OK && pp.role == kFirst) {
        rc = upload(&pp.tw_a[d], t.A[pi]);
        if (rc == TCU_DFT_OK && !t.B[pi].empty()) rc = upload(&pp.tw_b[d], t.B[pi]);
        if (rc == TCU_DFT_OK && !pp.q && !twiddle_map(&pp.tw_map[d], pp.tw_a[d], r, pp))
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
  if (rc == TCU_DFT_OK && npasses >= 2) {
    const PassPlan &p1 = p->pass[0], &p2 = p->pass[1];
    // fused kernels are instantiated for 2 + 2 stages
    p->fused = !is_mixed && !prec_bf16(precision) && npasses == 2 && p1.s == 2 &&
               p2.s == 2 && (flags & TCU_DFT_PLAN_FUSE);
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
      if (rc == TCU_DFT_OK && cudaMalloc((void **)&p->counters, p->counter_bytes) != cudaSuccess) {
        cudaGetLastError();
        rc = TCU_DFT_ERR_OOM;
      }
    }
    for (int i = 0; i < npasses - 1 && rc == TCU_DFT_OK; ++i)
      if (cudaMalloc((void **)&p->scratch[i], (size_t)scratch_tf * n * sizeof(float2)) !=
          cudaSuccess) {
        cudaGetLastError();
        rc = TCU_DFT_ERR_OOM;
      }
  }
  if (rc == TCU_DFT_OK) {
    bool ok = cudaStreamCreateWithFlags(&p->copy_in, cudaStreamNonBlocking) == cudaSuccess &&
              cudaStreamCreateWithFlags(&p->copy_out, cudaStreamNonBlocking) == cudaSuccess &&
              cudaEventCreateWithFlags(&p->ev_start, cudaEventDisableTiming) == cudaSuccess;
    for (int i = 0; i < kHostChunks && ok; ++i)
      ok = cudaEventCreateWithFlags(&p->ev_in[i], cudaEventDisableTiming) == cudaSuccess &&
           cudaEventCreateWithFlags(&p->ev_done[i], cudaEventDisableTiming) == cudaSuccess &&
           cudaEventCreateWithFlags(&p->ev_out[i], cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
      cudaGetLastError();
      rc = TCU_DFT_ERR_CUDA;
    }
    p->has_copy_streams = true;  // whatever was created is freed with the plan
  }
  if (rc != TCU_DFT_OK) {
    free_plan(p);
    g_last_error = rc;
    return nullptr;
  }
  return p;
}

// The transform of transforms [b0, b0 + count) of the plan's batch (in and
// out point at transform b0; count < 0: the whole batch).  The intermediates
// of that range sit at the same offset in the plan's scratch, so disjoint
// ranges may run concurrently on different streams (not fused plans).
static int exec_impl(tcu_dft_plan_t p, const void *in, void *out, int dir,
                     void *stream, void *const *events, long long queue_start = 0,
                     long long b0 = 0, long long count = -1) {
  if (!p || !in || !out || (dir != TCU_DFT_FORWARD && dir != TCU_DFT_INVERSE))
    return TCU_DFT_ERR_INVALID;
  if (((uintptr_t)in & 15) || ((uintptr_t)out & 15)) return TCU_DFT_ERR_INVALID;
  if (count < 0) count = p->batch;
  if (b0 < 0 || b0 + count > p->batch || (p->fused && count != p->batch))
    return TCU_DFT_ERR_INVALID;
  const size_t bytes = (size_t)count * p->n * sizeof(float2);
  if (in != out && overlaps(in, out, bytes)) return TCU_DFT_ERR_INVALID;
  cudaStream_t st = (cudaStream_t)stream;
  const int di = dir_index(dir);
  const bool inverse = dir == TCU_DFT_INVERSE;
  if (p->fused) {
    GArgs g;
    memset(&g, 0, sizeof(g));
    const long long ring_mask = ((long long)p->ring_chunks << p->log2C) - 1;
    g.p[0] = group_pass(p, 0, di, (const float2 *)in, p->scratch[0], -1, ring_mask, inverse,
                        p->batch);
    g.p[1] = group_pass(p, 1, di, p->scratch[0], (float2 *)out, ring_mask, -1, inverse,
                        p->batch);
    if (!input_map(&g.tm_in, in, p, p->pass[0], p->batch)) return TCU_DFT_ERR_CUDA;
    g.tm_tw = p->pass[0].tw_map[di];
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
    if (queue_start > 0) {
      // failure-detection self-test: start the queue past work that then
      // never runs (pageable source: copied before the call returns)
      const int head = (int)queue_start;
      if (cudaMemcpyAsync(p->counters, &head, sizeof(int), cudaMemcpyHostToDevice, st) !=
          cudaSuccess)
        return TCU_DFT_ERR_CUDA;
    }
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

  // in -> scratch[0] -> scratch[1] -> out
  const long long off = b0 * p->n;
  for (int pi = 0; pi < p->npasses; ++pi) {
    const PassPlan &pp = p->pass[pi];
    const float2 *src = (pi == 0) ? (const float2 *)in : p->scratch[pi - 1] + off;
    float2 *dst = pp.last ? (float2 *)out : p->scratch[pi] + off;
    if (events && cudaEventRecord((cudaEvent_t)events[pi], st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    if (pp.q) {
      if (launch_radix_q(pp.q, src, dst, count, pp.lo, pp.tw_a[di], pp.tw_b[di],
                         pp.roots[di], p->num_sms, st) != cudaSuccess)
        return TCU_DFT_ERR_CUDA;
      continue;
    }
    GArgs g;
    memset(&g, 0, sizeof(g));
    g.p[0] = group_pass(p, pi, di, src, dst, -1, -1, inverse, count);
    if (pp.role == kFirst) {
      if (!input_map(&g.tm_in, src, p, pp, count)) return TCU_DFT_ERR_CUDA;
      g.tm_tw = pp.tw_map[di];
    }
    g.bimg = p->bimg[di];
    g.err = p->err;
    bool team_plan = false;
    for (int i = 0; i < p->npasses; ++i) team_plan |= p->pass[i].tw > 1;
    if (pass_dispatch(p->r, p->precision, pp, g, p->num_sms, st, team_plan) != cudaSuccess)
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

int tcu_dft_exec_stalled(tcu_dft_plan_t p, const void *in, void *out, void *stream) {
  // the first items claimed are the pass-2 items of chunk 0, whose pass-1
  // items sit before the start and never run
  if (!p || !p->fused || p->nchunks < p->lag + 2) return TCU_DFT_ERR_INVALID;
  const long long start = (long long)(p->lag + 1) << p->log2_items_per_chunk;
  return exec_impl(p, in, out, TCU_DFT_FORWARD, stream, nullptr, start);
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
  if (!p || !h_in || !h_out || !d_work || (dir != TCU_DFT_FORWARD && dir != TCU_DFT_INVERSE))
    return TCU_DFT_ERR_INVALID;
  if ((uintptr_t)d_work & 15) return TCU_DFT_ERR_INVALID;
  const size_t bytes = (size_t)p->batch * p->n * sizeof(float2);
  cudaStream_t st = (cudaStream_t)stream;
  if (p->fused || !p->has_copy_streams || p->batch < 2) {
    if (cudaMemcpyAsync(d_work, h_in, bytes, cudaMemcpyHostToDevice, st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    const int rc = tcu_dft_exec_dir(p, d_work, d_work, dir, stream);
    if (rc != TCU_DFT_OK) return rc;
    if (cudaMemcpyAsync(h_out, d_work, bytes, cudaMemcpyDeviceToHost, st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    return TCU_DFT_OK;
  }
  // Pipelined over up to kHostChunks chunks of transforms: chunk c's host->device
  // copy (copy_in stream), its transform (the caller's stream) and its
  // device->host copy (copy_out stream) overlap with the neighbouring
  // chunks'; events order each chunk's three steps and join the copy
  // streams to the caller's stream at both ends.
  const long long C = p->batch < kHostChunks ? p->batch : kHostChunks;
  const long long per = (p->batch + C - 1) / C;
  float2 *d = (float2 *)d_work;
  const float2 *hin = (const float2 *)h_in;
  float2 *hout = (float2 *)h_out;
  if (cudaEventRecord(p->ev_start, st) != cudaSuccess ||
      cudaStreamWaitEvent(p->copy_in, p->ev_start, 0) != cudaSuccess ||
      cudaStreamWaitEvent(p->copy_out, p->ev_start, 0) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  int last = 0;
  for (long long c = 0; c < C; ++c) {
    const long long b0 = c * per;
    if (b0 >= p->batch) break;
    const long long cnt = (b0 + per <= p->batch) ? per : p->batch - b0;
    const size_t off = (size_t)(b0 * p->n), cb = (size_t)cnt * p->n * sizeof(float2);
    if (cudaMemcpyAsync(d + off, hin + off, cb, cudaMemcpyHostToDevice, p->copy_in) !=
            cudaSuccess ||
        cudaEventRecord(p->ev_in[c], p->copy_in) != cudaSuccess ||
        cudaStreamWaitEvent(st, p->ev_in[c], 0) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    const int rc = exec_impl(p, d + off, d + off, dir, stream, nullptr, 0, b0, cnt);
    if (rc != TCU_DFT_OK) return rc;
    if (cudaEventRecord(p->ev_done[c], st) != cudaSuccess ||
        cudaStreamWaitEvent(p->copy_out, p->ev_done[c], 0) != cudaSuccess ||
        cudaMemcpyAsync(hout + off, d + off, cb, cudaMemcpyDeviceToHost, p->copy_out) !=
            cudaSuccess ||
        cudaEventRecord(p->ev_out[c], p->copy_out) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    last = (int)c;
  }
  return cudaStreamWaitEvent(st, p->ev_out[last], 0) == cudaSuccess ? TCU_DFT_OK
                                                                     : TCU_DFT_ERR_CUDA;
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

int tcu_dft_plan_passes(int64_t n, int32_t sqrt_m, int32_t *stages) {
  if (n < 1 || !stages || (sqrt_m != 8 && sqrt_m != 16 && sqrt_m != 32)) return 0;
  const int r = sqrt_m;
  int k = 0;
  long long m = 1;
  while (m < n) {
    m *= r;
    ++k;
  }
  int st[kMaxPasses] = {0, 0, 0};
  int np = 0;
  if (m == n) {
    np = k >= 1 ? plan_stages(r, k, st) : 0;
  } else {
    PassPlan mixed[kMaxPasses];
    memset(mixed, 0, sizeof(mixed));
    np = plan_mixed(r, n, 1, mixed);
    for (int i = 0; i < np; ++i) st[i] = mixed[i].s;
  }
  for (int i = 0; i < np; ++i) stages[i] = st[i];
  return np;
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
  if (n < 1 || batch < 1 ||
      (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32 && !prec_bf16(precision)) ||
      !in || !out || (dir != TCU_DFT_FORWARD && dir != TCU_DFT_INVERSE))
    return TCU_DFT_ERR_INVALID;
  if (prec_bf16(precision)) return TCU_DFT_ERR_UNSUPPORTED;
  if (sqrt_m != 8 && sqrt_m != 16 && sqrt_m != 32) return TCU_DFT_ERR_UNSUPPORTED;
  const int r = sqrt_m, log2r = ilog2(r);
  int k = 0;
  long long m = 1;
  while (m < n) {
    m *= r;
    ++k;
  }
  if (m != n) return TCU_DFT_ERR_UNSUPPORTED;
  int st[kMaxPasses] = {0, 0, 0};
  const int npasses = plan_stages(r, k, st);
  if (npasses == 0 || npasses > 2 || n > kNaMaxN) return TCU_DFT_ERR_TOO_LARGE;
  if (npasses == 2 && batch * n > kNaMaxPoints) return TCU_DFT_ERR_TOO_LARGE;
  cudaStream_t stream_ = (cudaStream_t)stream;

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
  p.scratch[0] = D.scratch;
  p.err = D.err;
  for (int pi = 0; pi < npasses; ++pi) pass_geometry(p.pass[pi], pi, npasses, st, k, r, n, batch);
  for (int d = 0; d < 2; ++d) p.bimg[d] = D.img + (size_t)d * kNaImgFloats;
  for (int pi = 0; pi < npasses; ++pi)
    for (int d = 0; d < 2; ++d)
      p.pass[pi].tw_stage[d] = D.tw_stage + ((size_t)d * 2 + pi) * kNaStageTw;

  // ---- tables for this (n, r), refilled only when they change; table A of
  // the strided pass at the start of the direction's twiddle array, B after it
  DirTables t[2];
  for (int d = 0; d < 2; ++d) {
    dir_tables(&p, d, t[d]);
    for (int pi = 0; pi < npasses; ++pi)
      if (t[d].stage[pi].size() > (size_t)kNaStageTw) return TCU_DFT_ERR_TOO_LARGE;
    if (npasses == 2) {
      p.pass[0].tw_a[d] = D.tw_out + (size_t)d * kNaMaxN;
      if (!t[d].B[0].empty()) p.pass[0].tw_b[d] = p.pass[0].tw_a[d] + t[d].A[0].size();
    }
  }
  if (D.n != n || D.r != r) {
    D.n = 0;
    for (int d = 0; d < 2; ++d) {
      if (cudaMemcpyAsync(p.bimg[d], t[d].img.data(), t[d].img.size() * sizeof(float),
                          cudaMemcpyHostToDevice, stream_) != cudaSuccess)
        return TCU_DFT_ERR_CUDA;
      for (int pi = 0; pi < npasses; ++pi)
        if (cudaMemcpyAsync(p.pass[pi].tw_stage[d], t[d].stage[pi].data(),
                            t[d].stage[pi].size() * sizeof(float2), cudaMemcpyHostToDevice,
                            stream_) != cudaSuccess)
          return TCU_DFT_ERR_CUDA;
      if (npasses == 2) {
        if (cudaMemcpyAsync(p.pass[0].tw_a[d], t[d].A[0].data(),
                            t[d].A[0].size() * sizeof(float2), cudaMemcpyHostToDevice,
                            stream_) != cudaSuccess)
          return TCU_DFT_ERR_CUDA;
        if (!t[d].B[0].empty() &&
            cudaMemcpyAsync(p.pass[0].tw_b[d], t[d].B[0].data(),
                            t[d].B[0].size() * sizeof(float2), cudaMemcpyHostToDevice,
                            stream_) != cudaSuccess)
          return TCU_DFT_ERR_CUDA;
        if (!twiddle_map(&D.tw_map[d], p.pass[0].tw_a[d], r, p.pass[0]))
          return TCU_DFT_ERR_CUDA;
      }
    }
    D.n = n;
    D.r = r;
  }
  for (int d = 0; d < 2; ++d) p.pass[0].tw_map[d] = D.tw_map[d];

  // the timeout word must start at zero; then the ordinary launch path
  if (cudaMemsetAsync(D.err, 0, sizeof(int), stream_) != cudaSuccess) return TCU_DFT_ERR_CUDA;
  return exec_impl(&p, in, out, dir, stream, nullptr);
}

// =========================================================== 2-D transforms
// A 2-D DFT of batch row-major n1 x n2 arrays (Sec. 4.6: the 1-D DFT of
// every column, then of every row) is two warpgroup passes: the column pass
// (kCols: kFirst's strided geometry without a twiddle, T[b][k1][v]) and the
// row pass (kSingle over batch * n1 rows, natural order).  A circular
// convolution with a fixed array whose spectrum S is given is three:
// columns, rows (forward, times S, inverse -- on chip, one item at a time),
// inverse columns (1/(n1 n2) folded into the last stage's F images).

}  // extern "C"

struct tcu_dft2_plan_s {
  long long n1, n2, batch;
  int r, precision, num_sms;
  PassPlan cols, rows;
  float *bimg[2];     // [dir index]; scaled copies by 2^-log2(n1 n2)
  float *cimg;        // convolution rows: forward hi, lo | inverse hi, lo
  float2 *scratch;    // batch * n1 * n2
  int *err;
};

struct tcu_stencil_plan_s {
  long long side, N, Nw, tiles;
  int k, r, precision, num_sms;
  tcu_dft2_plan_t conv;   // N x N, batch = tiles
  tcu_dft2_plan_t wconv;  // N x N, batch 1 (spectrum of the kernel)
  tcu_dft2_plan_t wpow;   // Nw x Nw, batch 1 (Lemma 2)
  float2 *tile_buf;       // tiles * N * N
  float2 *wgrid;          // Nw * Nw
  float2 *wker;           // N * N: the kernel W', then its spectrum
};

namespace {

bool is_power_of(long long n, int r, int &k) {
  k = 0;
  long long m = 1;
  while (m < n) {
    m *= r;
    ++k;
  }
  return m == n && k >= 1;
}

// A single-pass stage count for radix r (the largest sub-transform of one
// warpgroup item).
int single_pass_stages(int r) { return r == 8 ? 3 : 2; }

void free_dft2(tcu_dft2_plan_s *p) {
  if (!p) return;
  for (int d = 0; d < 2; ++d) {
    cudaFree(p->bimg[d]);
    cudaFree(p->cols.tw_stage[d]);
    cudaFree(p->rows.tw_stage[d]);
  }
  cudaFree(p->cimg);
  cudaFree(p->scratch);
  cudaFree(p->err);
  delete p;
}

// Column-pass TMA map: [array][row a][column v], GG columns x n1 rows.
bool cols_map(CUtensorMap *m, const void *in, const tcu_dft2_plan_s *p) {
  const long long gg = (128ll * p->r) / p->n1;
  return encode_map(m, in, p->n2, p->n1, p->batch, p->n1 * p->n2, (int)gg,
                    p->n1 < 256 ? (int)p->n1 : 256);
}

PRun dft2_pass(const tcu_dft2_plan_s *p, const PassPlan &pp, int di, const float2 *in,
               float2 *out, bool scaled, const float2 *spec) {
  PRun g;
  memset(&g, 0, sizeof(g));
  g.in = in;
  g.out = out;
  g.in_bmask = g.out_bmask = -1;
  g.U = pp.U;
  g.tw_stage = pp.tw_stage[di];
  g.swz_tab = pp.swz_tab;
  g.last_img = scaled ? 2 * 16 * p->r * p->r : 0;
  g.spec = spec;
  g.spec_mask = p->n1 - 1;
  return g;
}

int run_dft2_pass(const tcu_dft2_plan_s *p, const PassPlan &pp, int di, const float2 *in,
                  float2 *out, bool scaled, const float2 *spec, cudaStream_t st) {
  GArgs g;
  memset(&g, 0, sizeof(g));
  g.p[0] = dft2_pass(p, pp, di, in, out, scaled, spec);
  if (pp.role == kCols && !cols_map(&g.tm_in, in, p)) return TCU_DFT_ERR_CUDA;
  g.bimg = p->bimg[di];
  g.err = p->err;
  return pass_dispatch(p->r, p->precision, pp, g, p->num_sms, st) == cudaSuccess
             ? TCU_DFT_OK
             : TCU_DFT_ERR_CUDA;
}

int check_buffers(const void *in, const void *out, size_t bytes) {
  if (!in || !out || ((uintptr_t)in & 15) || ((uintptr_t)out & 15)) return TCU_DFT_ERR_INVALID;
  if (in != out && overlaps(in, out, bytes)) return TCU_DFT_ERR_INVALID;
  return TCU_DFT_OK;
}

tcu_dft2_plan_s *make_dft2(int64_t n1, int64_t n2, int64_t batch, int32_t r,
                           int32_t precision, int &rc) {
  rc = TCU_DFT_OK;
  if (n1 < 1 || n2 < 1 || batch < 1 ||
      (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32 && !prec_bf16(precision))) {
    rc = TCU_DFT_ERR_INVALID;
    return nullptr;
  }
  if (prec_bf16(precision)) {  // the 2-D passes are instantiated for the TF32 modes
    rc = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  int k1 = 0, k2 = 0;
  if ((r != 8 && r != 16 && r != 32) || !is_power_of(n1, r, k1) || !is_power_of(n2, r, k2) ||
      k1 > single_pass_stages(r) || k2 > single_pass_stages(r) ||
      n1 * n2 < 128ll * r || batch * n1 * n2 > (1ll << 40)) {
    // each axis one warpgroup pass; a column item spans 128 r / n1 columns
    rc = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  int dev = 0;
  cudaDeviceProp prop;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaGetDeviceProperties(&prop, dev) != cudaSuccess ||
      prop.major != 10 || prop.minor != 3) {
    cudaGetLastError();
    rc = TCU_DFT_ERR_CUDA;
    return nullptr;
  }
  tcu_dft2_plan_s *p = new tcu_dft2_plan_s();
  memset(p, 0, sizeof(*p));
  p->n1 = n1;
  p->n2 = n2;
  p->batch = batch;
  p->r = r;
  p->precision = precision;
  p->num_sms = prop.multiProcessorCount;
  const int log2r = ilog2(r);
  PassPlan &c = p->cols, &w = p->rows;
  c.s = k1;
  c.role = kCols;
  c.so = k2;
  c.sp = 0;
  c.lo = log2r * k2;
  c.lp = 0;
  c.log2L = log2r * k1;
  c.U = batch * n2;
  c.modes[0] = c.modes[1] = c.modes[2] = kUF;
  c.tw = 1;
  c.swz_tab = choose_swizzle(r, c.s, c.modes, 1);
  w.s = k2;
  w.role = kSingle;
  w.so = w.sp = w.lo = w.lp = 0;
  w.log2L = log2r * k2;
  w.U = batch * n1;
  w.modes[0] = kQF;
  w.modes[1] = kUF;
  w.modes[2] = kRQF;
  w.tw = 1;
  w.swz_tab = choose_swizzle(r, w.s, w.modes, 1);
  std::vector<float> conv_img;
  for (int d = 0; d < 2 && rc == TCU_DFT_OK; ++d) {
    const int sign = d == 0 ? -1 : 1;
    std::vector<float> img;
    build_images(r, sign, ilog2(n1 * n2), precision, img);
    rc = upload(&p->bimg[d], img);
    // hi and lo of this direction (the first two images)
    conv_img.insert(conv_img.end(), img.begin(), img.begin() + img.size() / 2);
    if (rc == TCU_DFT_OK) rc = upload(&c.tw_stage[d], stage_twiddles(r, c.s, sign));
    if (rc == TCU_DFT_OK) rc = upload(&w.tw_stage[d], stage_twiddles(r, w.s, sign));
  }
  if (rc == TCU_DFT_OK) rc = upload(&p->cimg, conv_img);
  if (rc == TCU_DFT_OK &&
      (cudaMalloc((void **)&p->scratch, (size_t)(batch * n1 * n2) * sizeof(float2)) !=
           cudaSuccess ||
       cudaMalloc((void **)&p->err, sizeof(int)) != cudaSuccess ||
       cudaMemset(p->err, 0, sizeof(int)) != cudaSuccess)) {
    cudaGetLastError();
    rc = TCU_DFT_ERR_OOM;
  }
  if (rc != TCU_DFT_OK) {
    free_dft2(p);
    return nullptr;
  }
  return p;
}

void free_stencil(tcu_stencil_plan_s *p) {
  if (!p) return;
  free_dft2(p->conv);
  free_dft2(p->wconv);
  free_dft2(p->wpow);
  cudaFree(p->tile_buf);
  cudaFree(p->wgrid);
  cudaFree(p->wker);
  delete p;
}

// Smallest power of r, at least `need`, whose square holds a column item
// (128 r points) and that one warpgroup pass transforms; 0 if none.
long long grid_side(int r, long long need) {
  long long N = r;
  for (int s = 1; s <= single_pass_stages(r); ++s, N *= r)
    if (N >= need && N * N >= 128ll * r) return N;
  return 0;
}

}  // namespace

extern "C" {

tcu_dft2_plan_t tcu_dft2_plan(int64_t n1, int64_t n2, int64_t batch, int32_t sqrt_m,
                              int32_t precision) {
  int rc;
  tcu_dft2_plan_s *p = make_dft2(n1, n2, batch, sqrt_m, precision, rc);
  g_last_error = rc;
  return p;
}

int tcu_dft2_exec(tcu_dft2_plan_t p, const void *in, void *out, int dir, void *stream) {
  if (!p || (dir != TCU_DFT_FORWARD && dir != TCU_DFT_INVERSE)) return TCU_DFT_ERR_INVALID;
  const size_t bytes = (size_t)(p->batch * p->n1 * p->n2) * sizeof(float2);
  int rc = check_buffers(in, out, bytes);
  if (rc != TCU_DFT_OK) return rc;
  cudaStream_t st = (cudaStream_t)stream;
  const int di = dir_index(dir);
  rc = run_dft2_pass(p, p->cols, di, (const float2 *)in, p->scratch, false, nullptr, st);
  if (rc == TCU_DFT_OK)
    rc = run_dft2_pass(p, p->rows, di, p->scratch, (float2 *)out, dir == TCU_DFT_INVERSE,
                       nullptr, st);
  return rc;
}

int tcu_conv2_exec(tcu_dft2_plan_t p, const void *in, const void *spectrum, void *out,
                   void *stream) {
  if (!p || !spectrum || ((uintptr_t)spectrum & 15)) return TCU_DFT_ERR_INVALID;
  const size_t bytes = (size_t)(p->batch * p->n1 * p->n2) * sizeof(float2);
  int rc = check_buffers(in, out, bytes);
  if (rc != TCU_DFT_OK) return rc;
  cudaStream_t st = (cudaStream_t)stream;
  // columns: in -> scratch; rows forward, times the spectrum and inverse on
  // chip: scratch -> scratch (an item reads its rows before writing them);
  // inverse columns with 1/(n1 n2): scratch -> out
  rc = run_dft2_pass(p, p->cols, 0, (const float2 *)in, p->scratch, false, nullptr, st);
  if (rc != TCU_DFT_OK) return rc;
  GArgs g;
  memset(&g, 0, sizeof(g));
  g.p[0] = dft2_pass(p, p->rows, 0, p->scratch, p->scratch, false, (const float2 *)spectrum);
  g.p[1].tw_stage = p->rows.tw_stage[1];
  g.bimg = p->cimg;
  g.err = p->err;
  cudaError_t e;
  if (p->r == 8) e = launch_rowconv_r8(p->precision, p->rows.s, g, p->num_sms, st);
  else if (p->r == 16) e = launch_rowconv_r16(p->precision, p->rows.s, g, p->num_sms, st);
  else e = launch_rowconv_r32(p->precision, p->rows.s, g, p->num_sms, st);
  if (e != cudaSuccess) return TCU_DFT_ERR_CUDA;
  return run_dft2_pass(p, p->cols, 1, p->scratch, (float2 *)out, true, nullptr, st);
}

int tcu_dft2_check(tcu_dft2_plan_t p, void *stream) {
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

int tcu_dft2_destroy(tcu_dft2_plan_t p) {
  free_dft2(p);
  return TCU_DFT_OK;
}

tcu_stencil_plan_t tcu_stencil_plan(int64_t side, int32_t steps, int32_t sqrt_m,
                                    int32_t precision) {
  g_last_error = TCU_DFT_OK;
  if (side < 1 || steps < 1 ||
      (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32 && !prec_bf16(precision))) {
    g_last_error = TCU_DFT_ERR_INVALID;
    return nullptr;
  }
  if (prec_bf16(precision)) {
    g_last_error = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  const long long N = (sqrt_m == 8 || sqrt_m == 16 || sqrt_m == 32) ? grid_side(sqrt_m, 3ll * steps) : 0;
  const long long Nw = N ? grid_side(sqrt_m, 2ll * steps + 1) : 0;
  if (!N || !Nw || side % steps != 0) {
    g_last_error = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  const long long tpr = side / steps;
  tcu_stencil_plan_s *p = new tcu_stencil_plan_s();
  memset(p, 0, sizeof(*p));
  p->side = side;
  p->k = steps;
  p->r = sqrt_m;
  p->precision = precision;
  p->N = N;
  p->Nw = Nw;
  p->tiles = tpr * tpr;
  int rc = TCU_DFT_OK;
  p->conv = make_dft2(N, N, p->tiles, sqrt_m, precision, rc);
  if (rc == TCU_DFT_OK) p->wconv = make_dft2(N, N, 1, sqrt_m, precision, rc);
  if (rc == TCU_DFT_OK) p->wpow = make_dft2(Nw, Nw, 1, sqrt_m, precision, rc);
  if (rc == TCU_DFT_OK) {
    p->num_sms = p->conv->num_sms;
    if (cudaMalloc((void **)&p->tile_buf, (size_t)(p->tiles * N * N) * sizeof(float2)) !=
            cudaSuccess ||
        cudaMalloc((void **)&p->wgrid, (size_t)(Nw * Nw) * sizeof(float2)) != cudaSuccess ||
        cudaMalloc((void **)&p->wker, (size_t)(N * N) * sizeof(float2)) != cudaSuccess) {
      cudaGetLastError();
      rc = TCU_DFT_ERR_OOM;
    }
  }
  if (rc != TCU_DFT_OK) {
    free_stencil(p);
    g_last_error = rc;
    return nullptr;
  }
  return p;
}

// Lemma 2 on the device: P placed on the Nw x Nw grid, its 2-D DFT, the
// pointwise k-th power, the inverse 2-D DFT; W = the centred real part.
static int stencil_weight_grid(tcu_stencil_plan_t p, const float *w3x3, cudaStream_t st) {
  Stencil3 w;
  for (int i = 0; i < 9; ++i) w.w[i] = w3x3[i];
  const long long cnt = p->Nw * p->Nw;
  if (launch_place_poly(p->wgrid, p->Nw, w, p->num_sms, st) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  int rc = tcu_dft2_exec(p->wpow, p->wgrid, p->wgrid, TCU_DFT_FORWARD, st);
  if (rc != TCU_DFT_OK) return rc;
  if (launch_cpow(p->wgrid, cnt, p->k, p->num_sms, st) != cudaSuccess) return TCU_DFT_ERR_CUDA;
  return tcu_dft2_exec(p->wpow, p->wgrid, p->wgrid, TCU_DFT_INVERSE, st);
}

int tcu_stencil_weights(tcu_stencil_plan_t p, const float *w3x3, float *W, void *stream) {
  if (!p || !w3x3 || !W) return TCU_DFT_ERR_INVALID;
  cudaStream_t st = (cudaStream_t)stream;
  int rc = stencil_weight_grid(p, w3x3, st);
  if (rc != TCU_DFT_OK) return rc;
  return launch_extract_weights(W, p->wgrid, p->Nw, p->k, p->num_sms, st) == cudaSuccess
             ? TCU_DFT_OK
             : TCU_DFT_ERR_CUDA;
}

int tcu_stencil_exec(tcu_stencil_plan_t p, const float *w3x3, const float *A, float *Ak,
                     void *stream) {
  if (!p || !w3x3 || !A || !Ak) return TCU_DFT_ERR_INVALID;
  const size_t bytes = (size_t)(p->side * p->side) * sizeof(float);
  if (A != Ak && overlaps(A, Ak, bytes)) return TCU_DFT_ERR_INVALID;
  cudaStream_t st = (cudaStream_t)stream;
  // W (Lemma 2), the kernel W' and its spectrum
  int rc = stencil_weight_grid(p, w3x3, st);
  if (rc != TCU_DFT_OK) return rc;
  if (launch_place_kernel(p->wker, p->N, p->wgrid, p->Nw, p->k, p->num_sms, st) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  rc = tcu_dft2_exec(p->wconv, p->wker, p->wker, TCU_DFT_FORWARD, st);
  if (rc != TCU_DFT_OK) return rc;
  // Lemma 1: all tiles A'_{r,c} as one batch, circular convolution, centres
  if (launch_gather_tiles(p->tile_buf, A, p->side, p->k, p->N, p->num_sms, st) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  rc = tcu_conv2_exec(p->conv, p->tile_buf, p->wker, p->tile_buf, st);
  if (rc != TCU_DFT_OK) return rc;
  return launch_extract_tiles(Ak, p->tile_buf, p->side, p->k, p->N, p->num_sms, st) ==
                 cudaSuccess
             ? TCU_DFT_OK
             : TCU_DFT_ERR_CUDA;
}

int tcu_stencil_check(tcu_stencil_plan_t p, void *stream) {
  if (!p) return TCU_DFT_ERR_INVALID;
  int rc = tcu_dft2_check(p->wpow, stream);
  if (rc == TCU_DFT_OK) rc = tcu_dft2_check(p->wconv, stream);
  if (rc == TCU_DFT_OK) rc = tcu_dft2_check(p->conv, stream);
  return rc;
}

int tcu_stencil_destroy(tcu_stencil_plan_t p) {
  free_stencil(p);
  return TCU_DFT_OK;
}

}  // extern "C"
