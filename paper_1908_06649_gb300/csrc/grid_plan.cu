// grid_plan.cu -- the 2-D rows of the library (Sec. 4.6): 2-D DFT plans,
// circular 2-D convolution and the linear stencil of Lemmas 1 and 2.
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

// =========================================================== 2-D transforms
// A 2-D DFT of batch row-major n1 x n2 arrays (Sec. 4.6: the 1-D DFT of
// every column, then of every row) is two warpgroup passes: the column pass
// (kCols: kFirst's strided geometry without a twiddle, T[b][k1][v]) and the
// row pass (kSingle over batch * n1 rows, natural order).  A circular
// convolution with a fixed array whose spectrum S is given is three:
// columns, rows (forward, times S, inverse -- on chip, one item at a time),
// inverse columns (1/(n1 n2) folded into the last stage's F images).


// Axes beyond one warpgroup pass (or the BF16 modes): the general path.
// The rows of every array are one batched 1-D plan of length n2 (several
// passes where needed); the arrays are transposed so that the columns are
// contiguous, transformed by a 1-D plan of length n1 and transposed back.
// A convolution multiplies by the spectrum on the transposed layout (the
// spectrum transposed once per call into a plan buffer) between the forward
// and the inverse column plans.
struct tcu_dft2_plan_s {
  long long n1, n2, batch;
  int r, precision, num_sms;
  PassPlan cols, rows;
  float *bimg[2];     // [dir index]; scaled copies by 2^-log2(n1 n2)
  float *cimg;        // convolution rows: forward hi, lo | inverse hi, lo
  float2 *scratch;    // batch * n1 * n2
  int *err;
  bool general;
  tcu_dft_plan_t rows1d, cols1d;  // general path: length n2 / n1 plans
  float2 *spec_t;                 // general path: the spectrum transposed
};

struct tcu_stencil_plan_s {
  long long side, N, Nw, tiles;
  int B;  // output block side: N - 2k (Lemma 1's tiles are blocks of k)
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
  tcu_dft_destroy(p->rows1d);
  tcu_dft_destroy(p->cols1d);
  cudaFree(p->spec_t);
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
               float2 *out, bool scaled, const float2 *spec, int reverse = 0) {
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
  g.reverse = reverse;
  return g;
}

int run_dft2_pass(const tcu_dft2_plan_s *p, const PassPlan &pp, int di, const float2 *in,
                  float2 *out, bool scaled, const float2 *spec, cudaStream_t st) {
  GArgs g;
  memset(&g, 0, sizeof(g));
  // the row pass follows the column pass: items last to first (L2 reuse)
  g.p[0] = dft2_pass(p, pp, di, in, out, scaled, spec, pp.role == kCols ? 0 : 1);
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

// The general path: 1-D plans for the rows (n2, batch n1 of them) and the
// columns (n1, batch n2 of them), a scratch array and the transposed
// spectrum of a convolution.  UNSUPPORTED if either length has no 1-D plan.
tcu_dft2_plan_s *make_dft2_general(int64_t n1, int64_t n2, int64_t batch, int32_t r,
                                   int32_t precision, int &rc) {
  // both lengths must have a 1-D plan (a host-side question: no CUDA call)
  int32_t st[kMaxPasses];
  if (tcu_dft_plan_passes(n1, r, st) == 0 || tcu_dft_plan_passes(n2, r, st) == 0) {
    rc = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  tcu_dft2_plan_s *p = new tcu_dft2_plan_s();
  memset(p, 0, sizeof(*p));
  p->n1 = n1;
  p->n2 = n2;
  p->batch = batch;
  p->r = r;
  p->precision = precision;
  p->general = true;
  p->rows1d = tcu_dft_plan(n2, batch * n1, r, precision);
  rc = p->rows1d ? TCU_DFT_OK : tcu_dft_last_error();
  if (rc == TCU_DFT_OK) {
    p->cols1d = tcu_dft_plan(n1, batch * n2, r, precision);
    rc = p->cols1d ? TCU_DFT_OK : tcu_dft_last_error();
  }
  if (rc == TCU_DFT_OK) {
    p->num_sms = p->rows1d->num_sms;
    if (dev_malloc((void **)&p->scratch, (size_t)(batch * n1 * n2) * sizeof(float2)) !=
            cudaSuccess ||
        dev_malloc((void **)&p->spec_t, (size_t)(n1 * n2) * sizeof(float2)) != cudaSuccess ||
        dev_malloc((void **)&p->err, sizeof(int)) != cudaSuccess ||
        cudaMemset(p->err, 0, sizeof(int)) != cudaSuccess) {
      cudaGetLastError();
      rc = TCU_DFT_ERR_OOM;
    }
  }
  if (rc != TCU_DFT_OK) {
    free_dft2(p);
    return nullptr;
  }
  return p;
}

// General path: the 2-D transform of `in` into `out` (rows, transpose,
// columns, transpose back), or -- with keep_t -- left transposed in the
// plan's scratch after the columns (the convolution continues there).
int general_dft2(const tcu_dft2_plan_s *p, const void *in, void *out, int dir, bool keep_t,
                 cudaStream_t st) {
  int rc = tcu_dft_exec_dir(p->rows1d, in, out, dir, st);
  if (rc != TCU_DFT_OK) return rc;
  if (launch_transpose(p->scratch, (const float2 *)out, p->batch, p->n1, p->n2, p->num_sms,
                       st) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  rc = tcu_dft_exec_dir(p->cols1d, p->scratch, p->scratch, dir, st);
  if (rc != TCU_DFT_OK || keep_t) return rc;
  return launch_transpose((float2 *)out, p->scratch, p->batch, p->n2, p->n1, p->num_sms, st) ==
                 cudaSuccess
             ? TCU_DFT_OK
             : TCU_DFT_ERR_CUDA;
}

tcu_dft2_plan_s *make_dft2(int64_t n1, int64_t n2, int64_t batch, int32_t r,
                           int32_t precision, int &rc) {
  rc = TCU_DFT_OK;
  if (n1 < 1 || n2 < 1 || batch < 1 ||
      (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32 && !prec_bf16(precision))) {
    rc = TCU_DFT_ERR_INVALID;
    return nullptr;
  }
  int k1 = 0, k2 = 0;
  if ((r != 8 && r != 16 && r != 32) || !is_power_of(n1, r, k1) || !is_power_of(n2, r, k2) ||
      batch * n1 * n2 > (1ll << 40)) {
    rc = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  // each axis one warpgroup pass (a column item spans 128 r / n1 columns),
  // TF32 modes: the two-pass path; otherwise the general path
  if (prec_bf16(precision) || k1 > single_pass_stages(r) || k2 > single_pass_stages(r) ||
      n1 * n2 < 128ll * r)
    return make_dft2_general(n1, n2, batch, r, precision, rc);
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
    build_images(r, sign, n1 * n2, precision, img);
    rc = upload(&p->bimg[d], img);
    // hi and lo of this direction (the first two images)
    conv_img.insert(conv_img.end(), img.begin(), img.begin() + img.size() / 2);
    if (rc == TCU_DFT_OK) rc = upload(&c.tw_stage[d], stage_twiddles(r, c.s, sign));
    if (rc == TCU_DFT_OK) rc = upload(&w.tw_stage[d], stage_twiddles(r, w.s, sign));
  }
  if (rc == TCU_DFT_OK) rc = upload(&p->cimg, conv_img);
  if (rc == TCU_DFT_OK &&
      (dev_malloc((void **)&p->scratch, (size_t)(batch * n1 * n2) * sizeof(float2)) !=
           cudaSuccess ||
       dev_malloc((void **)&p->err, sizeof(int)) != cudaSuccess ||
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
// (128 r points): one warpgroup pass per axis where that suffices, else the
// general path up to 2^26 points per grid (8192^2); 0 if none.
long long grid_side(int r, long long need) {
  for (long long N = r; N * N <= (1ll << 26); N *= r)
    if (N >= need && N * N >= 128ll * r) return N;
  return 0;
}

// Tile side of a stencil plan: the smallest N = r^s with N >= 3k and
// N^2 >= 128 r (one warpgroup pass per axis); 0 if none.  Larger tiles give
// larger output blocks (fewer tile points) but were measured slower per
// point where they take three radix-8 stages per axis or radix-32 rows
// (4096^2 x 16 steps: 512^2 tiles 1.31 ms against 0.856 ms for 64^2).
long long stencil_tile(int r, long long k, long long side) {
  (void)side;
  return grid_side(r, 3 * k);
}

}  // namespace

extern "C" {

int64_t tcu_stencil_tiles(int64_t side, int32_t steps, int32_t sqrt_m, int64_t *tile,
                          int64_t *block) {
  if (side < 1 || steps < 1 || (sqrt_m != 8 && sqrt_m != 16 && sqrt_m != 32)) return 0;
  const long long N = stencil_tile(sqrt_m, steps, side);
  if (!N) return 0;
  const long long B = N - 2ll * steps, tpr = (side + B - 1) / B;
  if (tile) *tile = N;
  if (block) *block = B;
  return tpr * tpr;
}

tcu_dft2_plan_t tcu_dft2_plan(int64_t n1, int64_t n2, int64_t batch, int32_t sqrt_m,
                              int32_t precision) {
  int rc;
  arm_alloc_faults();
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
  if (p->general) {
    const NvtxRange range("tcu_dft2 (general)");
    rc = general_dft2(p, in, out, dir, false, st);
    return rc == TCU_DFT_OK && debug_exec() ? tcu_dft2_check(p, stream) : rc;
  }
  {
    const NvtxRange range("tcu_dft2");
    rc = run_dft2_pass(p, p->cols, di, (const float2 *)in, p->scratch, false, nullptr, st);
    if (rc == TCU_DFT_OK)
      rc = run_dft2_pass(p, p->rows, di, p->scratch, (float2 *)out, dir == TCU_DFT_INVERSE,
                         nullptr, st);
  }
  return rc == TCU_DFT_OK && debug_exec() ? tcu_dft2_check(p, stream) : rc;
}

int tcu_conv2_exec(tcu_dft2_plan_t p, const void *in, const void *spectrum, void *out,
                   void *stream) {
  if (!p || !spectrum || ((uintptr_t)spectrum & 15)) return TCU_DFT_ERR_INVALID;
  const size_t bytes = (size_t)(p->batch * p->n1 * p->n2) * sizeof(float2);
  int rc = check_buffers(in, out, bytes);
  if (rc != TCU_DFT_OK) return rc;
  cudaStream_t st = (cudaStream_t)stream;
  const NvtxRange range("tcu_conv2");
  if (p->general) {
    // forward rows and columns (left transposed in the scratch), times the
    // spectrum transposed, inverse columns, transpose back, inverse rows
    rc = general_dft2(p, in, out, TCU_DFT_FORWARD, true, st);
    if (rc != TCU_DFT_OK) return rc;
    if (launch_transpose(p->spec_t, (const float2 *)spectrum, 1, p->n1, p->n2, p->num_sms,
                         st) != cudaSuccess ||
        launch_spectrum_product(p->scratch, p->spec_t, p->batch, p->n1 * p->n2, p->num_sms,
                                st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    rc = tcu_dft_exec_dir(p->cols1d, p->scratch, p->scratch, TCU_DFT_INVERSE, st);
    if (rc != TCU_DFT_OK) return rc;
    if (launch_transpose((float2 *)out, p->scratch, p->batch, p->n2, p->n1, p->num_sms, st) !=
        cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    rc = tcu_dft_exec_dir(p->rows1d, out, out, TCU_DFT_INVERSE, st);
    return rc == TCU_DFT_OK && debug_exec() ? tcu_dft2_check(p, stream) : rc;
  }
  // columns: in -> scratch; rows forward, times the spectrum and inverse on
  // chip: scratch -> scratch (an item reads its rows before writing them);
  // inverse columns with 1/(n1 n2): scratch -> out
  rc = run_dft2_pass(p, p->cols, 0, (const float2 *)in, p->scratch, false, nullptr, st);
  if (rc != TCU_DFT_OK) return rc;
  GArgs g;
  memset(&g, 0, sizeof(g));
  g.p[0] = dft2_pass(p, p->rows, 0, p->scratch, p->scratch, false, (const float2 *)spectrum, 1);
  g.p[1].tw_stage = p->rows.tw_stage[1];
  g.bimg = p->cimg;
  g.err = p->err;
  cudaError_t e;
  if (p->r == 8) e = launch_rowconv_r8(p->precision, p->rows.s, g, p->num_sms, st);
  else if (p->r == 16) e = launch_rowconv_r16(p->precision, p->rows.s, g, p->num_sms, st);
  else e = launch_rowconv_r32(p->precision, p->rows.s, g, p->num_sms, st);
  if (e != cudaSuccess) return TCU_DFT_ERR_CUDA;
  rc = run_dft2_pass(p, p->cols, 1, p->scratch, (float2 *)out, true, nullptr, st);
  return rc == TCU_DFT_OK && debug_exec() ? tcu_dft2_check(p, stream) : rc;
}

int tcu_dft2_check(tcu_dft2_plan_t p, void *stream) {
  if (!p) return TCU_DFT_ERR_INVALID;
  if (p->general) {
    int rc = tcu_dft_check(p->rows1d, stream);
    if (rc == TCU_DFT_OK) rc = tcu_dft_check(p->cols1d, stream);
    if (rc != TCU_DFT_OK) return rc;
  }
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return TCU_DFT_ERR_CUDA;
  int flag = 0;
  if (cudaMemcpy(&flag, p->err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  if (flag) cudaMemset(p->err, 0, sizeof(int));
  return word_status(flag);
}

int tcu_dft2_destroy(tcu_dft2_plan_t p) {
  free_dft2(p);
  return TCU_DFT_OK;
}

tcu_stencil_plan_t tcu_stencil_plan(int64_t side, int32_t steps, int32_t sqrt_m,
                                    int32_t precision) {
  g_last_error = TCU_DFT_OK;
  arm_alloc_faults();
  if (side < 1 || steps < 1 ||
      (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32 && !prec_bf16(precision))) {
    g_last_error = TCU_DFT_ERR_INVALID;
    return nullptr;
  }
  const long long N =
      (sqrt_m == 8 || sqrt_m == 16 || sqrt_m == 32) ? stencil_tile(sqrt_m, steps, side) : 0;
  const long long Nw = N ? grid_side(sqrt_m, 2ll * steps + 1) : 0;
  if (!N || !Nw) {
    g_last_error = TCU_DFT_ERR_UNSUPPORTED;
    return nullptr;
  }
  // output blocks of B = N - 2k >= k points a side: the (B + 2k)^2 input
  // window of a block fits the N x N tile without wrapping (Lemma 1 is
  // B = k); the last blocks of a row may be cut; N from stencil_tile
  const int B = (int)(N - 2ll * steps);
  const long long tpr = (side + B - 1) / B;
  tcu_stencil_plan_s *p = new tcu_stencil_plan_s();
  memset(p, 0, sizeof(*p));
  p->side = side;
  p->k = steps;
  p->r = sqrt_m;
  p->precision = precision;
  p->N = N;
  p->Nw = Nw;
  p->B = B;
  p->tiles = tpr * tpr;
  int rc = TCU_DFT_OK;
  p->conv = make_dft2(N, N, p->tiles, sqrt_m, precision, rc);
  if (rc == TCU_DFT_OK) p->wconv = make_dft2(N, N, 1, sqrt_m, precision, rc);
  if (rc == TCU_DFT_OK) p->wpow = make_dft2(Nw, Nw, 1, sqrt_m, precision, rc);
  if (rc == TCU_DFT_OK) {
    p->num_sms = p->conv->num_sms;
    if (dev_malloc((void **)&p->tile_buf, (size_t)(p->tiles * N * N) * sizeof(float2)) !=
            cudaSuccess ||
        dev_malloc((void **)&p->wgrid, (size_t)(Nw * Nw) * sizeof(float2)) != cudaSuccess ||
        dev_malloc((void **)&p->wker, (size_t)(N * N) * sizeof(float2)) != cudaSuccess) {
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
  const NvtxRange range("tcu_stencil");
  // W (Lemma 2), the kernel W' and its spectrum
  int rc = stencil_weight_grid(p, w3x3, st);
  if (rc != TCU_DFT_OK) return rc;
  if (launch_place_kernel(p->wker, p->N, p->wgrid, p->Nw, p->k, p->num_sms, st) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  rc = tcu_dft2_exec(p->wconv, p->wker, p->wker, TCU_DFT_FORWARD, st);
  if (rc != TCU_DFT_OK) return rc;
  // Lemma 1: every block's input window as one batch of tiles, circular
  // convolution, the B x B centres
  if (launch_gather_tiles(p->tile_buf, A, p->side, p->k, p->N, p->B, p->num_sms, st) !=
      cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  rc = tcu_conv2_exec(p->conv, p->tile_buf, p->wker, p->tile_buf, st);
  if (rc != TCU_DFT_OK) return rc;
  if (launch_extract_tiles(Ak, p->tile_buf, p->side, p->k, p->N, p->B, p->num_sms, st) !=
      cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  return debug_exec() ? tcu_stencil_check(p, stream) : TCU_DFT_OK;
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
