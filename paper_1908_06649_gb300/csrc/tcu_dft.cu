// tcu_dft.cu -- batched complex DFT on GB300 (sm_103a) tensor cores: the
// 1-D plan, pass scheduling and the 1-D half of the C ABI declared in
// include/tcu_dft.h.  The plan's tables and tensor maps are built in
// host_tables.cu, the allocation-free entry point is noalloc.cu, the 2-D
// transforms, convolutions and stencils are grid_plan.cu.
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

#include "host_plan.h"

using namespace tcu;
using namespace tcu::host;

#if defined(__CUDA_ARCH__) && (__CUDA_ARCH__ < 1000)
#error "tcu_dft targets sm_103a (tcgen05); compile with -gencode arch=compute_103a,code=sm_103a"
#endif

namespace tcu {
namespace host {

thread_local int g_last_error = TCU_DFT_OK;

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
// n = q r^k with q = 2 .. 16 not a power of two: the q-point pass, then one
// tensor-core pass over the q rows (role kSecondQ, q at run time).
int plan_mixed_q(int r, long long n, long long batch, PassPlan pass[kMaxPasses]) {
  const int log2r = ilog2(r);
  const int kmax = r == 8 ? 3 : 2;
  int k = 0;
  long long rest = n;
  while (rest % r == 0 && k < kmax) {
    rest /= r;
    ++k;
  }
  // the factor left must be a q the CUDA-core pass has, and r^k must hold
  // all of n's powers of r that fit one pass
  if (k < 1 || rest < 2 || rest > 16 || (rest & (rest - 1)) == 0) return 0;
  if (rest % r == 0) return 0;
  const int q = (int)rest;
  PassPlan &p0 = pass[0];
  p0.q = q;
  p0.s = 1;
  p0.role = kFirst;
  p0.log2L = 0;  // not a power of two: the q-pass uses q itself
  p0.lo = k * log2r;
  p0.lp = 0;
  p0.U = batch * (n / q);
  for (int d = 0; d < 2; ++d)
    for (int m = 0; m < 16; ++m) p0.roots[d].w[m] = root(m % q, q, d == 0 ? -1 : 1);
  PassPlan &pp = pass[1];
  pp.mixed = true;
  pp.s = k;
  pp.log2L = log2r * k;
  pp.last = true;
  pp.role = kSecondQ;
  pp.lo = 0;
  pp.lp = 0;
  pp.qrt = q;
  pp.U = batch * q;
  pp.modes[0] = kQF;
  pp.modes[1] = kUF;
  pp.modes[2] = kUF;
  pp.tw = 1;
  pp.swz_tab = choose_swizzle(r, pp.s, pp.modes, 1);
  return 2;
}

int plan_mixed(int r, long long n, long long batch, PassPlan pass[kMaxPasses]) {
  const int log2r = ilog2(r);
  if (n < 1) return 0;
  if (n & (n - 1)) return plan_mixed_q(r, n, batch, pass);
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
                          cudaStream_t st, bool team_plan) {
  if (pp.mixed) {
    if (r == 8) return launch_pass_mixed_r8(prec, pp.s, pp.lo, pp.role, pp.lp, a, num_sms, st);
    if (r == 16) return launch_pass_mixed_r16(prec, pp.s, pp.lo, pp.role, pp.lp, a, num_sms, st);
    return launch_pass_mixed_r32(prec, pp.s, pp.lo, pp.role, pp.lp, a, num_sms, st);
  }
  if (prec_bf16(prec)) {
    if (r == 8) return launch_pass_bf16_r8(prec, pp.s, pp.lo, pp.role, pp.lp, pp.tw, a, num_sms, st);
    if (r == 16)
      return launch_pass_bf16_r16(prec, pp.s, pp.lo, pp.role, pp.lp, pp.tw, a, num_sms, st);
    return launch_pass_bf16_r32(prec, pp.s, pp.lo, pp.role, pp.lp, pp.tw, a, num_sms, st);
  }
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
  // every second pass runs its items last to first: it starts on what the
  // pass before wrote last, still in L2 (measured 0.5-2.5 % per pass; not on
  // team passes, where it measured 1.5 % slower)
  g.reverse = (pi & 1) && pp.tw == 1;
  g.q = pp.qrt;
  // the inverse's last stage uses the F images scaled by 1/n
  g.last_img = (pp.last && inverse) ? 2 * (prec_bf16(p->precision) ? 8 : 16) * p->r * p->r : 0;
  return g;
}

void dir_tables(const tcu_dft_plan_s *p, int d, DirTables &t) {
  const int sign = d == 0 ? -1 : 1;
  build_images(p->r, sign, p->n, p->precision, t.img);
  for (int pi = 0; pi < p->npasses; ++pi) {
    const PassPlan &pp = p->pass[pi];
    t.stage[pi] = stage_twiddles(p->r, pp.q ? 1 : pp.s, sign);
    // the q-point pass has L = q rows (any q); a tensor-core pass L = r^s
    if (pp.role == kFirst)
      pass_twiddles(pp.q ? pp.q : (1ll << pp.log2L), 1ll << pp.lo, sign, t.A[pi], t.B[pi]);
  }
}

int exec_impl(tcu_dft_plan_t p, const void *in, void *out, int dir,
                     void *stream, void *const *events, long long queue_start,
                     long long b0, long long count) {
  if (!p || !in || !out || (dir != TCU_DFT_FORWARD && dir != TCU_DFT_INVERSE))
    return TCU_DFT_ERR_INVALID;
  if (((uintptr_t)in & 15) || ((uintptr_t)out & 15)) return TCU_DFT_ERR_INVALID;
  if (count < 0) count = p->batch;
  if (b0 < 0 || b0 + count > p->batch || ((p->fused || p->pair) && count != p->batch))
    return TCU_DFT_ERR_INVALID;
  const size_t bytes = (size_t)count * p->n * sizeof(float2);
  if (in != out && overlaps(in, out, bytes)) return TCU_DFT_ERR_INVALID;
  cudaStream_t st = (cudaStream_t)stream;
  const int di = dir_index(dir);
  const bool inverse = dir == TCU_DFT_INVERSE;
  if (p->pair) {
    // both passes in one launch; cluster c's intermediates in slots 2c, 2c+1
    GArgs g;
    memset(&g, 0, sizeof(g));
    g.p[0] = group_pass(p, 0, di, (const float2 *)in, p->scratch[0], -1, 1, inverse, p->batch);
    g.p[1] = group_pass(p, 1, di, p->scratch[0], (float2 *)out, 1, -1, inverse, p->batch);
    if (!input_map(&g.tm_in, in, p, p->pass[0], p->batch)) return TCU_DFT_ERR_CUDA;
    g.tm_tw = p->pass[0].tw_map[di];
    g.bimg = p->bimg[di];
    g.err = p->err;
    g.batch = p->batch;
    g.items1_per_tf = p->items1_per_tf;
    if (events && cudaEventRecord((cudaEvent_t)events[0], st) != cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    const NvtxRange range("tcu_dft one pass (cluster pairs)");
    if (launch_pair_r16(p->precision, p->pass[0].s, p->pass[1].s, g, p->pair_clusters, st) !=
        cudaSuccess)
      return TCU_DFT_ERR_CUDA;
    if (events && (cudaEventRecord((cudaEvent_t)events[1], st) != cudaSuccess ||
                   cudaEventRecord((cudaEvent_t)events[2], st) != cudaSuccess))
      return TCU_DFT_ERR_CUDA;
    return TCU_DFT_OK;
  }
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
    const NvtxRange range("tcu_dft fused passes");
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
  static const char *const kRange[kMaxPasses] = {"tcu_dft pass 1", "tcu_dft pass 2",
                                                 "tcu_dft pass 3"};
  for (int pi = 0; pi < p->npasses; ++pi) {
    const NvtxRange range(kRange[pi]);
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

}  // namespace host
}  // namespace tcu

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
    case TCU_DFT_ERR_BOUNDS: return "index out of range (checked build)";
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
  arm_alloc_faults();
  if (n < 1 || batch < 1 ||
      (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32 && !prec_bf16(precision)) ||
      (flags & ~(uint32_t)(TCU_DFT_PLAN_NO_FUSE | TCU_DFT_PLAN_FUSE | TCU_DFT_PLAN_ONE_PASS)) ||
      ((flags & TCU_DFT_PLAN_NO_FUSE) && (flags & (TCU_DFT_PLAN_FUSE | TCU_DFT_PLAN_ONE_PASS))) ||
      ((flags & TCU_DFT_PLAN_FUSE) && (flags & TCU_DFT_PLAN_ONE_PASS))) {
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
  // the BF16 modes are instantiated for n = r^k (no mixed radix)
  if (npasses == 0 || (long long)batch * n > (1ll << 40) ||
      (prec_bf16(precision) && is_mixed)) {
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
    if (dev_malloc((void **)&p->err, sizeof(int)) != cudaSuccess ||
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
    // one HBM pass on cluster pairs: radix 16, 2 + 2 stages (n = 16^4)
    p->pair = !is_mixed && !prec_bf16(precision) && r == 16 && npasses == 2 && p1.s == 2 &&
              p2.s == 2 && (flags & TCU_DFT_PLAN_ONE_PASS) && p->num_sms >= 2;
    long long scratch_tf = batch;
    if (p->pair) {
      const long long gg1 = (128ll * r) >> p1.log2L;
      p->items1_per_tf = (int)((1ll << p2.log2L) / gg1);
      // one cluster per two SMs, no more than there are pairs of transforms;
      // two slots of scratch per cluster
      const long long pairs = (batch + 1) / 2;
      p->pair_clusters = (int)(pairs < p->num_sms / 2 ? pairs : p->num_sms / 2);
      scratch_tf = 2ll * p->pair_clusters;
    }
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
      if (rc == TCU_DFT_OK && dev_malloc((void **)&p->counters, p->counter_bytes) != cudaSuccess) {
        cudaGetLastError();
        rc = TCU_DFT_ERR_OOM;
      }
    }
    for (int i = 0; i < npasses - 1 && rc == TCU_DFT_OK; ++i)
      if (dev_malloc((void **)&p->scratch[i], (size_t)scratch_tf * n * sizeof(float2)) !=
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


int tcu_dft_exec_dir(tcu_dft_plan_t p, const void *in, void *out, int dir,
                     void *stream) {
  const int rc = exec_impl(p, in, out, dir, stream, nullptr);
  return rc == TCU_DFT_OK && debug_exec() ? tcu_dft_check(p, stream) : rc;
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
  const int rc = exec_impl(p, in, out, dir, stream, events);
  return rc == TCU_DFT_OK && debug_exec() ? tcu_dft_check(p, stream) : rc;
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
  if (p->fused || p->pair || !p->has_copy_streams || p->batch < 2) {
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
  if (flag) cudaMemset(p->err, 0, sizeof(int));
  return word_status(flag);
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

int tcu_dft_is_fused(tcu_dft_plan_t p) { return p ? ((p->fused || p->pair) ? 1 : 0) : -1; }

int tcu_dft_pass_stages(tcu_dft_plan_t p, int i) {
  if (!p || i < 0 || i >= p->npasses) return -1;
  return p->pass[i].s;
}

}  // extern "C"
