// noalloc.cu -- tcu_dft_exec_noalloc: the transform without a plan and
// without any device allocation (its working memory is fixed arrays here).
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

namespace {

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

int tcu_dft_exec_noalloc(int64_t n, int64_t batch, int32_t sqrt_m, int32_t precision,
                         const void *in, void *out, int dir, void *stream) {
  // ---- arguments (no CUDA call before they are known to be good)
  if (n < 1 || batch < 1 ||
      (precision != TCU_DFT_TF32 && precision != TCU_DFT_3XTF32 && !prec_bf16(precision)) ||
      !in || !out || (dir != TCU_DFT_FORWARD && dir != TCU_DFT_INVERSE))
    return TCU_DFT_ERR_INVALID;
  if (((uintptr_t)in & 15) || ((uintptr_t)out & 15)) return TCU_DFT_ERR_INVALID;
  if (prec_bf16(precision)) return TCU_DFT_ERR_UNSUPPORTED;
  if (sqrt_m != 8 && sqrt_m != 16 && sqrt_m != 32) return TCU_DFT_ERR_UNSUPPORTED;
  const int r = sqrt_m, log2r = ilog2(r);
  int k = 0;
  long long m = 1;
  while (m < n) {
    m *= r;
    ++k;
  }
  // n = r^k with k >= 1, as tcu_dft_plan requires
  if (m != n || k < 1) return TCU_DFT_ERR_UNSUPPORTED;
  int st[kMaxPasses] = {0, 0, 0};
  const int npasses = plan_stages(r, k, st);
  if (npasses == 0 || npasses > 2 || n > kNaMaxN) return TCU_DFT_ERR_TOO_LARGE;
  if (npasses == 2 && batch * n > kNaMaxPoints) return TCU_DFT_ERR_TOO_LARGE;
  // in == out is allowed; a partial overlap is not
  if (in != out && overlaps(in, out, (size_t)batch * n * sizeof(float2)))
    return TCU_DFT_ERR_INVALID;
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

  // ---- tables for this (n, r): table A of the strided pass at the start of
  // the direction's twiddle array, B (more than 256 columns) after it
  if (npasses == 2) {
    const long long n2 = 1ll << p.pass[0].lo, VL = n2 > 256 ? 256 : n2;
    for (int d = 0; d < 2; ++d) {
      p.pass[0].tw_a[d] = D.tw_out + (size_t)d * kNaMaxN;
      if (n2 > VL) p.pass[0].tw_b[d] = p.pass[0].tw_a[d] + (1ll << p.pass[0].log2L) * VL;
    }
  }
  // built and uploaded only when (n, r) changes: a call that changes them
  // copies from host memory on `stream` and so must not be captured
  if (D.n != n || D.r != r) {
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(stream_, &cap) != cudaSuccess) {
      cudaGetLastError();
      return TCU_DFT_ERR_CUDA;
    }
    if (cap != cudaStreamCaptureStatusNone) return TCU_DFT_ERR_INVALID;
    DirTables t[2];
    for (int d = 0; d < 2; ++d) {
      dir_tables(&p, d, t[d]);
      for (int pi = 0; pi < npasses; ++pi)
        if (t[d].stage[pi].size() > (size_t)kNaStageTw) return TCU_DFT_ERR_TOO_LARGE;
    }
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
  const int rc = exec_impl(&p, in, out, dir, stream, nullptr);
  if (rc != TCU_DFT_OK || !debug_exec()) return rc;
  // TCU_DFT_DEBUG=1: wait for the launches and report the error word (a
  // device-side wait timeout) as tcu_dft_check does for plans
  int flag = 0;
  if (cudaStreamSynchronize(stream_) != cudaSuccess ||
      cudaMemcpy(&flag, D.err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  return word_status(flag);
}

}  // extern "C"
