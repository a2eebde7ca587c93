// host_plan.h -- internal declarations shared by the host side of the
// library: pass plans, table builders, launches and the 1-D plan itself.
// Not part of the C ABI (include/tcu_dft.h).
#pragma once
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "../../include/tcu_dft.h"
#include "launch.h"

namespace tcu {
namespace host {

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
  int qrt;          // kSecondQ: the factor q of n = q r^s (runtime prefix count)
  int tw;           // warpgroups per item (teams for the 3-stage radix-8 passes)
};

// Status of the last plan call on this thread (tcu_dft_last_error).
extern thread_local int g_last_error;

// ---- tables, tensor maps and small helpers (host_tables.cu)
int ilog2(long long v);
int dir_index(int dir);
// cuTensorMapEncodeTiled from the driver, through the runtime (no -lcuda).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder();
// TMA map of a [depth][rows][cols] array of complex64 (cols contiguous, row
// pitch cols, plane pitch plane_elems), seen as fp32 pairs; boxes of
// box_cols complex x box_rows rows x 1 plane.
bool encode_map(CUtensorMap *m, const void *base, long long cols, long long rows,
                long long depth, long long plane_elems, int box_cols, int box_rows);
// Round an fp32 value to TF32 (10 explicit mantissa bits), nearest, ties away
// from zero -- the same rule as PTX cvt.rna.tf32.f32.
float host_tf32_rna(float x);
// exp(sign * 2 pi i * m / period) with m reduced mod period, fp64 -> fp32
float2 root(long long m, long long period, int sign);
// Round an fp32 value to bf16 (8 significant bits), nearest-even; the bits.
uint16_t host_bf16_rne(float x);
float host_bf16_value(uint16_t h);
bool prec_bf16(int precision);
// B operand images of the real 2r x 2r block form of F_r for one direction,
// in the canonical no-swizzle K-major layout the MMA reads: hi, lo, and the
// same two scaled by 2^-log2n (exact: a power of two) for the inverse's last
// stage, which folds the 1/n normalisation into the product.  Core matrices
// are 8 rows x 16 bytes: 4 fp32 (TF32 modes) or 8 bf16 (BF16 modes) of K;
// the four images sit at multiples of their size (16 r^2 or 8 r^2 bytes) in
// a buffer of 64 r^2 bytes.
void build_images(int r, int sign, long long n, int precision, std::vector<float> &out);
// Stage twiddles of a warpgroup pass: for t = 1 .. s-1 a block [j][lo],
// j < r, lo < r^(s-t), holding w_L^{j * lo * r^(t-1)}.
std::vector<float2> stage_twiddles(int r, int s, int sign);
int stage_mode(const int modes[3], int t, int S);
// Shared-memory wavefronts per warp-wide 8-byte access of the warpgroup
// kernel's transposes (1.0 = conflict free), for swizzle table `tab`:
// phys(P) = P ^ ((tab[ul & 15] ^ (P >> 4)) & 15).
double swizzle_cost(int r, int S, const int modes[3], unsigned long long tab, int team);
unsigned long long choose_swizzle(int r, int S, const int modes[3], int team);
// Inter-pass twiddles of a strided pass: w_M^{k v}, k < L, v < n2, M = L n2;
// A[k][vl] for vl < min(n2, 256) and, if n2 > 256, B[vh][k] = w_M^{k vh 256}.
void pass_twiddles(long long L, long long n2, int sign, std::vector<float2> &A,
                   std::vector<float2> &B);
// TMA map of table A of a strided pass (boxes of GG columns x L rows).
bool twiddle_map(CUtensorMap *m, const float2 *A, int r, const PassPlan &pp);
// TMA map of a strided pass's input: sequences of M = L n2 points, batch *
// r^sp of them, seen as [sequence][row a][column v].
bool input_map(CUtensorMap *m, const void *in, const tcu_dft_plan_s *p, const PassPlan &pp,
               long long batch);
bool overlaps(const void *a, const void *b, size_t bytes);

// Tables of a plan for one direction d: F images, stage twiddles and the
// inter-pass twiddles, as host vectors (uploaded by the caller).
struct DirTables {
  std::vector<float> img;
  std::vector<float2> stage[kMaxPasses], A[kMaxPasses], B[kMaxPasses];
};

// Device allocation of the plans (cudaMalloc), with a host-side fault
// injector for the tests of the plans' error paths: with TCU_DFT_FAIL_ALLOC=k
// (k >= 1) in the environment, the k-th allocation after arm_alloc_faults()
// on this thread fails as if the device were out of memory.  No GPU fault is
// involved: the allocation is simply not made.
void arm_alloc_faults();
cudaError_t dev_malloc(void **ptr, size_t bytes);

// TCU_DFT_DEBUG=1 in the environment: every exec call synchronises its
// stream and returns the plan's error word (as tcu_dft_check) instead of
// returning as soon as the launches are queued.
bool debug_exec();

// An NVTX range over the launches of one pass (host side; seen by nsys and
// by ncu's --nvtx filters, free when no tool is attached).
struct NvtxRange {
  explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange &) = delete;
  NvtxRange &operator=(const NvtxRange &) = delete;
};

// Status recorded in a plan's error word (0: none): the kernels write
// TCU_DFT_ERR_TIMEOUT, the bounds-checked build also TCU_DFT_ERR_BOUNDS.
int word_status(int flag);

template <typename T>
int upload(T **dst, const std::vector<T> &src) {
  if (dev_malloc((void **)dst, src.size() * sizeof(T)) != cudaSuccess) {
    cudaGetLastError();
    *dst = nullptr;
    return TCU_DFT_ERR_OOM;
  }
  if (cudaMemcpy(*dst, src.data(), src.size() * sizeof(T), cudaMemcpyHostToDevice) !=
      cudaSuccess)
    return TCU_DFT_ERR_CUDA;
  return TCU_DFT_OK;
}

}  // namespace host
}  // namespace tcu

struct tcu_dft_plan_s {
  long long n, batch;
  int r, log2r, k, precision;
  int npasses;
  int num_sms;
  tcu::host::PassPlan pass[tcu::host::kMaxPasses];
  float *bimg[2];          // [dir index] hi | lo | scaled hi | scaled lo images
  float2 *scratch[2];      // intermediates (or the fused ring in scratch[0])
  // fused two-pass schedule
  bool fused;
  // one HBM pass on cluster pairs (scratch[0]: two slots per cluster)
  bool pair;
  int pair_clusters;
  int log2C, nchunks, lag, ring_chunks;
  int items1_per_tf, log2_items_per_chunk;
  int *counters;
  size_t counter_bytes;
  int *err;
  int device;
  // host-buffer path: copy streams and per-chunk events (created by the plan)
  cudaStream_t copy_in, copy_out;
  cudaEvent_t ev_start, ev_in[tcu::host::kHostChunks], ev_done[tcu::host::kHostChunks],
      ev_out[tcu::host::kHostChunks];
  bool has_copy_streams;
};

namespace tcu {
namespace host {

// ---- plans and launches (tcu_dft.cu)
// Stages per pass.  Passes hold at most two stages (three for r = 8, whose
// 3-stage sub-transforms of 512 points still fit a 128-row item); up to
// three passes; the earlier passes take the smaller shares, so the strided
// passes have shorter sub-transforms, more adjacent columns per item and
// wider TMA rows.  Returns the number of passes, 0 if n is too long.
int plan_stages(int r, int k, int st[kMaxPasses]);
// Mixed radix n = q r^k (the base case of the recursion is a DFT of size
// q): a CUDA-core q-point first pass, then the r^k-point transforms of its q
// rows in tensor-core passes.  q < r a power of two: one or two passes
// (stage split as plan_stages; k = 2..4 for r = 8 and 16, k = 2..3 for
// r = 32).  Any other q = 2 .. 16 (odd factors): one pass with a runtime
// q, k = 1..3 for r = 8, k = 1..2 for r = 16 and 32.  Returns the number of
// passes (0: not such an n) and fills the passes.
int plan_mixed(int r, long long n, long long batch, PassPlan pass[kMaxPasses]);
// Warpgroups per item of pass pp: 4 for the 3-stage radix-8 passes of
// two-pass transforms (an item of 512 rows holds 8 sub-transforms of 512
// points, so the strided side moves 64-byte runs), else 1.
int team_size(int r, int npasses, const PassPlan &pp);
// Role, neighbouring stage counts, size and row maps of pass `pi`.
void pass_geometry(PassPlan &pp, int pi, int P, const int st[kMaxPasses], int k, int r,
                   long long n, long long batch);
void free_plan(tcu_dft_plan_s *p);
// ---------------------------------------------------------------- launches
cudaError_t pass_dispatch(int r, int prec, const PassPlan &pp, const GArgs &a, int num_sms,
                          cudaStream_t st, bool team_plan = false);
cudaError_t fused_dispatch(int r, int prec, int s1, int s2, const GArgs &a, int num_sms,
                           cudaStream_t st);
// Warpgroup-kernel description of pass `pi` between buffers `in` and `out`.
PRun group_pass(const tcu_dft_plan_s *p, int pi, int di, const float2 *in, float2 *out,
                long long in_bmask, long long out_bmask, bool inverse, long long batch);
void dir_tables(const tcu_dft_plan_s *p, int d, DirTables &t);

// The transform of transforms [b0, b0 + count) of the plan's batch (in and
// out point at transform b0; count < 0: the whole batch).  The intermediates
// of that range sit at the same offset in the plan's scratch, so disjoint
// ranges may run concurrently on different streams (not fused plans).
int exec_impl(tcu_dft_plan_t p, const void *in, void *out, int dir,
                     void *stream, void *const *events, long long queue_start = 0,
                     long long b0 = 0, long long count = -1);

}  // namespace host
}  // namespace tcu
