// launch.h -- host-side entry points of the kernels (one translation unit
// per radix defines them; see launch_impl.cuh).
#pragma once
#include <cuda_runtime.h>

#include "group_kernel.cuh"

namespace tcu {

// One warpgroup pass of radix 8, 16 or 32: s stages, role kSingle / kFirst /
// kSecond / kCols; lo = log2 of the columns of a strided pass or of the
// points before a last pass; lp = log2 of the prefix count of a strided pass.
// cudaErrorInvalidValue for a combination that is not instantiated.
cudaError_t launch_pass_r8(int prec, int s, int lo, int role, int lp, const GArgs &a,
                           int num_sms, cudaStream_t st);
cudaError_t launch_pass_r16(int prec, int s, int lo, int role, int lp, const GArgs &a,
                            int num_sms, cudaStream_t st);
cudaError_t launch_pass_r32(int prec, int s, int lo, int role, int lp, const GArgs &a,
                            int num_sms, cudaStream_t st);
// The row pass of a circular 2-D convolution: each row transformed,
// multiplied by the spectrum and transformed back on chip (s stages).
cudaError_t launch_rowconv_r8(int prec, int s, const GArgs &a, int num_sms, cudaStream_t st);
cudaError_t launch_rowconv_r16(int prec, int s, const GArgs &a, int num_sms, cudaStream_t st);
cudaError_t launch_rowconv_r32(int prec, int s, const GArgs &a, int num_sms, cudaStream_t st);
// Radix-8 passes whose items are teams of tw warpgroups (kernels_r8.cu).
cudaError_t launch_team_r8(int prec, int s, int lo, int role, int lp, int tw, const GArgs &a,
                           int num_sms, cudaStream_t st);
// Radix-16 team passes (kernels_r16.cu).
cudaError_t launch_team_r16(int prec, int s, int lo, int role, int lp, int tw, const GArgs &a,
                            int num_sms, cudaStream_t st);
// Both passes of a two-pass transform in one launch on clusters of two CTAs,
// each cluster's intermediate in two L2-resident slots (radix 16, 2 + 2).
cudaError_t launch_pair_r16(int prec, int s1, int s2, const GArgs &a, int clusters,
                            cudaStream_t st);
// Both passes of a two-pass transform fused in one launch (s1, s2 >= 2).
cudaError_t launch_fused_r8(int prec, int s1, int s2, const GArgs &a, int num_sms,
                            cudaStream_t st);
cudaError_t launch_fused_r16(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st);
cudaError_t launch_fused_r32(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st);

// Element-wise steps of the stencil path (grid_kernels.cu).
struct Stencil3 {
  float w[9];  // w[(a + 1) * 3 + (b + 1)], a, b in {-1, 0, 1}
};
cudaError_t launch_place_poly(float2 *g, long long Nw, const Stencil3 &w, int num_sms,
                              cudaStream_t st);
cudaError_t launch_cpow(float2 *g, long long count, int k, int num_sms, cudaStream_t st);
cudaError_t launch_extract_weights(float *W, const float2 *g, long long Nw, int k,
                                   int num_sms, cudaStream_t st);
cudaError_t launch_place_kernel(float2 *w, long long N, const float2 *g, long long Nw, int k,
                                int num_sms, cudaStream_t st);
cudaError_t launch_gather_tiles(float2 *tiles, const float *A, long long side, int k,
                                long long N, int B, int num_sms, cudaStream_t st);
cudaError_t launch_extract_tiles(float *Ak, const float2 *tiles, long long side, int k,
                                 long long N, int B, int num_sms, cudaStream_t st);

// 2-D transforms whose axes need several passes (grid_kernels.cu): the
// transpose of every n1 x n2 array of a batch (out[b][j][i] = in[b][i][j]),
// and the pointwise product of every array with one spectrum.
cudaError_t launch_transpose(float2 *out, const float2 *in, long long batch, long long n1,
                             long long n2, int num_sms, cudaStream_t st);
cudaError_t launch_spectrum_product(float2 *x, const float2 *spec, long long batch,
                                    long long n, int num_sms, cudaStream_t st);

// The q-point first pass of a mixed-radix transform (grid_kernels.cu).
struct RootsQ {
  float2 w[16];  // w_q^m, m < q, of the direction
};
cudaError_t launch_radix_q(int q, const float2 *x, float2 *out, long long batch, int log2n2,
                           const float2 *twA, const float2 *twB, const RootsQ &roots,
                           int num_sms, cudaStream_t st);
// BF16-mode (precision 4, 5) passes of n = r^k (kernels_bf16_r{8,16,32}.cu).
cudaError_t launch_pass_bf16_r8(int prec, int s, int lo, int role, int lp, int tw,
                                const GArgs &a, int num_sms, cudaStream_t st);
cudaError_t launch_pass_bf16_r32(int prec, int s, int lo, int role, int lp, int tw,
                                 const GArgs &a, int num_sms, cudaStream_t st);
cudaError_t launch_pass_bf16_r16(int prec, int s, int lo, int role, int lp, int tw,
                                 const GArgs &a, int num_sms, cudaStream_t st);
// Mixed-radix warpgroup passes (kernels_mixed_r*.cu): same arguments as
// launch_pass_r*.
cudaError_t launch_pass_mixed_r8(int prec, int s, int lo, int role, int lp, const GArgs &a,
                                 int num_sms, cudaStream_t st);
cudaError_t launch_pass_mixed_r16(int prec, int s, int lo, int role, int lp, const GArgs &a,
                                  int num_sms, cudaStream_t st);
cudaError_t launch_pass_mixed_r32(int prec, int s, int lo, int role, int lp, const GArgs &a,
                                  int num_sms, cudaStream_t st);

}  // namespace tcu
