// launch.h -- host-side entry points of the kernels (one translation unit
// per radix defines them; see launch_impl.cuh).
#pragma once
#include <cuda_runtime.h>

#include "group_kernel.cuh"
#include "tile_kernel.cuh"

namespace tcu {

// One warpgroup pass: radix r, s stages, the other pass has so stages
// (0 for a single pass), role kSingle / kFirst / kSecond.
cudaError_t launch_pass(int r, int prec, int s, int so, int role, const GArgs &a,
                        int num_sms, cudaStream_t st);
// Both passes fused in one launch (s1, s2 >= 2).
cudaError_t launch_fused(int r, int prec, int s1, int s2, const GArgs &a, int num_sms,
                         cudaStream_t st);
// One tile-kernel pass.
cudaError_t launch_tile(int r, int prec, const PassArgs &a, long long grid,
                        cudaStream_t st);

bool pass_supported(int r, int s, int so, int role);
bool fused_supported(int r, int s1, int s2);

// per-radix definitions
cudaError_t launch_pass_r8(int prec, int s, int so, int role, const GArgs &a, int num_sms,
                           cudaStream_t st);
cudaError_t launch_pass_r16(int prec, int s, int so, int role, const GArgs &a, int num_sms,
                            cudaStream_t st);
cudaError_t launch_pass_r32(int prec, int s, int so, int role, const GArgs &a, int num_sms,
                            cudaStream_t st);
cudaError_t launch_fused_r8(int prec, int s1, int s2, const GArgs &a, int num_sms,
                            cudaStream_t st);
cudaError_t launch_fused_r16(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st);
cudaError_t launch_fused_r32(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st);
cudaError_t launch_tile_r8(int prec, const PassArgs &a, long long grid, cudaStream_t st);
cudaError_t launch_tile_r16(int prec, const PassArgs &a, long long grid, cudaStream_t st);
cudaError_t launch_tile_r32(int prec, const PassArgs &a, long long grid, cudaStream_t st);

}  // namespace tcu
