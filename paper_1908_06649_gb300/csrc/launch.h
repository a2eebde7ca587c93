// launch.h -- host-side entry points of the kernels (one translation unit
// per radix defines them; see launch_impl.cuh).
#pragma once
#include <cuda_runtime.h>

#include "group_kernel.cuh"

namespace tcu {

// One warpgroup pass of radix 8, 16 or 32: s stages, role kSingle / kFirst /
// kSecond; so = stages after a kFirst pass or before a kSecond pass; sp =
// stages before a kFirst pass.  cudaErrorInvalidValue for a combination that
// is not instantiated.
cudaError_t launch_pass_r8(int prec, int s, int so, int role, int sp, const GArgs &a,
                           int num_sms, cudaStream_t st);
cudaError_t launch_pass_r16(int prec, int s, int so, int role, int sp, const GArgs &a,
                            int num_sms, cudaStream_t st);
cudaError_t launch_pass_r32(int prec, int s, int so, int role, int sp, const GArgs &a,
                            int num_sms, cudaStream_t st);
// Both passes of a two-pass transform fused in one launch (s1, s2 >= 2).
cudaError_t launch_fused_r8(int prec, int s1, int s2, const GArgs &a, int num_sms,
                            cudaStream_t st);
cudaError_t launch_fused_r16(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st);
cudaError_t launch_fused_r32(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st);

}  // namespace tcu
