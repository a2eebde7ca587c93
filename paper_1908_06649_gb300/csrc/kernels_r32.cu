// kernels_r32.cu -- radix-32 kernel instantiations (sqrt(m) = 32).
#include "launch_impl.cuh"

namespace tcu {

cudaError_t launch_pass_r32(int prec, int s, int so, int role, const GArgs &a, int num_sms,
                            cudaStream_t st) {
  constexpr int R = 32;
  TCU_PASS_CASE(1, 0, kSingle)
  TCU_PASS_CASE(2, 0, kSingle)
  TCU_PASS_CASE(1, 2, kFirst)   // n = 32^3
  TCU_PASS_CASE(2, 1, kSecond)
  TCU_PASS_CASE(2, 1, kFirst)
  TCU_PASS_CASE(1, 2, kSecond)
  TCU_PASS_CASE(2, 2, kFirst)   // n = 32^4
  TCU_PASS_CASE(2, 2, kSecond)
  return cudaErrorInvalidValue;
}

cudaError_t launch_fused_r32(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st) {
  constexpr int R = 32;
  TCU_FUSED_CASE(2, 2)
  return cudaErrorInvalidValue;
}

cudaError_t launch_tile_r32(int prec, const PassArgs &a, long long grid, cudaStream_t st) {
  return prec == 3 ? launch_tile_t<32, 3>(a, grid, st) : launch_tile_t<32, 1>(a, grid, st);
}

}  // namespace tcu
