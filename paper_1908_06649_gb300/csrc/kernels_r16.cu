// kernels_r16.cu -- radix-16 kernel instantiations (sqrt(m) = 16).
#include "launch_impl.cuh"

namespace tcu {

cudaError_t launch_pass_r16(int prec, int s, int so, int role, const GArgs &a, int num_sms,
                            cudaStream_t st) {
  constexpr int R = 16;
  TCU_PASS_CASE(1, 0, kSingle)
  TCU_PASS_CASE(2, 0, kSingle)
  TCU_PASS_CASE(1, 2, kFirst)   // n = 16^3
  TCU_PASS_CASE(2, 1, kSecond)
  TCU_PASS_CASE(2, 1, kFirst)
  TCU_PASS_CASE(1, 2, kSecond)
  TCU_PASS_CASE(2, 2, kFirst)   // n = 16^4
  TCU_PASS_CASE(2, 2, kSecond)
  TCU_PASS_CASE(2, 3, kSecond)  // n = 16^5 after a 3-stage tile pass
  return cudaErrorInvalidValue;
}

cudaError_t launch_fused_r16(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st) {
  constexpr int R = 16;
  TCU_FUSED_CASE(2, 2)
  return cudaErrorInvalidValue;
}

cudaError_t launch_tile_r16(int prec, const PassArgs &a, long long grid, cudaStream_t st) {
  return prec == 3 ? launch_tile_t<16, 3>(a, grid, st) : launch_tile_t<16, 1>(a, grid, st);
}

}  // namespace tcu
