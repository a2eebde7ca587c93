// kernels_r8.cu -- radix-8 kernel instantiations (sqrt(m) = 8).
#include "launch_impl.cuh"

namespace tcu {

cudaError_t launch_pass_r8(int prec, int s, int so, int role, const GArgs &a, int num_sms,
                           cudaStream_t st) {
  constexpr int R = 8;
  TCU_PASS_CASE(1, 0, kSingle)
  TCU_PASS_CASE(2, 0, kSingle)
  TCU_PASS_CASE(3, 0, kSingle)
  TCU_PASS_CASE(2, 2, kFirst)   // n = 8^4
  TCU_PASS_CASE(2, 2, kSecond)
  TCU_PASS_CASE(2, 3, kFirst)   // n = 8^5
  TCU_PASS_CASE(3, 2, kSecond)
  TCU_PASS_CASE(3, 2, kFirst)
  TCU_PASS_CASE(2, 3, kSecond)
  TCU_PASS_CASE(3, 3, kFirst)   // n = 8^6
  TCU_PASS_CASE(3, 3, kSecond)
  TCU_PASS_CASE(3, 4, kSecond)  // n = 8^7 after a 4-stage tile pass
  return cudaErrorInvalidValue;
}

cudaError_t launch_fused_r8(int prec, int s1, int s2, const GArgs &a, int num_sms,
                            cudaStream_t st) {
  constexpr int R = 8;
  TCU_FUSED_CASE(2, 2)
  TCU_FUSED_CASE(2, 3)
  TCU_FUSED_CASE(3, 2)
  TCU_FUSED_CASE(3, 3)
  return cudaErrorInvalidValue;
}

cudaError_t launch_tile_r8(int prec, const PassArgs &a, long long grid, cudaStream_t st) {
  return prec == 3 ? launch_tile_t<8, 3>(a, grid, st) : launch_tile_t<8, 1>(a, grid, st);
}

}  // namespace tcu
