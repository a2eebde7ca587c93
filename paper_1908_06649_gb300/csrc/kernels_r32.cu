// kernels_r32.cu -- radix-32 kernel instantiations (sqrt(m) = 32).
#include "launch_impl.cuh"

namespace tcu {

// (stages, stages after (kFirst) or before (kSecond), role, stages before)
cudaError_t launch_pass_r32(int prec, int s, int lo, int role, int lp, const GArgs &a,
                            int num_sms, cudaStream_t st) {
  constexpr int R = 32;
  TCU_PASS_CASE(1, 0, kSingle, 0)
  TCU_PASS_CASE(2, 0, kSingle, 0)
  TCU_PASS_CASE(1, 2, kFirst, 0)   // n = 32^3: 1 + 2
  TCU_PASS_CASE(2, 1, kSecond, 0)
  TCU_PASS_CASE(2, 2, kFirst, 0)   // n = 32^4: 2 + 2
  TCU_PASS_CASE(2, 2, kSecond, 0)
  TCU_PASS_CASE(1, 4, kFirst, 0)   // n = 32^5: 1 + 2 + 2
  TCU_PASS_CASE(2, 2, kFirst, 1)
  TCU_PASS_CASE(2, 3, kSecond, 0)
  TCU_PASS_CASE(2, 4, kFirst, 0)   // n = 32^6: 2 + 2 + 2
  TCU_PASS_CASE(2, 2, kFirst, 2)
  TCU_PASS_CASE(2, 4, kSecond, 0)
  TCU_PASS_CASE(1, 2, kCols, 0)   // 2-D DFT column passes: n1 = R^s, n2 = R^so
  TCU_PASS_CASE(2, 1, kCols, 0)
  TCU_PASS_CASE(2, 2, kCols, 0)
  return cudaErrorInvalidValue;
}

cudaError_t launch_fused_r32(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st) {
  constexpr int R = 32;
  TCU_FUSED_CASE(2, 2)
  return cudaErrorInvalidValue;
}

cudaError_t launch_rowconv_r32(int prec, int s, const GArgs &a, int num_sms,
                               cudaStream_t st) {
  constexpr int R = 32;
  TCU_ROWCONV_CASE(1)
  TCU_ROWCONV_CASE(2)
  return cudaErrorInvalidValue;
}

}  // namespace tcu
