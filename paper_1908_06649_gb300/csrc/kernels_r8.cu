// kernels_r8.cu -- radix-8 kernel instantiations (sqrt(m) = 8).
#include "launch_impl.cuh"

namespace tcu {

// (stages, stages after (kFirst) or before (kSecond), role, stages before)
cudaError_t launch_pass_r8(int prec, int s, int lo, int role, int lp, const GArgs &a,
                           int num_sms, cudaStream_t st) {
  constexpr int R = 8;
  TCU_PASS_CASE(1, 0, kSingle, 0)
  TCU_PASS_CASE(2, 0, kSingle, 0)
  TCU_PASS_CASE(3, 0, kSingle, 0)
  TCU_PASS_CASE(2, 2, kFirst, 0)   // n = 8^4: 2 + 2
  TCU_PASS_CASE(2, 2, kSecond, 0)
  TCU_PASS_CASE(1, 4, kFirst, 0)   // n = 8^5: 1 + 2 + 2
  TCU_PASS_CASE(2, 2, kFirst, 1)
  TCU_PASS_CASE(2, 3, kSecond, 0)
  TCU_PASS_CASE(2, 4, kFirst, 0)   // n = 8^6: 2 + 2 + 2
  TCU_PASS_CASE(2, 2, kFirst, 2)
  TCU_PASS_CASE(2, 4, kSecond, 0)
  TCU_PASS_CASE(2, 5, kFirst, 0)   // n = 8^7: 2 + 2 + 3
  TCU_PASS_CASE(2, 3, kFirst, 2)
  TCU_PASS_CASE(3, 4, kSecond, 0)
  TCU_PASS_CASE(2, 6, kFirst, 0)   // n = 8^8: 2 + 3 + 3
  TCU_PASS_CASE(3, 3, kFirst, 2)
  TCU_PASS_CASE(3, 5, kSecond, 0)
  TCU_PASS_CASE(3, 6, kFirst, 0)   // n = 8^9: 3 + 3 + 3
  TCU_PASS_CASE(3, 3, kFirst, 3)
  TCU_PASS_CASE(3, 6, kSecond, 0)
  TCU_PASS_CASE(1, 3, kCols, 0)   // 2-D DFT column passes: n1 = R^s, n2 = R^so
  TCU_PASS_CASE(2, 2, kCols, 0)
  TCU_PASS_CASE(2, 3, kCols, 0)
  TCU_PASS_CASE(3, 1, kCols, 0)
  TCU_PASS_CASE(3, 2, kCols, 0)
  TCU_PASS_CASE(3, 3, kCols, 0)
  return cudaErrorInvalidValue;
}

// Team passes (items of tw warpgroups) for the 3-stage radix-8 passes of
// two-pass transforms: 8^5 = 2 + 3, 8^6 = 3 + 3.
cudaError_t launch_team_r8(int prec, int s, int lo, int role, int lp, int tw, const GArgs &a,
                           int num_sms, cudaStream_t st) {
  constexpr int R = 8;
  TCU_PASS_CASE(2, 3, kFirst, 0)   // 8^5: the 2-stage strided pass (one warpgroup)
  TCU_TEAM_CASE(3, 2, kSecond, 0, 2)
  TCU_TEAM_CASE(3, 2, kSecond, 0, 4)
  TCU_TEAM_CASE(3, 3, kFirst, 0, 2)  // 8^6
  TCU_TEAM_CASE(3, 3, kFirst, 0, 4)
  TCU_TEAM_CASE(3, 3, kSecond, 0, 2)
  TCU_TEAM_CASE(3, 3, kSecond, 0, 4)
  return cudaErrorInvalidValue;
}

cudaError_t launch_fused_r8(int prec, int s1, int s2, const GArgs &a, int num_sms,
                            cudaStream_t st) {
  constexpr int R = 8;
  TCU_FUSED_CASE(2, 2)
  return cudaErrorInvalidValue;
}

cudaError_t launch_rowconv_r8(int prec, int s, const GArgs &a, int num_sms,
                               cudaStream_t st) {
  constexpr int R = 8;
  TCU_ROWCONV_CASE(1)
  TCU_ROWCONV_CASE(2)
  TCU_ROWCONV_CASE(3)
  return cudaErrorInvalidValue;
}

}  // namespace tcu
