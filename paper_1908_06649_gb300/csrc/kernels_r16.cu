// kernels_r16.cu -- radix-16 kernel instantiations (sqrt(m) = 16).
#include "launch_impl.cuh"

namespace tcu {

// (stages, stages after (kFirst) or before (kSecond), role, stages before)
cudaError_t launch_pass_r16(int prec, int s, int lo, int role, int lp, const GArgs &a,
                            int num_sms, cudaStream_t st) {
  constexpr int R = 16;
  TCU_PASS_CASE(1, 0, kSingle, 0)
  TCU_PASS_CASE(2, 0, kSingle, 0)
  TCU_PASS_CASE(2, 2, kFirst, 0)   // n = 16^4: 2 + 2
  TCU_PASS_CASE(2, 2, kSecond, 0)
  TCU_PASS_CASE(1, 4, kFirst, 0)   // n = 16^5: 1 + 2 + 2
  TCU_PASS_CASE(2, 2, kFirst, 1)
  TCU_PASS_CASE(2, 3, kSecond, 0)
  TCU_PASS_CASE(2, 4, kFirst, 0)   // n = 16^6: 2 + 2 + 2
  TCU_PASS_CASE(2, 2, kFirst, 2)
  TCU_PASS_CASE(2, 4, kSecond, 0)
  TCU_PASS_CASE(1, 2, kCols, 0)   // 2-D DFT column passes: n1 = R^s, n2 = R^so
  TCU_PASS_CASE(2, 1, kCols, 0)
  TCU_PASS_CASE(2, 2, kCols, 0)
  return cudaErrorInvalidValue;
}

// Team passes: 16^3 in one pass on items of two warpgroups.
cudaError_t launch_team_r16(int prec, int s, int lo, int role, int lp, int tw, const GArgs &a,
                            int num_sms, cudaStream_t st) {
  constexpr int R = 16;
  TCU_TEAM_CASE(3, 0, kSingle, 0, 2)
  return cudaErrorInvalidValue;
}

cudaError_t launch_fused_r16(int prec, int s1, int s2, const GArgs &a, int num_sms,
                             cudaStream_t st) {
  constexpr int R = 16;
  TCU_FUSED_CASE(2, 2)
  return cudaErrorInvalidValue;
}

cudaError_t launch_pair_r16(int prec, int s1, int s2, const GArgs &a, int clusters,
                            cudaStream_t st) {
  constexpr int R = 16;
  TCU_PAIR_CASE(2, 2)
  return cudaErrorInvalidValue;
}

cudaError_t launch_rowconv_r16(int prec, int s, const GArgs &a, int num_sms,
                               cudaStream_t st) {
  constexpr int R = 16;
  TCU_ROWCONV_CASE(1)
  TCU_ROWCONV_CASE(2)
  return cudaErrorInvalidValue;
}

}  // namespace tcu
