// kernels_mixed_r8.cu -- radix-8 passes of mixed-radix transforms
// n = q 8^k (q < 8 a power of two), after the q-point first pass:
// the last pass with n1 = q 8^s points before it, and the strided pass
// after the q prefix sequences.
#include "launch_impl.cuh"

namespace tcu {

// (stages, log2 other size, role, log2 prefix)
cudaError_t launch_pass_mixed_r8(int prec, int s, int lo, int role, int lp,
                                  const GArgs &a, int num_sms, cudaStream_t st) {
  constexpr int R = 8;
  TCU_PASS_CASE_L(2, 1, kSecond, 0)
  TCU_PASS_CASE_L(3, 1, kSecond, 0)
  TCU_PASS_CASE_L(2, 6, kFirst, 1)
  TCU_PASS_CASE_L(2, 7, kSecond, 0)
  TCU_PASS_CASE_L(2, 2, kSecond, 0)
  TCU_PASS_CASE_L(3, 2, kSecond, 0)
  TCU_PASS_CASE_L(2, 6, kFirst, 2)
  TCU_PASS_CASE_L(2, 8, kSecond, 0)
  // n = q 8^s with any q = 2 .. 16 (runtime q; one tensor-core pass)
  TCU_PASS_CASE_L(1, 0, kSecondQ, 0)
  TCU_PASS_CASE_L(2, 0, kSecondQ, 0)
  TCU_PASS_CASE_L(3, 0, kSecondQ, 0)
  return cudaErrorInvalidValue;
}

}  // namespace tcu
