// kernels_mixed_r16.cu -- radix-16 passes of mixed-radix transforms
// n = q 16^k (q < 16 a power of two), after the q-point first pass:
// the last pass with n1 = q 16^s points before it, and the strided pass
// after the q prefix sequences.
#include "launch_impl.cuh"

namespace tcu {

// (stages, log2 other size, role, log2 prefix)
cudaError_t launch_pass_mixed_r16(int prec, int s, int lo, int role, int lp,
                                  const GArgs &a, int num_sms, cudaStream_t st) {
  constexpr int R = 16;
  TCU_PASS_CASE_L(2, 1, kSecond, 0)
  TCU_PASS_CASE_L(1, 8, kFirst, 1)
  TCU_PASS_CASE_L(2, 5, kSecond, 0)
  TCU_PASS_CASE_L(2, 8, kFirst, 1)
  TCU_PASS_CASE_L(2, 9, kSecond, 0)
  TCU_PASS_CASE_L(2, 2, kSecond, 0)
  TCU_PASS_CASE_L(1, 8, kFirst, 2)
  TCU_PASS_CASE_L(2, 6, kSecond, 0)
  TCU_PASS_CASE_L(2, 8, kFirst, 2)
  TCU_PASS_CASE_L(2, 10, kSecond, 0)
  TCU_PASS_CASE_L(2, 3, kSecond, 0)
  TCU_PASS_CASE_L(1, 8, kFirst, 3)
  TCU_PASS_CASE_L(2, 7, kSecond, 0)
  TCU_PASS_CASE_L(2, 8, kFirst, 3)
  TCU_PASS_CASE_L(2, 11, kSecond, 0)
  // n = q 16^s with any q = 2 .. 16 (runtime q; one tensor-core pass)
  TCU_PASS_CASE_L(1, 0, kSecondQ, 0)
  TCU_PASS_CASE_L(2, 0, kSecondQ, 0)
  return cudaErrorInvalidValue;
}

}  // namespace tcu
