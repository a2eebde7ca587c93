// kernels_bf16_r16.cu -- the BF16 precision modes (4: BF16, 5: 3xBF16;
// tcgen05 kind::f16 with bf16 operands) of the radix-16 passes of n = 16^k.
#include "launch_impl.cuh"

namespace tcu {

cudaError_t launch_pass_bf16_r16(int prec, int s, int lo, int role, int lp, int tw,
                                 const GArgs &a, int num_sms, cudaStream_t st) {
  constexpr int R = 16;
  TCU_BF16_TEAM_CASE(3, 0, kSingle, 0, 2)  // 16^3 in one pass
  TCU_BF16_CASE(1, 0, kSingle, 0)
  TCU_BF16_CASE(2, 0, kSingle, 0)
  TCU_BF16_CASE(2, 2, kFirst, 0)   // n = 16^4: 2 + 2
  TCU_BF16_CASE(2, 2, kSecond, 0)
  TCU_BF16_CASE(1, 4, kFirst, 0)   // n = 16^5: 1 + 2 + 2
  TCU_BF16_CASE(2, 2, kFirst, 1)
  TCU_BF16_CASE(2, 3, kSecond, 0)
  TCU_BF16_CASE(2, 4, kFirst, 0)   // n = 16^6: 2 + 2 + 2
  TCU_BF16_CASE(2, 2, kFirst, 2)
  TCU_BF16_CASE(2, 4, kSecond, 0)
  return cudaErrorInvalidValue;
}

}  // namespace tcu
