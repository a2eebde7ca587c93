// kernels_bf16_r8.cu -- the BF16 precision modes (4: BF16, 5: 3xBF16;
// tcgen05 kind::f16 with bf16 operands, N = 16, one K = 16 product per
// term) of the radix-8 passes of n = 8^k; the same pass table as the TF32
// modes, with the 3-stage passes of two-pass transforms on team items.
#include "launch_impl.cuh"

namespace tcu {

cudaError_t launch_pass_bf16_r8(int prec, int s, int lo, int role, int lp, int tw,
                                const GArgs &a, int num_sms, cudaStream_t st) {
  constexpr int R = 8;
  TCU_BF16_CASE(1, 0, kSingle, 0)
  TCU_BF16_CASE(2, 0, kSingle, 0)
  TCU_BF16_CASE(3, 0, kSingle, 0)
  TCU_BF16_CASE(2, 2, kFirst, 0)   // n = 8^4: 2 + 2
  TCU_BF16_CASE(2, 2, kSecond, 0)
  TCU_BF16_CASE(2, 3, kFirst, 0)   // n = 8^5: 2 + 3 (team)
  TCU_BF16_TEAM_CASE(3, 2, kSecond, 0, 4)
  TCU_BF16_TEAM_CASE(3, 3, kFirst, 0, 4)  // n = 8^6: 3 + 3 (teams)
  TCU_BF16_TEAM_CASE(3, 3, kSecond, 0, 4)
  TCU_BF16_CASE(2, 5, kFirst, 0)   // n = 8^7: 2 + 2 + 3
  TCU_BF16_CASE(2, 3, kFirst, 2)
  TCU_BF16_CASE(3, 4, kSecond, 0)
  TCU_BF16_CASE(2, 6, kFirst, 0)   // n = 8^8: 2 + 3 + 3
  TCU_BF16_CASE(3, 3, kFirst, 2)
  TCU_BF16_CASE(3, 5, kSecond, 0)
  TCU_BF16_CASE(3, 6, kFirst, 0)   // n = 8^9: 3 + 3 + 3
  TCU_BF16_CASE(3, 3, kFirst, 3)
  TCU_BF16_CASE(3, 6, kSecond, 0)
  return cudaErrorInvalidValue;
}

}  // namespace tcu
