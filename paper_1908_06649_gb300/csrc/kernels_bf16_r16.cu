// kernels_bf16_r16.cu -- the BF16 precision modes (4: BF16, 5: 3xBF16;
// tcgen05 kind::f16 with bf16 operands) of the radix-16 passes of n = 16^k.
#include "launch_impl.cuh"

namespace tcu {

#define TCU_BF16_CASE(S, SO, ROLE, SP)                                                     \
  if (s == S && lo == 4 * (SO) && role == ROLE && lp == 4 * (SP) && tw == 1)               \
    return prec == 5 ? launch_pass_t<16, 5, S, 4 * (SO), ROLE, 4 * (SP)>(a, num_sms, st)  \
                     : launch_pass_t<16, 4, S, 4 * (SO), ROLE, 4 * (SP)>(a, num_sms, st);

cudaError_t launch_pass_bf16_r16(int prec, int s, int lo, int role, int lp, int tw,
                                 const GArgs &a, int num_sms, cudaStream_t st) {
  if (s == 3 && lo == 0 && role == kSingle && lp == 0 && tw == 2)  // 16^3, one pass
    return prec == 5 ? launch_team_t<16, 5, 3, 0, kSingle, 0, 2>(a, num_sms, st)
                     : launch_team_t<16, 4, 3, 0, kSingle, 0, 2>(a, num_sms, st);
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
