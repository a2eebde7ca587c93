// launch_impl.cuh -- launch wrappers for one radix; included once per radix
// by kernels_r8.cu / kernels_r16.cu / kernels_r32.cu.
#pragma once
#include <string.h>

#include "launch.h"

namespace tcu {

template <int R, int PREC, int S, int LO, int ROLE, int LP>
cudaError_t launch_pass_t(const GArgs &a, int num_sms, cudaStream_t st) {
  using G = Geo<R, S, LO, ROLE, LP>;
  const size_t sm =
      SmemLayout<R, G::NWG, G::TW_ENTRIES, 0, G::TW_SMEM, G::TWB, 1, G::KS>::BYTES;
  cudaError_t e = cudaFuncSetAttribute(dft_pass_kernel<R, PREC, S, LO, ROLE, LP>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sm);
  if (e != cudaSuccess) return e;
  // one CTA per SM, each item on its own SM while there are fewer items
  // than SMs (latency), several per SM otherwise
  const long long nitems = (a.p[0].U + G::GG - 1) >> G::LOG2GG;
  long long grid = nitems < num_sms ? nitems : num_sms;
  dft_pass_kernel<R, PREC, S, LO, ROLE, LP><<<(unsigned)grid, G::THREADS, sm, st>>>(a);
  return cudaGetLastError();
}

// A team pass: items of TW warpgroups (128 TW rows), four warpgroups a CTA.
template <int R, int PREC, int S, int LO, int ROLE, int LP, int TW>
cudaError_t launch_team_t(const GArgs &a, int num_sms, cudaStream_t st) {
  using G = Geo<R, S, LO, ROLE, LP, 4, TW>;
  const size_t sm = SmemLayout<R, 4, G::TW_ENTRIES, 0, G::TW_SMEM, G::TWB, TW>::BYTES;
  cudaError_t e = cudaFuncSetAttribute(dft_pass_kernel<R, PREC, S, LO, ROLE, LP, false, TW>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sm);
  if (e != cudaSuccess) return e;
  const long long nitems = (a.p[0].U + G::GG - 1) >> G::LOG2GG;
  long long grid = nitems < num_sms ? nitems : num_sms;
  dft_pass_kernel<R, PREC, S, LO, ROLE, LP, false, TW>
      <<<(unsigned)grid, G::THREADS, sm, st>>>(a);
  return cudaGetLastError();
}

#define TCU_TEAM_CASE(S, SO, ROLE, SP, TW)                                               \
  if (s == S && lo == log2_radix(R) * (SO) && role == ROLE && lp == log2_radix(R) * (SP) && \
      tw == TW)                                                                           \
    return prec == 3 ? launch_team_t<R, 3, S, log2_radix(R) * (SO), ROLE,               \
                                     log2_radix(R) * (SP), TW>(a, num_sms, st)           \
                     : launch_team_t<R, 1, S, log2_radix(R) * (SO), ROLE,               \
                                     log2_radix(R) * (SP), TW>(a, num_sms, st);

// The convolution row pass (forward rows, spectrum product, inverse rows).
template <int R, int PREC, int S>
cudaError_t launch_rowconv_t(const GArgs &a, int num_sms, cudaStream_t st) {
  using G = Geo<R, S, 0, kSingle, 0, whole_k_nwg(R, kSingle)>;
  const size_t sm = SmemLayout<R, G::NWG, G::TW_ENTRIES, G::TW_ENTRIES, false, 0>::BYTES;
  cudaError_t e = cudaFuncSetAttribute(dft_pass_kernel<R, PREC, S, 0, kSingle, 0, true>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sm);
  if (e != cudaSuccess) return e;
  const long long nitems = (a.p[0].U + G::GG - 1) >> G::LOG2GG;
  long long grid = nitems < num_sms ? nitems : num_sms;
  dft_pass_kernel<R, PREC, S, 0, kSingle, 0, true><<<(unsigned)grid, G::THREADS, sm, st>>>(a);
  return cudaGetLastError();
}

#define TCU_ROWCONV_CASE(S)                                                         \
  if (s == S)                                                                       \
    return prec == 3 ? launch_rowconv_t<R, 3, S>(a, num_sms, st)                    \
                     : launch_rowconv_t<R, 1, S>(a, num_sms, st);

template <int R, int PREC, int S1, int S2>
cudaError_t launch_fused_t(const GArgs &a, int num_sms, cudaStream_t st) {
  using G1 = Geo<R, S1, log2_radix(R) * S2, kFirst, 0, whole_k_nwg(R, kFirst)>;
  using G2 = Geo<R, S2, log2_radix(R) * S1, kSecond, 0, G1::NWG>;
  const size_t sm =
      SmemLayout<R, G1::NWG, G1::TW_ENTRIES, G2::TW_ENTRIES, G1::TW_SMEM, G1::TWB>::BYTES;
  cudaError_t e = cudaFuncSetAttribute(dft_fused_kernel<R, PREC, S1, S2>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sm);
  if (e != cudaSuccess) return e;
  dft_fused_kernel<R, PREC, S1, S2><<<(unsigned)num_sms, G1::THREADS, sm, st>>>(a);
  return cudaGetLastError();
}

// Both passes of a two-pass transform in one launch on clusters of two CTAs
// (dft_pair_kernel): grid = 2 x clusters, one CTA per SM.
template <int R, int PREC, int S1, int S2>
cudaError_t launch_pair_t(const GArgs &a, int clusters, cudaStream_t st) {
  using PL = PairLayout<R, S1, S2>;
  const size_t sm = PL::BYTES;
  cudaError_t e = cudaFuncSetAttribute(dft_pair_kernel<R, PREC, S1, S2>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3((unsigned)(2 * clusters), 1, 1);
  cfg.blockDim = dim3(PL::G1::THREADS, 1, 1);
  cfg.dynamicSmemBytes = sm;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, dft_pair_kernel<R, PREC, S1, S2>, a);
}

#define TCU_PAIR_CASE(S1, S2)                                                       \
  if (s1 == S1 && s2 == S2)                                                         \
    return prec == 3 ? launch_pair_t<R, 3, S1, S2>(a, clusters, st)                 \
                     : launch_pair_t<R, 1, S1, S2>(a, clusters, st);

// Supported combinations of the warpgroup pass kernel for radix R, listed as
// a compile-time table; the plan only asks for these.  The dispatcher gets
// (s, lo, role, lp): stages, log2 of the other size (columns of a strided
// pass, points before the last pass) and log2 of the prefix count.
// TCU_PASS_CASE names sizes in stages of R, TCU_PASS_CASE_L in log2 units
// (mixed radix, where a factor q < R enters).
#define TCU_PASS_CASE_L(S, LO, ROLE, LP)                                            \
  if (s == S && lo == LO && role == ROLE && lp == LP)                               \
    return prec == 3 ? launch_pass_t<R, 3, S, LO, ROLE, LP>(a, num_sms, st)         \
                     : launch_pass_t<R, 1, S, LO, ROLE, LP>(a, num_sms, st);
#define TCU_PASS_CASE(S, SO, ROLE, SP) \
  TCU_PASS_CASE_L(S, log2_radix(R) * (SO), ROLE, log2_radix(R) * (SP))
// The BF16 modes (precision 4: BF16, 5: 3xBF16; tcgen05 kind::f16) of a
// pass or a team pass (items of TW warpgroups).
#define TCU_BF16_CASE(S, SO, ROLE, SP)                                                  \
  if (s == S && lo == log2_radix(R) * (SO) && role == ROLE &&                           \
      lp == log2_radix(R) * (SP) && tw == 1)                                            \
    return prec == 5 ? launch_pass_t<R, 5, S, log2_radix(R) * (SO), ROLE,               \
                                     log2_radix(R) * (SP)>(a, num_sms, st)              \
                     : launch_pass_t<R, 4, S, log2_radix(R) * (SO), ROLE,               \
                                     log2_radix(R) * (SP)>(a, num_sms, st);
#define TCU_BF16_TEAM_CASE(S, SO, ROLE, SP, TW)                                         \
  if (s == S && lo == log2_radix(R) * (SO) && role == ROLE &&                           \
      lp == log2_radix(R) * (SP) && tw == TW)                                           \
    return prec == 5 ? launch_team_t<R, 5, S, log2_radix(R) * (SO), ROLE,               \
                                     log2_radix(R) * (SP), TW>(a, num_sms, st)          \
                     : launch_team_t<R, 4, S, log2_radix(R) * (SO), ROLE,               \
                                     log2_radix(R) * (SP), TW>(a, num_sms, st);
#define TCU_FUSED_CASE(S1, S2)                                                      \
  if (s1 == S1 && s2 == S2)                                                         \
    return prec == 3 ? launch_fused_t<R, 3, S1, S2>(a, num_sms, st)                 \
                     : launch_fused_t<R, 1, S1, S2>(a, num_sms, st);

}  // namespace tcu
