// group_kernel.cuh -- warpgroup kernels for passes whose sub-transforms fit
// in one item of 128 TW data rows (L = r^S <= 128 TW r, TW = 1, 2 or 4
// warpgroups per item).
//
// A CTA (one per SM, persistent) holds NWG warpgroups grouped into teams of
// TW.  A warpgroup owns one TMEM slot (A_hi | A_lo | D for its 128 rows) and
// its product mbarrier; a team owns SMEM staging and transpose buffers, the
// staging mbarriers and one named barrier, and processes work items; an item
// is GG = 128 TW r / L consecutive sub-transforms, i.e. exactly 128 TW data
// rows per stage, so every stage of an item is one M=128 tall-left tcgen05
// product with F_r per warpgroup (the (m,l)-TCU call of Sec. 3 / Theorem 7)
// and the transposition between stages stays inside the team.
//
// Per item: the item's input block arrives in SMEM by TMA (a 1-D bulk copy
// when it is contiguous, a 3-D tensor box for a strided pass), issued by an
// elected lane of the team's first warp a whole item ahead; every thread
// reads its stage-1 row from there, splits it into hi/lo parts (TF32, or
// BF16 packed two per column) and stores them into TMEM as the A operand;
// an elected lane of each warpgroup's first warp issues its products; the
// epilogue reads D from TMEM, multiplies by the stage twiddles w_L^{k_t c_t}
// and writes the transposed rows of the next stage to SMEM; the last stage's
// outputs go straight from registers to global memory in natural order, with
// the inter-pass twiddle w_M^{k v} of a strided pass (staged by TMA from two
// small tables) applied on the way.  The inverse's 1/n is folded, exactly,
// into a 2^-log2(n)-scaled copy of F_r used by the last stage.
//
// Radix-32 passes of two stages run half-K items: a slot holds A for half
// of K, each stage's products run in two K halves, and staging and
// transpose share one buffer (so the next item's copy is issued after the
// last transpose read); four warpgroups then fit TMEM where whole-K slots
// fit two.  Every second pass of a plan processes its items last to first,
// starting on the part of its input the previous pass wrote last, which is
// still in L2.
//
// The whole geometry of a pass (radix, stages, other-side size, role, prefix,
// team) is a template parameter, so every stride is a compile-time constant.
//
// Kernels sharing the item routines:
//   dft_pass_kernel   -- one pass, items assigned round-robin; with CONV, the
//     row pass of a circular 2-D convolution (forward stages, spectrum
//     product, inverse stages of every row, on chip);
//   dft_fused_kernel  -- both passes of a two-pass (four-step) transform in
//     ONE launch: a work queue interleaves the passes by chunks of C
//     transforms, pass-1 items write their output to a small ring of chunks
//     that stays resident in L2, and pass-2 items read it back once all
//     pass-1 items of their transform have signalled (release/acquire
//     counters).  HBM then sees each point read once and written once.
#pragma once
#include <cuda.h>

#include "../../include/tcu_dft.h"
#include <cuda_bf16.h>

#include "tcgen05.cuh"

namespace tcu {

enum RowMode { kQF = 0, kUF = 1, kRQF = 2 };
// kSecondQ: the last pass of a mixed-radix transform n = q R^S whose factor
// q (2 .. 16, any integer) is a runtime value: the q-point first pass's
// output T[b n + v L + a], v < q, -> y[b n + v + k q]
enum Role { kSingle = 0, kFirst = 1, kSecond = 2, kCols = 3, kSecondQ = 4 };

__host__ __device__ constexpr int log2_radix(int R) { return R == 8 ? 3 : (R == 16 ? 4 : 5); }
// Warpgroups per CTA: TMEM holds 512 columns, a warpgroup's slot 3 Q of
// them; a radix-16 first (strided) pass also stages its inter-pass twiddles
// in SMEM, which leaves room for four; a radix-16 last pass of several runs
// four too (measured faster than five: 0.165 instead of 0.181 ms for the
// second pass of n = 16^4 x 1024).  A radix-32 pass of two stages runs
// four warpgroups whose slots hold A for half of K (the products of a stage
// in two K halves); one-stage radix-32 passes (already near the copy rate),
// the convolution row pass and the fused schedule keep whole-K slots, two
// per CTA at radix 32 (whole_k_nwg).
__host__ __device__ constexpr int pass_nwg(int R, int ROLE, int S = 2) {
  return R == 32 ? (S >= 2 ? 4 : 2) : ((ROLE == 1 || ROLE == 2) && R == 16 ? 4 : 5);
}
__host__ __device__ constexpr int whole_k_nwg(int R, int ROLE) {
  return R == 32 ? 2 : pass_nwg(R, ROLE);
}

// Compile-time geometry of one pass: S stages of radix R.  A transform of
// length n is computed in up to three passes (the four-step split applied
// recursively); a pass splits sequences of length M = R^S * 2^LO into
// L = R^S rows by n2 = 2^LO columns.  (With n = R^k every size is a power
// of R; a mixed-radix transform n = q R^k has one more factor q = 2^LP.)
//   kSingle: x[b n + a]                        -> y[b n + k]
//   kFirst : strided pass after a prefix of P = 2^LP sequences per
//            transform.  Sequence b' = (b, p), p < P, holds z[b' M + a n2 + v];
//            the DFT over a, times w_M^{v k}, goes to T[b n + (k P + p) n2 + v]
//            (for LP = 0: T[b n + k n2 + v])
//   kCols  : the column pass of a 2-D DFT of n1 x n2 arrays (n1 = R^S,
//            n2 = 2^LO): kFirst's geometry with LP = 0 and no twiddle,
//            x[b n + a n2 + v] -> X[b n + k n2 + v]
//   kSecond: last of several passes, n1 = 2^LO points before it per row:
//            T[b n + v L + a] -> y[b n + v + k n1]
//
// An item is the work of a team of TW warpgroups: 128 TW data rows, each
// warpgroup's 128 rows one M = 128 product per stage into its own TMEM slot;
// the team shares the item's SMEM staging and transpose buffers and
// synchronises on one named barrier.  TW > 1 lets an item hold sub-transforms
// longer than 128 rows, or more columns of a strided pass.
template <int R, int S, int LO, int ROLE, int LP = 0, int NWG_ = pass_nwg(R, ROLE, S),
          int TW_ = 1>
struct Geo {
  static constexpr int LOG2R = log2_radix(R);
  static constexpr int NWG = NWG_;
  static constexpr int TW = TW_;
  static constexpr int LOG2TW = TW == 1 ? 0 : (TW == 2 ? 1 : 2);
  static constexpr int NTEAM = NWG / TW;
  static constexpr int ROWS = 128 * TW;
  static constexpr int THREADS = 128 * NWG;
  static constexpr int LOG2GPTS = 7 + LOG2TW + LOG2R;   // ROWS rows of R points
  static constexpr int GPTS = 1 << LOG2GPTS;
  static constexpr int LOG2L = LOG2R * S;
  static constexpr int L = 1 << LOG2L;
  static constexpr int LOG2N = LOG2R * S + LO;          // sequence length M
  static constexpr int LOG2PRE = ROLE == kFirst ? LP : 0;
  static constexpr int LOG2NT = LOG2N + LOG2PRE;        // transform length n
  static constexpr int LOG2RPS = LOG2L - LOG2R;   // rows per sub-transform
  static constexpr int LOG2GG = LOG2GPTS - LOG2L; // sub-transforms per item
  static constexpr int GG = 1 << LOG2GG;
  static constexpr int LOG2O = LO;
  static constexpr int LOG2UPER = ROLE == kSingle ? 0 : LOG2O;
  static constexpr long long OUT_STRIDE =
      ROLE == kSingle ? 1 : (1ll << (LOG2O + LOG2PRE));
  static constexpr long long OUT_VSTRIDE = ROLE == kSingle ? 0 : 1;
  static constexpr bool STRIDED = ROLE == kFirst || ROLE == kCols;
  // the sub-transforms' prefix count q is a runtime value (PRun::q)
  static constexpr bool RTQ = ROLE == kSecondQ;
  static constexpr int MODE_FIRST = STRIDED ? kUF : kQF;
  static constexpr int MODE_MID = kUF;
  static constexpr int MODE_LAST = ROLE == kSingle ? kRQF : kUF;
  static constexpr bool TW_OUT = ROLE == kFirst;
  // inter-pass twiddles staged by TMA per item (else read from the
  // L2-resident tables): measured faster for radix 16 and for the radix-8
  // team items; the one-warpgroup radix-8 items run faster with five
  // warpgroups and global reads, radix 32 has no SMEM to spare
  static constexpr bool TW_SMEM = TW_OUT && (R == 16 || (R == 8 && TW > 1));
  // w_M^{k v} with v = vh 2^VL + vl: table A [k][vl] and, for more than 256
  // columns, table B [vh][k] (two-level, so that no table exceeds L * 256)
  static constexpr int LOG2VL = (TW_OUT && LOG2UPER > 8) ? 8 : LOG2UPER;
  static constexpr bool TW2L = TW_OUT && LOG2UPER > 8;
  static constexpr int TWB = (TW2L && TW_SMEM) ? L : 0;  // SMEM row of table B
  static constexpr int TMA_ROWS = L < 256 ? L : 256;  // tensor box height
  static constexpr int Q = (2 * R > 32) ? 2 * R : 32;
  // half-K products (radix 32, four warpgroups): A regions of Q/2 columns
  static constexpr bool KS = R == 32 && NWG == 4 && TW == 1;
  static constexpr int QA = KS ? Q / 2 : Q;
  // TMEM slot: A_hi (QA) | A_lo (QA) | D (Q)
  static constexpr int GCOLS = 2 * QA + Q;
  static constexpr int IMG_BYTES = 16 * R * R;
  // entries of the stage twiddle tables: sum over t < S of R * R^(S-t)
  static constexpr int TW_ENTRIES = S == 1 ? 0 : (S == 2 ? R * R : R * R * R + R * R);
  static_assert(LOG2GG >= 0, "sub-transform longer than one item");
  static_assert(LOG2GG <= LOG2VL || !TW_OUT, "an item spans one twiddle column block");
  static_assert(LOG2GG <= LOG2UPER || !STRIDED, "an item spans columns of one sequence");
  static_assert(NWG * GCOLS <= 512, "TMEM budget");
  static_assert(NTEAM * TW == NWG && (TW == 1 || TW == 2 || TW == 4), "team size");
};

// Runtime part of a pass.
struct PRun {
  const float2 *in;
  float2 *out;
  long long in_bmask, out_bmask;  // transform index mask (ring) or ~0
  long long U;                    // sub-transforms in the pass
  const float2 *tw_out;           // kFirst: w_M^{vl k} as [k][vl]
  const float2 *tw_b;             // kFirst, two-level: w_M^{vh 2^VL k} as [vh][k]
  const float2 *tw_stage;         // stage twiddles [t][j][lo]
  unsigned long long swz_tab;     // SMEM swizzle nibble per (ul & 15)
  int last_img;                   // byte offset of the last stage's F images
  // kSingle: if set, output k of sub-transform u is multiplied by
  // spec[(u & spec_mask) L + k] (a 2-D spectrum whose rows are the
  // sub-transforms: the pointwise product of a circular convolution)
  const float2 *spec;
  long long spec_mask;
  // process the items last to first: set on a pass that reads what the
  // previous pass wrote, whose latest output is still in L2
  int reverse;
  // kSecondQ: the factor q of n = q R^S (sub-transforms per transform)
  int q;
};

struct GArgs {
  PRun p[2];
  CUtensorMap tm_in;    // kFirst input  x as [b][a][2 v + re/im] floats
  CUtensorMap tm_tw;    // kFirst twiddles tw_out as [1][k][2 v + re/im]
  const float *bimg;    // F_r images: hi, lo, hi*2^-log2n, lo*2^-log2n
  int *err;
  // fused schedule
  int *counters;        // [0] queue head, [1, 1+batch) done1, then done2
  long long batch;
  int nchunks, lag, ring_chunks;
  int items1_per_tf;          // pass-1 items per transform
  int log2_items_per_chunk;   // items of one chunk, the same in both passes
};

// Offset of stage t's block [j][lo] in the stage twiddle table.
template <int R, int S>
__host__ __device__ constexpr int tw_stage_offset(int t) {
  int off = 0, p = 1;
  for (int i = 0; i < S - 1; ++i) p *= R;  // R^(S-1)
  for (int u = 1; u < t; ++u) {
    off += R * p;  // block u holds R * R^(S-u) entries
    p /= R;
  }
  return off;
}

// Shared memory: 4 F images | stage twiddles of two passes | per warpgroup
// transpose buffer, input staging and twiddle staging | mbarriers (3 per
// warpgroup: products, input staging, twiddle staging) | TMEM slot |
// scheduler mailboxes.
template <int R, int NWG, int TW1, int TW2, bool TWS, int TWB = 0, int TEAM = 1,
          bool SHARE = false>
struct SmemLayout {
  static constexpr int NTEAM = NWG / TEAM;
  static constexpr size_t IMG = 4 * 16 * R * R;
  static constexpr size_t OFF_TW1 = IMG;
  static constexpr size_t OFF_TW2 = OFF_TW1 + (size_t)TW1 * 8;
  static constexpr size_t PTS = 128 * (size_t)TEAM * R;  // points per item
  // transpose buffers aligned to 1024 bytes (swz_addr XORs address bits)
  static constexpr size_t OFF_BUF = (OFF_TW2 + (size_t)TW2 * 8 + 1023) / 1024 * 1024;
  // SHARE: staging and transpose in one buffer (the half-K radix-32 items)
  static constexpr size_t OFF_STG = OFF_BUF + (SHARE ? 0 : (size_t)NTEAM * PTS * 8);
  static constexpr size_t OFF_TWS = OFF_STG + (size_t)NTEAM * PTS * 8;
  static constexpr size_t TWS_BYTES = TWS ? (size_t)NTEAM * PTS * 8 : 0;
  static constexpr size_t OFF_TWB = OFF_TWS + TWS_BYTES;  // [k] row of table B
  static constexpr size_t TWB_PER_WG = TWB;               // per team
  static constexpr size_t TWB_BYTES = (size_t)NTEAM * TWB * 8;
  static constexpr size_t OFF_BAR = OFF_TWB + TWB_BYTES;
  // 3 mbarriers per warpgroup, the TMEM slot word, the tables' mbarrier
  static constexpr size_t OFF_SCHED = OFF_BAR + 8 * 3 * NWG + 16;
  static constexpr size_t BYTES = OFF_SCHED + 32 * NWG;
  static_assert(BYTES <= 227 * 1024, "shared memory budget");
};

// Per-warpgroup state.
struct WG {
  uint32_t slot;      // TMEM column base of this warpgroup's slot
  uint32_t lane_off;  // this warp's TMEM lane quarter
  uint32_t img_addr;  // SMEM address of the F images
  uint32_t bar_mma;   // mbarrier: products done
  uint32_t bar_stg;   // mbarrier: input staging full
  uint32_t bar_tws;   // mbarrier: twiddle staging full
  int bar_id;         // named barrier id (one per team)
  int bar_count;      // threads of the team
  int rho;            // this thread's row within the item (0 .. 128 TW - 1)
  bool wg_lead;       // warp 0 of its warpgroup: issues the warpgroup's products
  bool team_lead;     // warp 0 of the team: runs the schedule
  bool copy_lead;     // issues the team's copies: warp 0 of the team, or warp 1
                      // in the strided passes of two or more stages
  float2 *buf;        // SMEM transpose buffer
  float2 *stg;        // SMEM input staging (one item)
  float2 *tws;        // SMEM twiddle staging (one item)
  float2 *twb;        // SMEM row of twiddle table B (two-level tables)
  uint32_t ph_mma, ph_stg, ph_tws;
  bool fail;
  bool tws_inflight;  // warp 0: a twiddle copy has not been waited on
#ifdef TCU_DFT_CHECKED
  int *err;           // error word: index violations are recorded at once
#endif
};

// Bounds-checked build (-DTCU_DFT_CHECKED): false when index i is outside
// [0, n), with TCU_DFT_ERR_BOUNDS recorded in the error word; the caller
// then skips the access (no trap, no fault).  The constant true otherwise,
// so the normal build is unchanged.
__device__ __forceinline__ bool in_range(const WG &w, long long i, long long n) {
#ifdef TCU_DFT_CHECKED
  if (i >= 0 && i < n) return true;
  atomicCAS(w.err, 0, TCU_DFT_ERR_BOUNDS);
  return false;
#else
  (void)w;
  (void)i;
  (void)n;
  return true;
#endif
}

template <class G>
__device__ __forceinline__ void row_of(int mode, int rho, int &ul, int &q) {
  if (mode == kUF) {
    ul = rho & (G::GG - 1);
    q = rho >> G::LOG2GG;
  } else {
    ul = rho >> G::LOG2RPS;
    q = rho & ((1 << G::LOG2RPS) - 1);
    if (mode == kRQF) {  // digit-reversed q over S-1 digits
      int rq = 0, v = q;
#pragma unroll
      for (int i = 0; i < G::LOG2RPS / G::LOG2R; ++i) {
        rq = (rq << G::LOG2R) | (v & ((1 << G::LOG2R) - 1));
        v >>= G::LOG2R;
      }
      q = rq;
    }
  }
}

// Swizzle of the transpose buffer: the 8-byte slot (p mod 16) of index p is
// XORed with the table value of its sub-transform column and with bits 4-7
// of p; for sub-transforms longer than 256 points (WIDE) also with bits
// 8-11, where the leading digit of a 16^3 or 8^3 row lives.  A bijection on
// every 16-entry block; the host picks the table by a bank-conflict cost
// model of the same function.
template <bool WIDE>
__device__ __forceinline__ int gswz(int p, uint32_t tabv) {
  uint32_t h = tabv ^ (uint32_t)(p >> 4);
  if (WIDE) h ^= (uint32_t)(p >> 8);
  return p ^ (int)(h & 15u);
}

// The swizzle with a zero table value, at compile time.
template <bool WIDE>
__host__ __device__ constexpr int gswz0(int p) {
  return p ^ (((p >> 4) ^ (WIDE ? (p >> 8) : 0)) & 15);
}

// Shared address of entry gswz(base | (j << SH)) of a transpose buffer,
// for a row whose base index has no bit in [SH, SH + log2 R): the swizzle
// is linear over XOR, so the entry is gswz(base) ^ gswz0(j << SH).  `a` is
// the address of gswz(base) in a buffer aligned to 1024 bytes, so that an
// XOR below bit 10 of the byte offset is an XOR of the address; the part
// of j << SH above the first 16 entries (SH >= 4) is disjoint from the
// other bits and is added instead (an immediate offset of the access).
template <bool WIDE, int SH>
__device__ __forceinline__ uint32_t swz_addr(uint32_t a, int j) {
  const int c = gswz0<WIDE>(j << SH);
  const int hi = SH >= 4 ? (j << SH) : 0;
  return (a ^ (uint32_t)(8 * (c ^ hi))) + (uint32_t)(8 * hi);
}

// Precision modes: 1 TF32, 3 3xTF32 (kind::tf32, K = 8 fp32 per product);
// 4 BF16, 5 3xBF16 (kind::f16 with bf16 operands, K = 16 per product, two
// values packed per 32-bit TMEM column).
__host__ __device__ constexpr bool is_bf16(int PREC) { return PREC >= 4; }
__host__ __device__ constexpr bool is_split(int PREC) { return PREC == 3 || PREC == 5; }
// TMEM columns of the A operand for 8 complex values, and bytes of one F_r
// image (2r x 2r elements).
__host__ __device__ constexpr int a_cols8(int PREC) { return is_bf16(PREC) ? 8 : 16; }
// Values per register chunk of the loops that load operands (twiddles, rows,
// spectra) ahead of the asm stores that consume them: 16, or 8 where five
// warpgroups share the registers (at most 102 a thread).
__host__ __device__ constexpr int load_chunk(int R, int NWG) {
  return (R < 16 || NWG >= 5) ? 8 : 16;
}
__host__ __device__ constexpr int img_bytes(int R, int PREC) {
  return (is_bf16(PREC) ? 8 : 16) * R * R;
}

// Split of 8 complex values, stored as A operand columns of this thread's
// TMEM lane.  3xTF32: hi keeps the top 10 explicit mantissa bits (exactly
// representable in TF32) and lo = v - hi is exact in fp32.  TF32: hi rounded
// to nearest.  BF16 modes: hi = bf16 rounding of v, lo = bf16 rounding of
// v - hi (exact in fp32 before rounding), packed two per column.
template <int PREC>
__device__ __forceinline__ void split_store8(const float2 *x, uint32_t col_hi,
                                             uint32_t col_lo) {
  if constexpr (is_bf16(PREC)) {
    uint32_t ph[8], pl[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      // both parts rounded to nearest by one packed conversion (re in the
      // low half, im in the high half, as the B images expect)
      const __nv_bfloat162 h = __floats2bfloat162_rn(x[j].x, x[j].y);
      ph[j] = *reinterpret_cast<const uint32_t *>(&h);
      if (PREC == 5) {
        const __nv_bfloat162 l =
            __floats2bfloat162_rn(x[j].x - __low2float(h), x[j].y - __high2float(h));
        pl[j] = *reinterpret_cast<const uint32_t *>(&l);
      }
    }
    tmem_st8u(col_hi, ph);
    if (PREC == 5) tmem_st8u(col_lo, pl);
  } else {
    float vh[16], vl[16];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (PREC == 3) {
        const float hx = __uint_as_float(__float_as_uint(x[j].x) & 0xFFFFE000u);
        const float hy = __uint_as_float(__float_as_uint(x[j].y) & 0xFFFFE000u);
        vh[2 * j] = hx;
        vh[2 * j + 1] = hy;
        vl[2 * j] = x[j].x - hx;
        vl[2 * j + 1] = x[j].y - hy;
      } else {
        vh[2 * j] = tf32_rna(x[j].x);
        vh[2 * j + 1] = tf32_rna(x[j].y);
      }
    }
    tmem_st16(col_hi, vh);
    if (PREC == 3) tmem_st16(col_lo, vl);
  }
}

// One stage: D = A * Bf for the 128 rows of this warpgroup's slot.
// Split modes: one accumulator chain over three K-blocks, [A_lo | A_hi |
// A_hi] times [Bhi; Blo; Bhi] stacked -- lo*Bhi + hi*Blo + hi*Bhi, small
// terms first (lo*Blo is dropped: below the target precision).  The
// K-blocks read the same TMEM columns of A_hi twice; D has N = 2r columns.
// Each product covers 32 bytes of K: 8 fp32 (kind::tf32) or 16 bf16
// (kind::f16), i.e. 8 TMEM columns of A and two 16-byte core matrices of B.
//
// HALF >= 0: only the products of K half HALF, with A (QA columns per
// operand) holding that half; half 1 accumulates onto half 0.
template <int R, int PREC, int QA = ((2 * R > 32) ? 2 * R : 32), int HALF = -1>
__device__ __forceinline__ void issue_stage_mma(uint32_t slot, uint32_t img_addr) {
  constexpr bool BF = is_bf16(PREC);
  constexpr int IMG = img_bytes(R, PREC), LBO = 128, SBO = (BF ? 32 : 64) * R;
  constexpr int KSTEPS = 2 * R / (BF ? 16 : 8);
  constexpr int K0 = HALF < 0 ? 0 : HALF * (KSTEPS / 2);
  constexpr int K1 = HALF < 0 ? KSTEPS : K0 + KSTEPS / 2;
  constexpr uint32_t idesc = BF ? idesc_bf16(128, 2 * R) : idesc_tf32(128, 2 * R);
  const uint32_t ahi = slot, alo = slot + QA, d = slot + 2 * QA;
  const uint32_t ihi = img_addr, ilo = img_addr + IMG;
  uint32_t acc = HALF > 0 ? 1 : 0;
  if (is_split(PREC)) {
#pragma unroll
    for (int kk = K0; kk < K1; ++kk) {
      mma_ts<BF>(d, alo + 8 * (kk - K0), smem_desc_noswz(ihi + kk * 2 * LBO, LBO, SBO), idesc,
                 acc);
      acc = 1;
    }
#pragma unroll
    for (int kk = K0; kk < K1; ++kk)
      mma_ts<BF>(d, ahi + 8 * (kk - K0), smem_desc_noswz(ilo + kk * 2 * LBO, LBO, SBO), idesc,
                 1);
  }
#pragma unroll
  for (int kk = K0; kk < K1; ++kk) {
    mma_ts<BF>(d, ahi + 8 * (kk - K0), smem_desc_noswz(ihi + kk * 2 * LBO, LBO, SBO), idesc,
               acc);
    acc = 1;
  }
}

// This thread's whole D row (2r values), TMEM loads under one wait.
template <class G, int PREC>
__device__ __forceinline__ void load_d_row(const WG &w, float *d) {
  constexpr int R = 1 << G::LOG2R;
  const uint32_t base = w.slot + 2 * G::QA + w.lane_off;
  if (R == 8) {
    tmem_ld16(base, d);
  } else if (R == 16) {
    tmem_ld32(base, d);
  } else {
    tmem_ld32x2(base, base + 32, d);
  }
}

// ---- TMA issue (warp 0 of the warpgroup, converged; one elected lane
// issues): the input block of `item` into staging
template <class G, bool HINT = false>
__device__ __forceinline__ void issue_input(const PRun &P, const CUtensorMap *tm,
                                            long long item, const WG &w, uint64_t pol = 0) {
  const long long u0 = item << G::LOG2GG;
  const uint32_t dst = smem_u32(w.stg);
  if (G::MODE_FIRST == kUF) {
    // strided first pass: box of GG sub-transforms x L points
    const long long b = u0 >> G::LOG2UPER;
    const int v0 = (int)(u0 & ((1ll << G::LOG2UPER) - 1));
    if (elect_one()) {
      mbar_expect_tx(w.bar_stg, G::GPTS * 8);
#pragma unroll
      for (int a0 = 0; a0 < G::L; a0 += G::TMA_ROWS) {
        if (HINT)
          tma_load_3d_hint(dst + a0 * G::GG * 8, tm, 2 * v0, a0, (int)b, w.bar_stg, pol);
        else
          tma_load_3d(dst + a0 * G::GG * 8, tm, 2 * v0, a0, (int)b, w.bar_stg);
      }
    }
  } else {
    // contiguous block of GG sub-transforms (the last item may be short)
    long long rem = P.U - u0;
    if (rem > G::GG) rem = G::GG;
    const uint32_t bytes = (uint32_t)(rem << G::LOG2L) * 8u;
    const long long b = u0 >> G::LOG2UPER;
    const long long v = u0 & ((1ll << G::LOG2UPER) - 1);
    // with a runtime q the sub-transforms are simply consecutive
    const long long off =
        G::RTQ ? (u0 << G::LOG2L) : ((b & P.in_bmask) << G::LOG2N) + (v << G::LOG2L);
    const float2 *src = P.in + off;
    const long long in_elems =
        (P.in_bmask == -1 || G::RTQ) ? (P.U << G::LOG2L) : ((P.in_bmask + 1) << G::LOG2N);
    const bool ok = in_range(w, off + (rem << G::LOG2L) - 1, in_elems);
    if (elect_one()) {
      // a skipped copy still completes the phase (no bytes expected)
      mbar_expect_tx(w.bar_stg, ok ? bytes : 0u);
      if (ok) {
        if (HINT)
          tma_load_1d_hint(dst, src, bytes, w.bar_stg, pol);
        else
          tma_load_1d(dst, src, bytes, w.bar_stg);
      }
    }
  }
  __syncwarp();
}

// ---- TMA issue (warp 0, converged): the inter-pass twiddles of a strided
// item -- the [k][vl] box of table A and, for two-level tables, the row of
// table B for the item's vh
template <class G>
__device__ __forceinline__ void issue_twiddles(const PRun &P, const CUtensorMap *tm,
                                               long long item, const WG &w) {
  if constexpr (G::TW_SMEM) {
    const long long u0 = item << G::LOG2GG;
    const long long v0 = u0 & ((1ll << G::LOG2UPER) - 1);
    const int vl0 = (int)(v0 & ((1 << G::LOG2VL) - 1));
    const uint32_t dst = smem_u32(w.tws);
    const long long boff = (v0 >> G::LOG2VL) << G::LOG2L;
    const bool ok =
        !G::TW2L || in_range(w, boff + G::L - 1, (1ll << (G::LOG2UPER - G::LOG2VL)) << G::LOG2L);
    if (elect_one()) {
      mbar_expect_tx(w.bar_tws, G::GPTS * 8 + (G::TW2L && ok ? G::L * 8 : 0));
#pragma unroll
      for (int k0 = 0; k0 < G::L; k0 += G::TMA_ROWS)
        tma_load_3d(dst + k0 * G::GG * 8, tm, 2 * vl0, k0, 0, w.bar_tws);
      if (G::TW2L && ok) tma_load_1d(smem_u32(w.twb), P.tw_b + boff, G::L * 8, w.bar_tws);
    }
    __syncwarp();
  }
}

// ---- products of one stage (warp 0, converged): issue and commit from one
// elected lane
template <int R, int PREC>
__device__ __forceinline__ void issue_stage(uint32_t slot, uint32_t img_addr,
                                            uint32_t bar_mma) {
  if (elect_one()) {
    issue_stage_mma<R, PREC>(slot, img_addr);
    mma_commit(bar_mma);
  }
  __syncwarp();
}

// This thread's stage-1 row, from the staged input block.
template <class G>
__device__ __forceinline__ void staged_row(const WG &w, float2 *x) {
  constexpr int R = 1 << G::LOG2R;
  int ul, q;
  row_of<G>(G::MODE_FIRST, w.rho, ul, q);
  constexpr int JS = 1 << (G::LOG2L - G::LOG2R);  // a = j * R^(S-1) + q
  const float2 zero = make_float2(0.f, 0.f);
  if (G::MODE_FIRST == kUF) {
    const int i0 = q * G::GG + ul;  // staging [a][ul]
    const float2 *p = w.stg + i0;
#pragma unroll
    for (int j = 0; j < R; ++j)
      x[j] = in_range(w, i0 + j * JS * G::GG, G::GPTS) ? p[j * JS * G::GG] : zero;
  } else {
    const int i0 = (ul << G::LOG2L) + q;  // staging [ul][a]
    const float2 *p = w.stg + i0;
#pragma unroll
    for (int j = 0; j < R; ++j) x[j] = in_range(w, i0 + j * JS, G::GPTS) ? p[j * JS] : zero;
  }
}

// Epilogue of stage T < S: D -> registers, stage twiddle, transposed write.
template <class G, int PREC, int T>
__device__ __forceinline__ void stage_epilogue(const PRun &P, const float2 *tws,
                                               const WG &w) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  constexpr int SH = G::LOG2R * (S - T);  // digits below the current one
  constexpr int TWOFF = tw_stage_offset<R, S>(T);
  int ul, q;
  row_of<G>(T == 1 ? G::MODE_FIRST : G::MODE_MID, w.rho, ul, q);
  const int hi = q >> SH, lo = q & ((1 << SH) - 1);
  const int base = (ul << G::LOG2L) + (hi << (SH + G::LOG2R)) + lo;
  const uint32_t tabv = (uint32_t)(P.swz_tab >> (4 * (ul & 15))) & 15u;
  const float2 *twrow = tws + TWOFF + lo;  // [j][lo], row length R^(S-T)
#ifndef TCU_DFT_CHECKED
  const uint32_t a = smem_u32(w.buf) + 8u * (uint32_t)gswz<(G::LOG2L > 8)>(base, tabv);
#endif
  // The twiddles of a chunk are loaded before its stores (and the first
  // chunk's before the TMEM load): the stores and the TMEM load are asm
  // statements with a memory clobber, so a load written after one of them
  // would be issued only after it, one shared-memory round trip per value.
  constexpr int CH = load_chunk(R, G::NWG);
  float2 t[CH];
#pragma unroll
  for (int jj = 0; jj < CH; ++jj)
    t[jj] = in_range(w, TWOFF + lo + (jj << SH), G::TW_ENTRIES) ? twrow[jj << SH]
                                                                 : make_float2(1.f, 0.f);
  float d[2 * R];
  load_d_row<G, PREC>(w, d);
#pragma unroll
  for (int c = 0; c < R; c += CH) {
    if (c > 0) {
#pragma unroll
      for (int jj = 0; jj < CH; ++jj)
        t[jj] = in_range(w, TWOFF + lo + ((c + jj) << SH), G::TW_ENTRIES)
                    ? twrow[(c + jj) << SH]
                    : make_float2(1.f, 0.f);
    }
#pragma unroll
    for (int jj = 0; jj < CH; ++jj) {
      const int j = c + jj;
      const float2 y = cmul(make_float2(d[2 * j], d[2 * j + 1]), t[jj]);
#ifdef TCU_DFT_CHECKED
      const int bi = gswz<(G::LOG2L > 8)>(base + (j << SH), tabv);
      if (in_range(w, bi, G::GPTS)) w.buf[bi] = y;
#else
      st_shared_f2(swz_addr<(G::LOG2L > 8), SH>(a, j), y);
#endif
    }
  }
}

// Rows of stage T >= 2 from the SMEM buffer into TMEM.
template <class G, int PREC, int T>
__device__ __forceinline__ void stage_rows(const PRun &P, const WG &w) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  constexpr int SH = G::LOG2R * (S - T);
  int ul, q;
  row_of<G>(T == S ? G::MODE_LAST : G::MODE_MID, w.rho, ul, q);
  const int hi = q >> SH, lo = q & ((1 << SH) - 1);
  const int base = (ul << G::LOG2L) + (hi << (SH + G::LOG2R)) + lo;
  const uint32_t tabv = (uint32_t)(P.swz_tab >> (4 * (ul & 15))) & 15u;
#ifndef TCU_DFT_CHECKED
  const uint32_t a = smem_u32(w.buf) + 8u * (uint32_t)gswz<(G::LOG2L > 8)>(base, tabv);
#endif
  // a whole chunk is loaded before its TMEM stores (asm with a memory
  // clobber, which a later load could not pass)
  constexpr int CH = load_chunk(R, G::NWG);
#pragma unroll
  for (int c = 0; c < R; c += CH) {
    float2 row[CH];
#pragma unroll
    for (int jj = 0; jj < CH; ++jj) {
#ifdef TCU_DFT_CHECKED
      const int bi = gswz<(G::LOG2L > 8)>(base + ((c + jj) << SH), tabv);
      row[jj] = in_range(w, bi, G::GPTS) ? w.buf[bi] : make_float2(0.f, 0.f);
#else
      row[jj] = ld_shared_f2(swz_addr<(G::LOG2L > 8), SH>(a, c + jj));
#endif
    }
#pragma unroll
    for (int c8 = 0; c8 < CH; c8 += 8)
      split_store8<PREC>(row + c8, w.slot + w.lane_off + a_cols8(PREC) * (c + c8) / 8,
                         w.slot + G::Q + w.lane_off + a_cols8(PREC) * (c + c8) / 8);
  }
}

// Last stage: D -> registers -> natural-order output.
template <class G, int PREC, bool OUT_L2, bool SPEC = true>
__device__ __forceinline__ void last_stage_store(const PRun &P, long long item, WG &w) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  int ul, q;
  row_of<G>(G::MODE_LAST, w.rho, ul, q);
  const long long u = (item << G::LOG2GG) + ul;
  float d[2 * R];
  load_d_row<G, PREC>(w, d);
  if constexpr (G::TW_SMEM) {
    if (mbar_wait_bounded(w.bar_tws, w.ph_tws))
      w.tws_inflight = false;
    else
      w.fail = true;
    w.ph_tws ^= 1;
  }
  if (u >= P.U) return;
  int klow = 0, vq = q;
#pragma unroll
  for (int i = 0; i < S - 1; ++i) {
    klow = (klow << G::LOG2R) | (vq & (R - 1));
    vq >>= G::LOG2R;
  }
  long long b = u >> G::LOG2UPER;
  long long v = u & ((1ll << G::LOG2UPER) - 1);
  // kFirst after a prefix: sequence b = (transform, p) -> transform-major,
  // k above p
  const long long bt = b >> G::LOG2PRE, bp = b & ((1ll << G::LOG2PRE) - 1);
  float2 *dst = P.out + ((bt & P.out_bmask) << G::LOG2NT) + (bp << G::LOG2UPER) +
                v * G::OUT_VSTRIDE + klow * G::OUT_STRIDE;
  long long JS = G::OUT_STRIDE << (G::LOG2L - G::LOG2R);
  if constexpr (G::RTQ) {
    // transform b = u / q, row v = u mod q: y[b q L + v + k q]
    const long long q = P.q;
    b = u / q;
    v = u - b * q;
    dst = P.out + b * (q << G::LOG2L) + v + klow * q;
    JS = q << (G::LOG2L - G::LOG2R);
  }
  // twiddle of output k = klow + j r^(S-1): table A staged as [k][ul] in SMEM,
  // or read from global [k][vl]; two-level: times B[vh][k]
  const float2 *tws = w.tws + klow * G::GG + ul;
  constexpr int TJS = G::GG << (G::LOG2L - G::LOG2R);
  const long long vl = v & ((1ll << G::LOG2VL) - 1), vh = v >> G::LOG2VL;
  const float2 *twg = P.tw_out + ((long long)klow << G::LOG2VL) + vl;
  constexpr long long TWG = 1ll << (G::LOG2VL + G::LOG2L - G::LOG2R);
  const float2 *twbs = w.twb + klow;
  const float2 *twbg = P.tw_b + (vh << G::LOG2L) + klow;
  constexpr int TBJ = 1 << (G::LOG2L - G::LOG2R);
  const long long soff = ((u & P.spec_mask) << G::LOG2L) + klow;
  const float2 *sp = P.spec + soff;
  const bool mul = SPEC && G::MODE_LAST == kRQF && P.spec != nullptr;
  // index bounds of the checked build (element offsets from each base)
  const long long doff = dst - P.out;
  const long long out_elems =
      P.out_bmask == -1 ? (P.U << G::LOG2L) : ((P.out_bmask + 1) << G::LOG2NT);
  const long long toff = klow * G::GG + ul, goff = ((long long)klow << G::LOG2VL) + vl;
  const long long gboff = (vh << G::LOG2L) + klow;
  const float2 one = make_float2(1.f, 0.f);
  // The factors of a chunk of outputs (spectrum, twiddles) are loaded before
  // its stores: the stores are asm with a memory clobber, so a load written
  // after one of them would wait for it, a round trip per value.
  constexpr int CH = (G::TW2L || G::MODE_LAST == kRQF) ? 8 : load_chunk(R, G::NWG);
#pragma unroll
  for (int c = 0; c < R; c += CH) {
    float2 fs[CH], fa[CH], fb[CH];
#pragma unroll
    for (int jj = 0; jj < CH; ++jj) {
      const int j = c + jj;
      if (G::MODE_LAST == kRQF && mul)
        fs[jj] = in_range(w, soff + j * JS, (P.spec_mask + 1) << G::LOG2L) ? __ldg(sp + j * JS)
                                                                          : one;
      if (G::TW_SMEM) {
        fa[jj] = in_range(w, toff + j * TJS, G::GPTS) ? tws[j * TJS] : one;
        if (G::TW2L) fb[jj] = in_range(w, klow + j * TBJ, G::L) ? twbs[j * TBJ] : one;
      } else if (G::TW_OUT) {
        fa[jj] = in_range(w, goff + j * TWG, (long long)G::L << G::LOG2VL) ? __ldg(twg + j * TWG)
                                                                          : one;
        if (G::TW2L)
          fb[jj] = in_range(w, gboff + j * TBJ, (1ll << (G::LOG2UPER - G::LOG2VL)) << G::LOG2L)
                       ? __ldg(twbg + j * TBJ)
                       : one;
      }
    }
#pragma unroll
    for (int jj = 0; jj < CH; ++jj) {
      const int j = c + jj;
      float2 y = make_float2(d[2 * j], d[2 * j + 1]);
      if (G::MODE_LAST == kRQF && mul) y = cmul(y, fs[jj]);
      if (G::TW_SMEM || G::TW_OUT) y = G::TW2L ? cmul(y, cmul(fa[jj], fb[jj])) : cmul(y, fa[jj]);
      if (in_range(w, doff + j * JS, out_elems)) {
        if (OUT_L2)
          __stcg(dst + j * JS, y);
        else
          __stcs(dst + j * JS, y);
      }
    }
  }
}

// The whole item.  `mid` supplies the next-item logic (warp 0 of the
// warpgroup runs issue() right after the stage-1 products and publish() just
// before the first epilogue barrier).  On entry the item's input copy has been issued.
template <class G, int PREC, bool OUT_L2, class Mid>
__device__ __forceinline__ void process_item(const PRun &P, const CUtensorMap *tm_tw,
                                             const float2 *tws, long long item, WG &w,
                                             Mid &mid) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  if (!mbar_wait_bounded(w.bar_stg, w.ph_stg)) w.fail = true;
  w.ph_stg ^= 1;
  mid.after_load(w);
  {
    float2 x[R];
    staged_row<G>(w, x);
#pragma unroll
    for (int c = 0; c < R; c += 8)
      split_store8<PREC>(x + c, w.slot + w.lane_off + a_cols8(PREC) * c / 8,
                         w.slot + G::Q + w.lane_off + a_cols8(PREC) * c / 8);
  }
  tmem_wait_st();
  fence_before_sync();
  if (named_bar_or(w.bar_id, w.bar_count, w.fail)) {
    w.fail = true;
    return;
  }
  // staging is free again: the next item's copy may land there
  if (w.wg_lead) {
    fence_after_sync();
    issue_stage<R, PREC>(w.slot, w.img_addr + (S == 1 ? P.last_img : 0), w.bar_mma);
  }
  if (w.copy_lead) {
    if (G::TW_SMEM) {
      issue_twiddles<G>(P, tm_tw, item, w);
      w.tws_inflight = true;
    }
    mid.issue(w);
  }
  if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
  w.ph_mma ^= 1;
  fence_after_sync();
  constexpr int S2 = S >= 2 ? 2 : S, S3 = S >= 3 ? 3 : S2;
#pragma unroll
  for (int t = 1; t < S; ++t) {
    if (t == 1) stage_epilogue<G, PREC, 1>(P, tws, w);
    if (t == 2) stage_epilogue<G, PREC, S2>(P, tws, w);
    if (t == 1 && w.team_lead) mid.publish();
    fence_before_sync();
    named_bar_or(w.bar_id, w.bar_count, false);
    if (t == 1) stage_rows<G, PREC, S2>(P, w);
    if (t == 2) stage_rows<G, PREC, S3>(P, w);
    tmem_wait_st();
    fence_before_sync();
    if (named_bar_or(w.bar_id, w.bar_count, w.fail)) {
      w.fail = true;
      return;
    }
    if (w.wg_lead) {
      fence_after_sync();
      issue_stage<R, PREC>(w.slot, w.img_addr + (t + 1 == S ? P.last_img : 0), w.bar_mma);
    }
    if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
    w.ph_mma ^= 1;
    fence_after_sync();
  }
  if (S == 1 && w.team_lead) mid.publish();
  mid.before_store(w);
  last_stage_store<G, PREC, OUT_L2>(P, item, w);
}

// ---- half-K items (radix 32, four warpgroups).  A warpgroup's TMEM slot
// holds A for one half of K (A_hi, A_lo: QA columns each) and the whole D,
// so four slots fit the 512 columns where whole-K slots fit two.  Each
// stage runs its products in two K halves: the rows' first R/2 values go
// into A, the products of that half are issued, and once they have read A
// the second R/2 values replace them and the second half accumulates onto
// D.  Staging and transpose share one buffer, so the next item's copy is
// issued once the last transpose has been read.

// Products of one K half (warp 0, converged; one elected lane).
template <int R, int PREC, int QA>
__device__ __forceinline__ void issue_stage_half(int h, uint32_t slot, uint32_t img_addr,
                                                 uint32_t bar_mma) {
  if (elect_one()) {
    if (h == 0)
      issue_stage_mma<R, PREC, QA, 0>(slot, img_addr);
    else
      issue_stage_mma<R, PREC, QA, 1>(slot, img_addr);
    mma_commit(bar_mma);
  }
  __syncwarp();
}

// Values h R/2 .. (h+1) R/2 - 1 of this thread's stage-1 row.
template <class G>
__device__ __forceinline__ void staged_row_half(const WG &w, float2 *x, int h) {
  constexpr int R = 1 << G::LOG2R, H = R / 2;
  int ul, q;
  row_of<G>(G::MODE_FIRST, w.rho, ul, q);
  constexpr int JS = 1 << (G::LOG2L - G::LOG2R);  // a = j * R^(S-1) + q
  const float2 zero = make_float2(0.f, 0.f);
  const int i0 = G::MODE_FIRST == kUF ? q * G::GG + ul : (ul << G::LOG2L) + q;
  constexpr int JST = G::MODE_FIRST == kUF ? JS * G::GG : JS;
#pragma unroll
  for (int j = 0; j < H; ++j) {
    const int i = i0 + (h * H + j) * JST;
    x[j] = in_range(w, i, G::GPTS) ? w.stg[i] : zero;
  }
}

// Values h R/2 .. (h+1) R/2 - 1 of this thread's stage-T row, from the
// transpose buffer into the half-K A region.
template <class G, int PREC, int T>
__device__ __forceinline__ void stage_rows_half(const PRun &P, const WG &w, int h) {
  constexpr int R = 1 << G::LOG2R, H = R / 2;
  constexpr int S = G::LOG2L / G::LOG2R;
  constexpr int SH = G::LOG2R * (S - T);
  int ul, q;
  row_of<G>(T == S ? G::MODE_LAST : G::MODE_MID, w.rho, ul, q);
  const int hi = q >> SH, lo = q & ((1 << SH) - 1);
  const int base = (ul << G::LOG2L) + (hi << (SH + G::LOG2R)) + lo;
  const uint32_t tabv = (uint32_t)(P.swz_tab >> (4 * (ul & 15))) & 15u;
#ifndef TCU_DFT_CHECKED
  const uint32_t a = smem_u32(w.buf) + 8u * (uint32_t)gswz<(G::LOG2L > 8)>(base, tabv);
#endif
  // the half row is loaded before its TMEM stores (asm with a memory
  // clobber, which a later load could not pass)
  float2 row[H];
#pragma unroll
  for (int jj = 0; jj < H; ++jj) {
#ifdef TCU_DFT_CHECKED
    const int bi = gswz<(G::LOG2L > 8)>(base + ((h * H + jj) << SH), tabv);
    row[jj] = in_range(w, bi, G::GPTS) ? w.buf[bi] : make_float2(0.f, 0.f);
#else
    row[jj] = ld_shared_f2(swz_addr<(G::LOG2L > 8), SH>(a, h * H + jj));
#endif
  }
#pragma unroll
  for (int c = 0; c < H; c += 8)
    split_store8<PREC>(row + c, w.slot + w.lane_off + a_cols8(PREC) * c / 8,
                       w.slot + G::QA + w.lane_off + a_cols8(PREC) * c / 8);
}

template <class G, int PREC, class Mid>
__device__ __forceinline__ void process_item_ks(const PRun &P, const float2 *tws,
                                                long long item, WG &w, Mid &mid) {
  constexpr int R = 1 << G::LOG2R, H = R / 2;
  constexpr int S = G::LOG2L / G::LOG2R;
  static_assert(G::KS && S <= 2 && !G::TW_SMEM, "half-K items: radix 32, at most two stages");
  if (!mbar_wait_bounded(w.bar_stg, w.ph_stg)) w.fail = true;
  w.ph_stg ^= 1;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    {
      float2 x[H];
      staged_row_half<G>(w, x, h);
#pragma unroll
      for (int c = 0; c < H; c += 8)
        split_store8<PREC>(x + c, w.slot + w.lane_off + a_cols8(PREC) * c / 8,
                           w.slot + G::QA + w.lane_off + a_cols8(PREC) * c / 8);
    }
    tmem_wait_st();
    fence_before_sync();
    if (named_bar_or(w.bar_id, w.bar_count, w.fail)) {
      w.fail = true;
      return;
    }
    if (w.wg_lead) {
      fence_after_sync();
      issue_stage_half<R, PREC, G::QA>(h, w.slot, w.img_addr + (S == 1 ? P.last_img : 0),
                                       w.bar_mma);
    }
    // one stage: the staging has been read and no transpose follows
    if (S == 1 && h == 1 && w.team_lead) mid.issue(w);
    if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
    w.ph_mma ^= 1;
    fence_after_sync();
  }
  if constexpr (S == 2) {
    stage_epilogue<G, PREC, 1>(P, tws, w);
    if (w.team_lead) mid.publish();
    fence_before_sync();
    named_bar_or(w.bar_id, w.bar_count, false);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      stage_rows_half<G, PREC, 2>(P, w, h);
      tmem_wait_st();
      fence_before_sync();
      if (named_bar_or(w.bar_id, w.bar_count, w.fail)) {
        w.fail = true;
        return;
      }
      if (w.wg_lead) {
        fence_after_sync();
        issue_stage_half<R, PREC, G::QA>(h, w.slot, w.img_addr + P.last_img, w.bar_mma);
      }
      // the transpose buffer (shared with the staging) has been read
      if (h == 1 && w.team_lead) mid.issue(w);
      if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
      w.ph_mma ^= 1;
      fence_after_sync();
    }
  } else {
    if (w.team_lead) mid.publish();
  }
  last_stage_store<G, PREC, false>(P, item, w);
}

// Convolution row item (kSingle geometry): the forward transform of each
// row, the product with the spectrum, and the inverse transform, all on chip.
// The thread that holds forward outputs k = klow + j r^(S-1) of a row after
// the last forward stage (digit-reversed row map) is the thread whose
// inverse stage-1 row is exactly those k in the same order (natural row
// map, same TMEM lane): it multiplies them by the spectrum and stores them
// straight back as its A operand.  F images in SMEM: forward hi, lo at 0,
// inverse hi, lo at 2 IMG; stage twiddles tw_f (forward), tw_i (inverse).
template <class G, int PREC>
__device__ __forceinline__ void conv_turn(const PRun &P, long long item, const WG &w) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  int ul, q;
  row_of<G>(kRQF, w.rho, ul, q);
  int klow = 0, vq = q;
#pragma unroll
  for (int i = 0; i < S - 1; ++i) {
    klow = (klow << G::LOG2R) | (vq & (R - 1));
    vq >>= G::LOG2R;
  }
  const long long u = (item << G::LOG2GG) + ul;
  float d[2 * R];
  load_d_row<G, PREC>(w, d);
  const float2 *sp = P.spec + ((u & P.spec_mask) << G::LOG2L) + klow;
  constexpr int JS = 1 << (G::LOG2L - G::LOG2R);
#pragma unroll
  for (int c = 0; c < R; c += 8) {
    float2 x[8];
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
#ifdef TCU_DFT_CHECKED
      const float2 s = in_range(w, (sp - P.spec) + (c + jj) * JS, (P.spec_mask + 1) << G::LOG2L)
                           ? __ldg(sp + (c + jj) * JS)
                           : make_float2(0.f, 0.f);
#else
      const float2 s = __ldg(sp + (c + jj) * JS);
#endif
      x[jj] = cmul(make_float2(d[2 * (c + jj)], d[2 * (c + jj) + 1]), s);
    }
    split_store8<PREC>(x, w.slot + w.lane_off + a_cols8(PREC) * c / 8,
                       w.slot + G::Q + w.lane_off + a_cols8(PREC) * c / 8);
  }
}

// Stages 2..S of one direction after the stage-1 products were issued:
// epilogue, transpose, next products (F images at img_off).
template <class G, int PREC, class Mid>
__device__ __forceinline__ bool later_stages(const PRun &P, const float2 *tws, WG &w,
                                             uint32_t img_off, Mid &mid, bool publish) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  constexpr int S2 = S >= 2 ? 2 : S, S3 = S >= 3 ? 3 : S2;
#pragma unroll
  for (int t = 1; t < S; ++t) {
    if (t == 1) stage_epilogue<G, PREC, 1>(P, tws, w);
    if (t == 2) stage_epilogue<G, PREC, S2>(P, tws, w);
    if (publish && t == 1 && w.team_lead) mid.publish();
    fence_before_sync();
    named_bar_or(w.bar_id, w.bar_count, false);
    if (t == 1) stage_rows<G, PREC, S2>(P, w);
    if (t == 2) stage_rows<G, PREC, S3>(P, w);
    tmem_wait_st();
    fence_before_sync();
    if (named_bar_or(w.bar_id, w.bar_count, w.fail)) {
      w.fail = true;
      return false;
    }
    if (w.wg_lead) {
      fence_after_sync();
      issue_stage<R, PREC>(w.slot, w.img_addr + img_off, w.bar_mma);
    }
    if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
    w.ph_mma ^= 1;
    fence_after_sync();
  }
  return true;
}

template <class G, int PREC, class Mid>
__device__ __forceinline__ void process_item_conv(const PRun &P, const float2 *tw_f,
                                                  const float2 *tw_i, long long item, WG &w,
                                                  Mid &mid) {
  constexpr int R = 1 << G::LOG2R;
  constexpr uint32_t INV = 2 * img_bytes(R, PREC);
  if (!mbar_wait_bounded(w.bar_stg, w.ph_stg)) w.fail = true;
  w.ph_stg ^= 1;
  {
    float2 x[R];
    staged_row<G>(w, x);
#pragma unroll
    for (int c = 0; c < R; c += 8)
      split_store8<PREC>(x + c, w.slot + w.lane_off + a_cols8(PREC) * c / 8,
                         w.slot + G::Q + w.lane_off + a_cols8(PREC) * c / 8);
  }
  tmem_wait_st();
  fence_before_sync();
  if (named_bar_or(w.bar_id, w.bar_count, w.fail)) {
    w.fail = true;
    return;
  }
  if (w.wg_lead) {
    fence_after_sync();
    issue_stage<R, PREC>(w.slot, w.img_addr, w.bar_mma);
  }
  if (w.team_lead) mid.issue(w);
  if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
  w.ph_mma ^= 1;
  fence_after_sync();
  if (!later_stages<G, PREC>(P, tw_f, w, 0, mid, true)) return;
  // the turn: forward outputs times the spectrum become the inverse A rows
  conv_turn<G, PREC>(P, item, w);
  tmem_wait_st();
  fence_before_sync();
  if (named_bar_or(w.bar_id, w.bar_count, w.fail)) {
    w.fail = true;
    return;
  }
  if (w.wg_lead) {
    fence_after_sync();
    issue_stage<R, PREC>(w.slot, w.img_addr + INV, w.bar_mma);
  }
  if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
  w.ph_mma ^= 1;
  fence_after_sync();
  if (!later_stages<G, PREC>(P, tw_i, w, INV, mid, false)) return;
  last_stage_store<G, PREC, false, false>(P, item, w);
}

// Common set-up: mbarriers, TMEM, and the F images and stage twiddles into
// SMEM by asynchronous bulk copies (issued by one thread, completing on the
// tables' mbarrier, the word after the TMEM slot) so that they overlap the
// first item's input copy; wait_tables() before the first use.  Every size
// is a multiple of 16 bytes (the images 64 r^2 bytes, the twiddle tables an
// even number of complex values).
// kernel_setup_start leaves the CTA unsynchronised, so that warp 0 can issue
// its first input copy (its mbarriers are initialised by then, in program
// order within warp 0) before kernel_setup_finish's CTA barrier.
template <int NWG, int THREADS>
__device__ __forceinline__ void kernel_setup_start(const float *bimg, int img_floats,
                                                   float *img, const float2 *tw_src0,
                                                   float2 *tw_dst0, int tw_n0,
                                                   const float2 *tw_src1, float2 *tw_dst1,
                                                   int tw_n1, uint64_t *mbar,
                                                   uint32_t *tmem_slot) {
  const int tid = threadIdx.x;
  uint64_t *tbar = mbar + 3 * NWG + 1;
  if (tid == 0) {
    for (int w = 0; w < 3 * NWG; ++w) mbar_init(smem_u32(mbar + w), 1);
    mbar_init(smem_u32(tbar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    const uint32_t bytes0 = (uint32_t)img_floats * 4u, bytes1 = (uint32_t)tw_n0 * 8u,
                   bytes2 = (uint32_t)tw_n1 * 8u;
    mbar_expect_tx(smem_u32(tbar), bytes0 + bytes1 + bytes2);
    tma_load_1d(smem_u32(img), bimg, bytes0, smem_u32(tbar));
    if (bytes1) tma_load_1d(smem_u32(tw_dst0), tw_src0, bytes1, smem_u32(tbar));
    if (bytes2) tma_load_1d(smem_u32(tw_dst1), tw_src1, bytes2, smem_u32(tbar));
  }
  if ((tid >> 5) == 0) {
    __syncwarp();
    tmem_alloc(smem_u32(tmem_slot), 512);
  }
}

__device__ __forceinline__ uint32_t kernel_setup_finish(const uint32_t *tmem_slot) {
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  return *tmem_slot;
}

template <int NWG, int THREADS>
__device__ __forceinline__ uint32_t kernel_setup(const float *bimg, int img_floats,
                                                 float *img, const float2 *tw_src0,
                                                 float2 *tw_dst0, int tw_n0,
                                                 const float2 *tw_src1, float2 *tw_dst1,
                                                 int tw_n1, uint64_t *mbar,
                                                 uint32_t *tmem_slot) {
  kernel_setup_start<NWG, THREADS>(bimg, img_floats, img, tw_src0, tw_dst0, tw_n0, tw_src1,
                                   tw_dst1, tw_n1, mbar, tmem_slot);
  return kernel_setup_finish(tmem_slot);
}

// Every thread, before the first use of the F images or stage twiddles.
__device__ __forceinline__ bool wait_tables(uint64_t *mbar, int nwg) {
  return mbar_wait_bounded(smem_u32(mbar + 3 * nwg + 1), 0);
}

// Leave: wait (bounded) for any copy still landing in this warpgroup's
// staging, then free TMEM.
__device__ __forceinline__ void kernel_teardown(uint32_t tbase, const WG &w, bool stg_pending,
                                                bool tws_pending) {
  // the first lane of the warp that issued the copies
  if (w.copy_lead && (threadIdx.x & 31) == 0) {
    if (stg_pending) mbar_wait_bounded(w.bar_stg, w.ph_stg);
    if (tws_pending) mbar_wait_bounded(w.bar_tws, w.ph_tws);
  }
  fence_before_sync();
  __syncthreads();
  if ((threadIdx.x >> 5) == 0) {
    fence_after_sync();
    tmem_dealloc(tbase, 512);
  }
}

template <int R, class SM, int GCOLS, int TW = 1>
__device__ __forceinline__ void init_wg(WG &w, uint32_t tbase, unsigned char *smem) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int wg = warp >> 2, team = wg / TW, wt = wg % TW;
  uint64_t *mbar = reinterpret_cast<uint64_t *>(smem + SM::OFF_BAR);
  w.rho = (wt * 4 + (warp & 3)) * 32 + lane;
  w.wg_lead = (warp & 3) == 0;
  w.team_lead = w.wg_lead && wt == 0;
  w.copy_lead = w.team_lead;
  w.slot = tbase + wg * GCOLS;
  w.lane_off = (uint32_t)((warp & 3) * 32) << 16;
  w.img_addr = smem_u32(smem);
  w.bar_mma = smem_u32(mbar + 3 * wg);
  // the team's copies complete on its first warpgroup's staging barriers
  w.bar_stg = smem_u32(mbar + 3 * (team * TW) + 1);
  w.bar_tws = smem_u32(mbar + 3 * (team * TW) + 2);
  w.bar_id = 1 + team;
  w.bar_count = 128 * TW;
  w.buf = reinterpret_cast<float2 *>(smem + SM::OFF_BUF) + team * SM::PTS;
  w.stg = reinterpret_cast<float2 *>(smem + SM::OFF_STG) + team * SM::PTS;
  w.tws = reinterpret_cast<float2 *>(smem + SM::OFF_TWS) + (SM::TWS_BYTES ? team * SM::PTS : 0);
  w.twb = reinterpret_cast<float2 *>(smem + SM::OFF_TWB) + team * SM::TWB_PER_WG;
  w.ph_mma = w.ph_stg = w.ph_tws = 0;
  // the transpose addressing needs the 1024-byte alignment the dynamic
  // shared memory is declared with; a base without it fails the launch
  w.fail = (smem_u32(smem) & 1023u) != 0;
  w.tws_inflight = false;
}

// ---------------------------------------------------------------- one pass
template <class G>
struct StaticNext {
  const PRun &P;
  const CUtensorMap *tm;
  long long next, nitems;
  bool issued;  // a copy for `next` is in flight
  __device__ void issue(const WG &w) {
    issued = next < nitems;
    if (issued) issue_input<G>(P, tm, G::TW == 1 && P.reverse ? nitems - 1 - next : next, w);
  }
  __device__ void publish() {}
  __device__ void after_load(const WG &) {}
  __device__ void before_store(WG &) {}
};

template <int R, int PREC, int S, int LO, int ROLE, int LP, bool CONV = false, int TW = 1>
__global__ void __launch_bounds__(
    Geo<R, S, LO, ROLE, LP,
        TW == 1 ? (CONV ? whole_k_nwg(R, ROLE) : pass_nwg(R, ROLE, S)) : 4, TW>::THREADS,
    1) dft_pass_kernel(const __grid_constant__ GArgs a) {
  using G =
      Geo<R, S, LO, ROLE, LP, TW == 1 ? (CONV ? whole_k_nwg(R, ROLE) : pass_nwg(R, ROLE, S)) : 4,
          TW>;
  static_assert(!CONV || ROLE == kSingle, "convolution rows are whole transforms");
  using SM = SmemLayout<R, G::NWG, G::TW_ENTRIES, CONV ? G::TW_ENTRIES : 0, G::TW_SMEM, G::TWB,
                        TW, G::KS>;
  extern __shared__ __align__(1024) unsigned char smem[];
  float2 *tw = reinterpret_cast<float2 *>(smem + SM::OFF_TW1);
  float2 *tw_inv = reinterpret_cast<float2 *>(smem + SM::OFF_TW2);
  uint64_t *mbar = reinterpret_cast<uint64_t *>(smem + SM::OFF_BAR);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mbar + 3 * G::NWG);
  const PRun &P = a.p[0];
  // a convolution row pass also holds the inverse stage twiddles (p[1])
  kernel_setup_start<G::NWG, G::THREADS>(
      a.bimg, (int)(SM::IMG / 4), reinterpret_cast<float *>(smem), P.tw_stage, tw,
      G::TW_ENTRIES, a.p[1].tw_stage, tw_inv, CONV ? G::TW_ENTRIES : 0, mbar, tmem_slot);
  WG w;
  init_wg<R, SM, G::GCOLS, TW>(w, 0, smem);  // TMEM slot set below
  // In a strided pass of two or more stages warp 1 issues the copies after
  // the first one (the inter-pass twiddles and the next input), beside warp
  // 0's products, which the other warps otherwise wait for at the next
  // barrier (measured: these passes 1 % faster; the others, and one-stage
  // strided passes, slower)
  if (ROLE == kFirst && S >= 2 && !G::KS && !CONV)
    w.copy_lead = (threadIdx.x >> 5) % (4 * TW) == 1;
#ifdef TCU_DFT_CHECKED
  w.err = a.err;
#endif

  const int team = (threadIdx.x >> 7) / TW;
  const long long nitems = (P.U + G::GG - 1) >> G::LOG2GG;
  const long long istride = (long long)gridDim.x * G::NTEAM;
  // team-major: with fewer items than SMs each CTA holds one item
  long long item = (long long)team * gridDim.x + blockIdx.x;
  StaticNext<G> nx{P, &a.tm_in, item, nitems, false};
  // item: position in this CTA's sequence; phys: the item processed there
  // (team passes always run forward: no reversal code in them)
  auto phys = [&](long long i) { return TW == 1 && P.reverse ? nitems - 1 - i : i; };
  // the first input copy of team 0 leaves with the tables (warp 0 set up its
  // mbarriers), the other teams' after the CTA barrier
  if (team == 0 && w.team_lead && item < nitems) issue_input<G>(P, &a.tm_in, phys(item), w);
  const uint32_t tbase = kernel_setup_finish(tmem_slot);
  w.slot = tbase + (uint32_t)((threadIdx.x >> 7) * G::GCOLS);
  if (team != 0 && w.team_lead && item < nitems) issue_input<G>(P, &a.tm_in, phys(item), w);
  // the tables have landed (the same answer in every thread of the team)
  if (named_bar_or(w.bar_id, w.bar_count, !wait_tables(mbar, G::NWG))) w.fail = true;
  while (item < nitems && !w.fail) {
    nx.next = item + istride;
    if constexpr (CONV)
      process_item_conv<G, PREC>(P, tw, tw_inv, phys(item), w, nx);
    else if constexpr (G::KS)
      process_item_ks<G, PREC>(P, tw, phys(item), w, nx);
    else
      // a strided pass writes the next pass's input: L2-cached stores keep
      // its latest part for the next pass (which starts there), streaming
      // stores otherwise
      process_item<G, PREC, ROLE == kFirst>(P, &a.tm_tw, tw, phys(item), w, nx);
    item += istride;
  }
  if (w.fail && w.rho == 0) atomicCAS(a.err, 0, TCU_DFT_ERR_TIMEOUT);
  // on failure a copy issued for the next item may still be landing
  kernel_teardown(tbase, w, w.fail && nx.issued, w.fail && w.tws_inflight);
}

// ------------------------------------------------------- fused two passes
__device__ __forceinline__ int ld_acquire(const int *p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void red_release_add(int *p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Queue position -> (pass, item).  Both passes have the same number of
// items per chunk, A = 2^lgA (every item is 128 r points).  Order:
// P1(0) .. P1(lag-1), then for c >= lag: P1(c), P2(c - lag); then the
// remaining P2 chunks.  Returns false past the end.
__device__ __forceinline__ bool decode_queue(const GArgs &a, long long pos, int &pass,
                                             long long &item, int &chunk) {
  const int lgA = a.log2_items_per_chunk;
  const long long A = 1ll << lgA;
  const int lag = a.lag, nc = a.nchunks;
  if (pos < ((long long)lag << lgA)) {
    pass = 0;
    chunk = (int)(pos >> lgA);
    item = pos;
    return true;
  }
  const long long p2 = pos - ((long long)lag << lgA);
  if (p2 < ((long long)(nc - lag) << (lgA + 1))) {
    const long long step = p2 >> (lgA + 1), off = p2 & (2 * A - 1);
    if (off < A) {
      pass = 0;
      chunk = (int)(lag + step);
      item = ((long long)chunk << lgA) + off;
    } else {
      pass = 1;
      chunk = (int)step;
      item = ((long long)chunk << lgA) + (off - A);
    }
    return true;
  }
  const long long p3 = p2 - ((long long)(nc - lag) << (lgA + 1));
  if (p3 < ((long long)lag << lgA)) {
    pass = 1;
    chunk = (int)(nc - lag + (p3 >> lgA));
    item = ((long long)chunk << lgA) + (p3 & (A - 1));
    return true;
  }
  return false;
}

struct __align__(8) FusedSched {  // per-warpgroup mailbox: the next item
  long long item;
  int pass;         // 0, 1, or -1 (queue exhausted)
  int chunk;
  int issued;       // its input copy is already in flight
  int pad;
};

struct QItem {
  long long item;
  int pass, chunk;
  bool valid;
};

// Next-item logic of the fused schedule, run by warp 0 of each warpgroup;
// its state is the same in all 32 lanes, except the results of the global
// atomic and the flag read, which lane 0 holds until they are needed.
// Items: cur (being processed), n1 (next), n2 (the one after).  During cur:
//   issue()   -- right after cur's first products: if n1's dependency value
//                (read one item earlier) says ready, issue n1's input copy;
//                claim the queue position of the item after n1 (atomicAdd,
//                its result is used only in publish());
//   publish() -- before cur's first epilogue barrier: publish the completion
//                of the previous item (red.release; every thread's stores of
//                it are ordered before by the barriers in between), tell the
//                warpgroup about n1, then decode n2 and start reading its
//                dependency flag (ld.acquire, used in the next issue()).
// So the latency of every atomic and flag read hides behind an item's work.
template <class G1, class G2>
struct FusedNext {
  const GArgs &a;
  FusedSched *box;
  QItem n1;
  int dep_raw;     // lane 0: value read from n1's dependency flag
  int dep_target;
  int pos2;        // lane 0: claimed queue position
  bool n1_issued;
  int *pend_flag;

  __device__ static bool lane0() { return (threadIdx.x & 31) == 0; }

  // A pass-1 item waits until the ring slot it overwrites has been drained
  // by pass 2; a pass-2 item until every pass-1 item of its transform has
  // been written.  Null flag: no dependency.
  __device__ const int *dep_flag(const QItem &q, int &target) const {
    if (q.pass == 0) {
      if (q.chunk < a.ring_chunks) return nullptr;
      target = 1 << a.log2_items_per_chunk;
      return a.counters + 1 + a.batch + (q.chunk - a.ring_chunks);
    }
    target = a.items1_per_tf;
    const long long u0 = q.item << G2::LOG2GG;
    return a.counters + 1 + (u0 >> G2::LOG2UPER);
  }

  __device__ void read_dep(const QItem &q) {
    dep_raw = 1;
    dep_target = 0;
    if (!q.valid) return;
    const int *flag = dep_flag(q, dep_target);
    if (flag && lane0()) dep_raw = ld_acquire(flag);
  }

  // Bounded wait (lane 0 polls) until q's dependency holds; uniform result.
  __device__ bool wait_deps(const QItem &q) const {
    int target = 0;
    const int *flag = dep_flag(q, target);
    int ok = 1;
    if (flag && lane0() && ld_acquire(flag) < target) {
      const unsigned long long t0 = global_ns();
      while (ld_acquire(flag) < target) {
        if (global_ns() - t0 > kWaitNs) {
          ok = 0;
          break;
        }
        __nanosleep(100);
      }
    }
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
  }

  __device__ QItem decode(long long pos) const {
    QItem q;
    q.valid = decode_queue(a, pos, q.pass, q.item, q.chunk);
    return q;
  }

  __device__ int claim() const {
    int p = 0;
    if (lane0()) p = atomicAdd(a.counters, 1);
    return p;
  }

  __device__ void issue_copy(const QItem &q, const WG &w) {
    fence_proxy_async_global();  // the acquire of its flag comes first
    if (q.pass == 0)
      issue_input<G1>(a.p[0], &a.tm_in, q.item, w);
    else
      issue_input<G2>(a.p[1], &a.tm_in, q.item, w);
  }

  __device__ void publish_pending() {
    if (pend_flag) {
      if (lane0()) red_release_add(pend_flag, 1);
      pend_flag = nullptr;
    }
  }

  __device__ void issue(const WG &w) {
    const int dep_val = __shfl_sync(0xffffffffu, dep_raw, 0);
    n1_issued = false;
    if (n1.valid && dep_val >= dep_target) {
      issue_copy(n1, w);
      n1_issued = true;
    }
    pos2 = claim();
  }

  __device__ void after_load(const WG &) {}
  __device__ void before_store(WG &) {}

  __device__ void publish() {
    publish_pending();
    if (lane0()) {
      box->item = n1.item;
      box->pass = n1.valid ? n1.pass : -1;
      box->chunk = n1.chunk;
      box->issued = n1_issued ? 1 : 0;
    }
    n1 = decode(__shfl_sync(0xffffffffu, pos2, 0));
    read_dep(n1);
  }
};

template <int R, int PREC, int S1, int S2>
__global__ void __launch_bounds__(
    Geo<R, S1, log2_radix(R) * S2, kFirst, 0, whole_k_nwg(R, kFirst)>::THREADS, 1)
    dft_fused_kernel(const __grid_constant__ GArgs a) {
  static_assert(S1 >= 2 && S2 >= 2, "the fused schedule needs an SMEM barrier per item");
  using G1 = Geo<R, S1, log2_radix(R) * S2, kFirst, 0, whole_k_nwg(R, kFirst)>;
  using G2 = Geo<R, S2, log2_radix(R) * S1, kSecond, 0, G1::NWG>;
  using SM = SmemLayout<R, G1::NWG, G1::TW_ENTRIES, G2::TW_ENTRIES, G1::TW_SMEM, G1::TWB>;
  constexpr int NWG = G1::NWG;
  extern __shared__ __align__(1024) unsigned char smem[];
  float2 *tw1 = reinterpret_cast<float2 *>(smem + SM::OFF_TW1);
  float2 *tw2 = reinterpret_cast<float2 *>(smem + SM::OFF_TW2);
  uint64_t *mbar = reinterpret_cast<uint64_t *>(smem + SM::OFF_BAR);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mbar + 3 * NWG);
  FusedSched *boxes = reinterpret_cast<FusedSched *>(smem + SM::OFF_SCHED);
  const uint32_t tbase = kernel_setup<NWG, G1::THREADS>(
      a.bimg, (int)(SM::IMG / 4), reinterpret_cast<float *>(smem), a.p[0].tw_stage, tw1,
      G1::TW_ENTRIES, a.p[1].tw_stage, tw2, G2::TW_ENTRIES, mbar, tmem_slot);
  WG w;
  init_wg<R, SM, G1::GCOLS>(w, tbase, smem);
#ifdef TCU_DFT_CHECKED
  w.err = a.err;
#endif
  const int wg = threadIdx.x >> 7;
  FusedSched *box = boxes + wg;

  FusedNext<G1, G2> nx{a, box};
  nx.pend_flag = nullptr;
  nx.n1_issued = false;

  // first item: claim it, wait for its dependencies, issue its copy; claim
  // the one after and start reading its dependency (warp 0)
  bool f = false;
  if (w.team_lead) {
    const QItem first = nx.decode(__shfl_sync(0xffffffffu, nx.claim(), 0));
    if (first.valid) {
      if (!nx.wait_deps(first)) f = true;
      else nx.issue_copy(first, w);
    }
    if (w.rho == 0) {
      box->item = first.item;
      box->pass = first.valid ? first.pass : -1;
      box->chunk = first.chunk;
      box->issued = first.valid && !f;
    }
    nx.n1 = nx.decode(__shfl_sync(0xffffffffu, nx.claim(), 0));
    nx.read_dep(nx.n1);
  }
  if (!wait_tables(mbar, NWG)) f = true;
  if (named_bar_or(w.bar_id, w.bar_count, f)) w.fail = true;

  bool stg_pending = false;
  while (!w.fail) {
    const long long item = box->item;
    const int pass = box->pass, chunk = box->chunk;
    const bool issued = box->issued != 0;
    if (pass < 0) break;
    if (!issued) {
      // its dependency was not ready at issue time: publish our own last
      // completion (it may be what it waits for; the barrier orders every
      // thread's stores of it first), wait, then copy
      bool ff = named_bar_or(w.bar_id, w.bar_count, false);
      if (w.team_lead) {
        nx.publish_pending();
        const QItem q{item, pass, chunk, true};
        if (!nx.wait_deps(q)) ff = true;
        else nx.issue_copy(q, w);
      }
      if (named_bar_or(w.bar_id, w.bar_count, ff)) {
        w.fail = true;
        break;
      }
    }
    if (pass == 0)
      process_item<G1, PREC, true>(a.p[0], &a.tm_tw, tw1, item, w, nx);
    else
      process_item<G2, PREC, false>(a.p[1], &a.tm_tw, tw2, item, w, nx);
    stg_pending = nx.n1_issued;
    if (w.fail) break;
    // the mailbox now names the next item; its completion is published
    // during the next item (after its first barrier), or below
    if (w.team_lead)
      nx.pend_flag = (pass == 0) ? a.counters + 1 + ((item << G1::LOG2GG) >> G1::LOG2UPER)
                                 : a.counters + 1 + a.batch + chunk;
  }
  // all stores of this warpgroup are issued: publish the last completion
  named_bar_or(w.bar_id, w.bar_count, false);
  if (w.team_lead) nx.publish_pending();
  if (w.rho == 0 && w.fail) atomicCAS(a.err, 0, TCU_DFT_ERR_TIMEOUT);
  kernel_teardown(tbase, w, w.fail && stg_pending, w.fail && w.tws_inflight);
}

// ------------------------------------------ one HBM pass on cluster pairs
// Both passes of a two-pass (four-step) transform in ONE launch, with the
// intermediate of each transform kept in L2 and every synchronisation local
// to a cluster of two CTAs.  Cluster c takes the transforms of pairs
// c, c + NC, c + 2 NC, ... (NC clusters; pair p holds transforms 2p, 2p+1),
// so its j-th transform is t_j = 2 (c + (j >> 1) NC) + (j & 1) and slot
// j & 1 of its two-transform scratch holds t_j's intermediate: pass-1 items
// write it with L2-cached stores, pass-2 items read it back by TMA.  HBM
// then sees each point read once and written once.
//
// Each transform has 2H pass-1 items and 2H pass-2 items; CTA rank k of the
// cluster takes items kH .. kH + H - 1 of both.  A CTA's sequence of items
// is P1(0) [H items], then for j = 0, 1, ...: P1(j+1) [H], P2(j) [H]; its
// warpgroups take positions round-robin.  Two mbarriers per slot in each
// CTA count items of both CTAs (2H arrivals per phase):
//   full[s]  -- pass-1 items of the slot's transform whose stores are
//               visible (released at cluster scope after the warpgroup's
//               barrier); a pass-2 item waits for it before copying;
//   empty[s] -- pass-2 items of the slot's transform whose input copy has
//               landed; a pass-1 item of transform j >= 2 waits for the
//               phase of transform j - 2 before storing into the slot.
// Every wait is for items at earlier positions of both CTAs' sequences, so
// the schedule cannot deadlock; every wait is bounded (ERR_TIMEOUT).
struct PairItem {
  int type;  // 0: pass-1 item, 1: pass-2 item
  int j;     // the CTA's transform (sequence index)
  int m;     // item within this CTA's half of the transform
  bool valid;
};

__device__ __forceinline__ PairItem pair_decode(long long pos, int H, int J) {
  PairItem it;
  it.valid = J > 0 && pos < 2ll * H * J;
  it.type = 0;
  it.j = 0;
  it.m = 0;
  if (!it.valid) return it;
  if (pos < H) {
    it.m = (int)pos;
    return it;
  }
  const long long q = pos - H;
  const int j = (int)(q / (2 * H)), r = (int)(q % (2 * H));
  if (j < J - 1 && r < H) {
    it.j = j + 1;
    it.m = r;
  } else {
    it.type = 1;
    it.j = j;
    it.m = j < J - 1 ? r - H : r;
  }
  return it;
}

template <class G1, class G2>
struct PairNext {
  const GArgs &a;
  const PRun &p1, &p2;
  uint32_t full_bar, empty_bar;  // this CTA's full[0], empty[0] (slot s at + 8 s)
  uint32_t peer;
  long long cid, nc;
  int crank, H, J;
  PairItem cur, nxt;
  bool issued;  // nxt's input copy is in flight

  __device__ long long tf(int j) const { return 2 * (cid + (long long)(j >> 1) * nc) + (j & 1); }
  __device__ long long gitem(const PairItem &it) const {
    return tf(it.j) * (2ll * H) + (long long)crank * H + it.m;
  }
  // parity of the phase of full[s] / empty[s] that belongs to transform j
  __device__ static uint32_t par(int j) { return (uint32_t)(j >> 1) & 1u; }

  int *mailbox;  // this warpgroup's word in SMEM: a pass-2 prefetch was issued

  uint64_t pol_first, pol_last;  // L2 policies: streaming data, the slots

  // the input x streams through L2 (first out); a slot is read back
  // without lowering its priority, since pass 1 rewrites it
  __device__ void copy(const PairItem &it, const WG &w) {
    if (it.type == 0) {
      issue_input<G1, true>(p1, &a.tm_in, gitem(it), w, pol_first);
    } else {
      fence_proxy_async_global();  // after the acquire of full[]
      issue_input<G2, true>(p2, nullptr, gitem(it), w, pol_last);
    }
  }
  // every thread of the warpgroup, once the staging buffer is free: warp 0
  // copies the next item's input -- a pass-1 item's always, a pass-2 item's
  // only if its transform's pass-1 items are all stored (a non-blocking
  // test; the answer reaches the other warps through the mailbox, read by
  // sync() after the warpgroup's next barrier)
  __device__ void issue(const WG &w) {
    issued = nxt.valid && nxt.type == 0;
    if (!nxt.valid || !w.team_lead) return;
    int ok = 1;
    if (nxt.type == 1) {
      if ((threadIdx.x & 31) == 0)
        ok = mbar_test_cluster(full_bar + 8 * (nxt.j & 1), par(nxt.j)) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if ((threadIdx.x & 31) == 0) *mailbox = ok;
    }
    if (ok) copy(nxt, w);
  }
  // every thread, after the warpgroup barrier that follows issue()
  __device__ void sync() {
    if (nxt.valid && nxt.type == 1) issued = *(volatile int *)mailbox != 0;
  }
  // warp 0, converged: bounded wait for a pass-2 item's dependency, then its
  // copy (the prefetch found the dependency unmet)
  __device__ bool wait_and_copy(const PairItem &it, const WG &w) {
    int ok = 1;
    if (it.type == 1 && (threadIdx.x & 31) == 0)
      ok = mbar_wait_cluster_bounded(full_bar + 8 * (it.j & 1), par(it.j)) ? 1 : 0;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (ok) copy(it, w);
    return ok != 0;
  }

  __device__ void publish() {}
  // a pass-2 item's input has landed in SMEM: its slot may be overwritten.
  // The arrival orders nothing but that copy, which has completed, so it is
  // relaxed (a release would wait for this warp's stores still in flight).
  __device__ void after_load(const WG &w) {
    if (cur.type == 1 && w.team_lead) {
      if (elect_one()) {
        const uint32_t b = empty_bar + 8 * (cur.j & 1);
        mbar_arrive_relaxed_local(b);
        mbar_arrive_relaxed_remote(mapa_shared(b, peer));
      }
      __syncwarp();
    }
  }
  // a pass-1 item of transform j >= 2 stores into the slot of j - 2 only
  // once every pass-2 item of j - 2 has copied it out
  __device__ void before_store(WG &w) {
    if (cur.type == 0 && cur.j >= 2 &&
        !mbar_wait_cluster_bounded(empty_bar + 8 * (cur.j & 1), par(cur.j - 2)))
      w.fail = true;
  }
  // pending publication of this warpgroup's pass-1 items of one transform
  int pend_j;
  uint32_t pend_count;  // 0: none
  // warp 0, converged, some time after the warpgroup's barrier that follows
  // the last of its `pend_count` pass-1 items of transform pend_j (their
  // stores have drained by then, so the fence is cheap): a release at
  // cluster scope, then pend_count arrivals on full[] of both CTAs
  __device__ void publish_full() {
    if (elect_one()) {
      fence_acq_rel_cluster();
      const uint32_t b = full_bar + 8 * (pend_j & 1);
      mbar_arrive_cluster_local_n(b, pend_count);
      mbar_arrive_cluster_remote_n(mapa_shared(b, peer), pend_count);
    }
    __syncwarp();
    pend_count = 0;
  }
};

// The inter-pass twiddles w_M^{k v} of this thread's last-stage outputs
// (k = klow + j r^(S-1), column v) from the L2-resident table A [k][vl];
// loaded while the last stage's products run.
template <class G>
__device__ __forceinline__ void out_twiddles(const PRun &P, long long item, const WG &w,
                                             float2 *tw) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  static_assert(G::TW_OUT && !G::TW2L, "one-level inter-pass table");
  int ul, q;
  row_of<G>(G::MODE_LAST, w.rho, ul, q);
  int klow = 0, vq = q;
#pragma unroll
  for (int i = 0; i < S - 1; ++i) {
    klow = (klow << G::LOG2R) | (vq & (R - 1));
    vq >>= G::LOG2R;
  }
  const long long u = (item << G::LOG2GG) + ul;
  const long long vl = u & ((1ll << G::LOG2VL) - 1);
  const long long goff = ((long long)klow << G::LOG2VL) + vl;
  constexpr long long TWG = 1ll << (G::LOG2VL + G::LOG2L - G::LOG2R);
#pragma unroll
  for (int j = 0; j < R; ++j)
    tw[j] = in_range(w, goff + j * TWG, (long long)G::L << G::LOG2VL) ? __ldg(P.tw_out + goff + j * TWG)
                                                                       : make_float2(1.f, 0.f);
}

// Last stage of a pass-1 item of the pair schedule: D -> registers, times
// the prefetched inter-pass twiddles, stores into the slot (last out of L2).
template <class G, int PREC>
__device__ __forceinline__ void pair_first_store(const PRun &P, long long item, const WG &w,
                                                 const float2 *tw, uint64_t pol) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  int ul, q;
  row_of<G>(G::MODE_LAST, w.rho, ul, q);
  const long long u = (item << G::LOG2GG) + ul;
  float d[2 * R];
  load_d_row<G, PREC>(w, d);
  if (u >= P.U) return;
  int klow = 0, vq = q;
#pragma unroll
  for (int i = 0; i < S - 1; ++i) {
    klow = (klow << G::LOG2R) | (vq & (R - 1));
    vq >>= G::LOG2R;
  }
  const long long b = u >> G::LOG2UPER;
  const long long v = u & ((1ll << G::LOG2UPER) - 1);
  float2 *dst = P.out + ((b & P.out_bmask) << G::LOG2NT) + v + klow * G::OUT_STRIDE;
  constexpr long long JS = G::OUT_STRIDE << (G::LOG2L - G::LOG2R);
  const long long doff = dst - P.out;
  const long long out_elems = (P.out_bmask + 1) << G::LOG2NT;
#pragma unroll
  for (int j = 0; j < R; ++j) {
    const float2 y = cmul(make_float2(d[2 * j], d[2 * j + 1]), tw[j]);
    if (in_range(w, doff + j * JS, out_elems)) st_global_hint(dst + j * JS, y, pol);
  }
}

// Last stage of a pass-2 item of the pair schedule: D -> registers ->
// natural-order output (first out of L2).
template <class G, int PREC>
__device__ __forceinline__ void pair_second_store(const PRun &P, long long item, const WG &w,
                                                  uint64_t pol) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  static_assert(G::MODE_LAST == kUF && !G::TW_OUT, "last pass of several");
  int ul, q;
  row_of<G>(G::MODE_LAST, w.rho, ul, q);
  const long long u = (item << G::LOG2GG) + ul;
  float d[2 * R];
  load_d_row<G, PREC>(w, d);
  if (u >= P.U) return;
  int klow = 0, vq = q;
#pragma unroll
  for (int i = 0; i < S - 1; ++i) {
    klow = (klow << G::LOG2R) | (vq & (R - 1));
    vq >>= G::LOG2R;
  }
  const long long b = u >> G::LOG2UPER;
  const long long v = u & ((1ll << G::LOG2UPER) - 1);
  float2 *dst = P.out + ((b & P.out_bmask) << G::LOG2NT) + v + klow * G::OUT_STRIDE;
  constexpr long long JS = G::OUT_STRIDE << (G::LOG2L - G::LOG2R);
  const long long doff = dst - P.out;
  const long long out_elems =
      P.out_bmask == -1 ? (P.U << G::LOG2L) : ((P.out_bmask + 1) << G::LOG2NT);
#pragma unroll
  for (int j = 0; j < R; ++j)
    if (in_range(w, doff + j * JS, out_elems))
      st_global_hint(dst + j * JS, make_float2(d[2 * j], d[2 * j + 1]), pol);
}

// One item of the pair schedule (two stages): TYPE 0 a pass-1 item (input
// staged by TMA from HBM, output into the slot), TYPE 1 a pass-2 item
// (input staged by TMA from the slot, output to HBM).  `mid` prefetches the
// next item's input into the staging buffer once it is free.
template <class G, int PREC, int TYPE, class Mid>
__device__ __forceinline__ void process_pair_item(const PRun &P, const float2 *tws,
                                                  long long item, WG &w, Mid &mid) {
  constexpr int R = 1 << G::LOG2R;
  constexpr int S = G::LOG2L / G::LOG2R;
  static_assert(S == 2, "two stages per pass");
  if (!mbar_wait_bounded(w.bar_stg, w.ph_stg)) w.fail = true;
  w.ph_stg ^= 1;
  // a pass-2 item's input has landed: its slot may be overwritten
  if (TYPE == 1) mid.after_load(w);
  {
    float2 x[R];
    staged_row<G>(w, x);
#pragma unroll
    for (int c = 0; c < R; c += 8)
      split_store8<PREC>(x + c, w.slot + w.lane_off + a_cols8(PREC) * c / 8,
                         w.slot + G::Q + w.lane_off + a_cols8(PREC) * c / 8);
  }
  tmem_wait_st();
  fence_before_sync();
  if (named_bar_or(w.bar_id, w.bar_count, w.fail)) {
    w.fail = true;
    return;
  }
  if (w.wg_lead) {
    fence_after_sync();
    issue_stage<R, PREC>(w.slot, w.img_addr, w.bar_mma);
    // the previous pass-1 items' stores have had an item's time to drain
    if (mid.pend_count) mid.publish_full();
  }
  if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
  w.ph_mma ^= 1;
  fence_after_sync();
  // the staging buffer is free: the next item's copy
  mid.issue(w);
  stage_epilogue<G, PREC, 1>(P, tws, w);
  fence_before_sync();
  named_bar_or(w.bar_id, w.bar_count, false);
  mid.sync();
  stage_rows<G, PREC, 2>(P, w);
  tmem_wait_st();
  fence_before_sync();
  if (named_bar_or(w.bar_id, w.bar_count, w.fail)) {
    w.fail = true;
    return;
  }
  if (w.wg_lead) {
    fence_after_sync();
    issue_stage<R, PREC>(w.slot, w.img_addr + P.last_img, w.bar_mma);
  }
  if constexpr (TYPE == 0) {
    float2 tw[R];
    out_twiddles<G>(P, item, w, tw);
    if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
    w.ph_mma ^= 1;
    fence_after_sync();
    mid.before_store(w);
    pair_first_store<G, PREC>(P, item, w, tw, mid.pol_last);
  } else {
    if (!mbar_wait_bounded(w.bar_mma, w.ph_mma)) w.fail = true;
    w.ph_mma ^= 1;
    fence_after_sync();
    pair_second_store<G, PREC>(P, item, w, mid.pol_first);
  }
}

template <int R, int S1, int S2>
struct PairLayout {
  using G1 = Geo<R, S1, log2_radix(R) * S2, kFirst, 0, whole_k_nwg(R, kFirst)>;
  // no twiddle staging: pass-1 items read their inter-pass twiddles from
  // the L2-resident table while their last products run
  using SM = SmemLayout<R, G1::NWG, G1::TW_ENTRIES, Geo<R, S2, log2_radix(R) * S1, kSecond, 0,
                                                        G1::NWG>::TW_ENTRIES,
                        false, 0>;
  static constexpr size_t OFF_PBAR = (SM::BYTES + 15) / 16 * 16;  // full[2], empty[2]
  static constexpr size_t OFF_MBOX = OFF_PBAR + 32;               // a word per warpgroup
  static constexpr size_t OFF_PRUN = OFF_MBOX + 16 * 4;           // per-CTA PRun copies
  static constexpr size_t BYTES = OFF_PRUN + 2 * sizeof(PRun);
  static_assert(BYTES <= 227 * 1024, "shared memory budget");
};

template <int R, int PREC, int S1, int S2>
__global__ void __launch_bounds__(
    Geo<R, S1, log2_radix(R) * S2, kFirst, 0, whole_k_nwg(R, kFirst)>::THREADS, 1)
    dft_pair_kernel(const __grid_constant__ GArgs a) {
  static_assert(S1 >= 2 && S2 >= 2, "the pair schedule needs an SMEM barrier per item");
  using PL = PairLayout<R, S1, S2>;
  using G1 = typename PL::G1;
  using G2 = Geo<R, S2, log2_radix(R) * S1, kSecond, 0, G1::NWG>;
  using SM = typename PL::SM;
  constexpr int NWG = G1::NWG;
  extern __shared__ __align__(1024) unsigned char smem[];
  float2 *tw1 = reinterpret_cast<float2 *>(smem + SM::OFF_TW1);
  float2 *tw2 = reinterpret_cast<float2 *>(smem + SM::OFF_TW2);
  uint64_t *mbar = reinterpret_cast<uint64_t *>(smem + SM::OFF_BAR);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mbar + 3 * NWG);
  uint64_t *pbar = reinterpret_cast<uint64_t *>(smem + PL::OFF_PBAR);
  PRun *prun = reinterpret_cast<PRun *>(smem + PL::OFF_PRUN);
  // H items per CTA and pass of a transform, a multiple of the warpgroups
  // (every warpgroup takes the same number of a transform's pass-1 items)
  const int H = a.items1_per_tf / 2;
  const long long cid = cluster_id_x(), nc = nclusters_x();
  const int crank = (int)cluster_ctarank();
  if (threadIdx.x == 0) {
    for (int i = 0; i < 4; ++i) mbar_init(smem_u32(pbar + i), 2 * H);
    // this cluster's two slots: pass-1 output (slot t & 1), pass-2 input
    const long long n = 1ll << G1::LOG2NT;
    prun[0] = a.p[0];
    prun[0].out = a.p[0].out + cid * 2 * n;
    prun[1] = a.p[1];
    prun[1].in = a.p[1].in + cid * 2 * n;
  }
  const uint32_t tbase = kernel_setup<NWG, G1::THREADS>(
      a.bimg, (int)(SM::IMG / 4), reinterpret_cast<float *>(smem), a.p[0].tw_stage, tw1,
      G1::TW_ENTRIES, a.p[1].tw_stage, tw2, G2::TW_ENTRIES, mbar, tmem_slot);
  // the peer's barriers exist before any arrival on them
  cluster_sync_all();
  WG w;
  init_wg<R, SM, G1::GCOLS>(w, tbase, smem);
#ifdef TCU_DFT_CHECKED
  w.err = a.err;
#endif
  // transforms of this cluster: t_j < batch for j < J
  int J = 0;
  {
    const long long pairs = (a.batch + 1) / 2;
    if (cid < pairs) {
      const long long np = (pairs - 1 - cid) / nc + 1;  // pairs of this cluster
      J = (int)(2 * np);
      if (2 * (cid + (np - 1) * nc) + 1 >= a.batch) --J;  // a last pair of one
    }
  }
  PairNext<G1, G2> nx{a,     prun[0], prun[1], smem_u32(pbar), smem_u32(pbar + 2),
                      (uint32_t)(crank ^ 1), cid, nc, crank, H, J};
  nx.issued = false;
  const int wg = threadIdx.x >> 7;
  nx.mailbox = reinterpret_cast<int *>(smem + PL::OFF_MBOX) + wg;
  long long pos = wg;
  nx.cur = pair_decode(pos, H, J);
  // the first items are pass-1 items: their copies need no wait.  Every
  // later pass-1 item's copy is issued during the item before it.  All
  // control flow below is the same in the four warps of a warpgroup (the
  // warpgroup's named barriers must match).
  nx.pend_count = 0;
  nx.pol_first = l2_policy_evict_first();
  nx.pol_last = l2_policy_evict_last();
  nx.issued = nx.cur.valid && nx.cur.type == 0;
  if (nx.issued && w.team_lead) nx.copy(nx.cur, w);
  if (!wait_tables(mbar, NWG)) w.fail = true;
  // a uniform failure state before the first barrier
  if (named_bar_or(w.bar_id, w.bar_count, w.fail)) w.fail = true;
  bool stg_pending = nx.issued;
  while (nx.cur.valid && !w.fail) {
    nx.nxt = pair_decode(pos + NWG, H, J);
    if (nx.cur.type == 0) {
      process_pair_item<G1, PREC, 0>(prun[0], tw1, nx.gitem(nx.cur), w, nx);
      // every thread's stores of the item; after this warpgroup's last
      // pass-1 item of the transform (items m, m - NWG, ... of the H
      // consecutive positions of its pass-1 items) the arrivals of all of
      // them on full[]
      if (named_bar_or(w.bar_id, w.bar_count, w.fail)) w.fail = true;
      if (nx.cur.m + NWG >= H) {
        nx.pend_j = nx.cur.j;
        nx.pend_count = (uint32_t)(nx.cur.m / NWG + 1);
      }
    } else {
      process_pair_item<G2, PREC, 1>(prun[1], tw2, nx.gitem(nx.cur), w, nx);
      if (named_bar_or(w.bar_id, w.bar_count, w.fail)) w.fail = true;
    }
    stg_pending = nx.issued;
    if (w.fail) break;
    pos += NWG;
    nx.cur = nx.nxt;
    if (nx.cur.valid && !nx.issued) {
      // a pass-2 item whose dependency was unmet at prefetch time: publish
      // this warpgroup's own pending pass-1 items (it may be waiting for
      // them), wait (bounded), then copy; the same branch in every warp
      bool f = false;
      if (w.team_lead && nx.pend_count) nx.publish_full();
      if (w.team_lead) f = !nx.wait_and_copy(nx.cur, w);
      if (named_bar_or(w.bar_id, w.bar_count, f)) {
        w.fail = true;
        break;
      }
      stg_pending = true;
    }
  }
  // a last publication (after the last item nobody waits for it, but the
  // arrivals keep the barriers' counts whole)
  if (!w.fail && w.team_lead && nx.pend_count) nx.publish_full();
  if (w.fail && w.rho == 0) atomicCAS(a.err, 0, TCU_DFT_ERR_TIMEOUT);
  // leave: copies of this warpgroup still landing (on failure), then the
  // cluster -- the peer may arrive on this CTA's barriers until it is done
  if (w.rho == 0 && w.fail) {
    if (stg_pending) mbar_wait_bounded(w.bar_stg, w.ph_stg);
    if (w.tws_inflight) mbar_wait_bounded(w.bar_tws, w.ph_tws);
  }
  fence_before_sync();
  __syncthreads();
  cluster_sync_all();
  if ((threadIdx.x >> 5) == 0) {
    fence_after_sync();
    tmem_dealloc(tbase, 512);
  }
}

}  // namespace tcu
