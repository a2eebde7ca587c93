// grid_kernels.cu -- the element-wise steps of the stencil path of
// arXiv 1908.06649, Sec. 4.6 (Lemmas 1 and 2) around the 2-D DFTs: placing
// the 3 x 3 stencil polynomial on a grid, the pointwise power of its
// spectrum, the flipped weight kernel W', and the gather / extract of the
// 3k x 3k tiles A'_{r,c}.  All are HBM-bound index maps (no contraction),
// so they are plain coalesced CUDA kernels: one thread per output element,
// grids in multiples of the SM count.
#include <cuda_runtime.h>
#include <stdint.h>

#include "launch.h"

namespace tcu {
namespace {

constexpr int kBlock = 256;

// Signed offset of grid index i on a periodic axis of length N: i for
// i <= N/2, i - N above.
__device__ __forceinline__ long long centred(long long i, long long N) {
  return i <= N / 2 ? i : i - N;
}

// P(x, y) = sum w3[a+1][b+1] x^a y^b on an Nw x Nw periodic grid:
// g[a mod Nw][b mod Nw] = w3[a+1][b+1] for a, b in {-1, 0, 1}, 0 elsewhere.
__global__ void place_poly_kernel(float2 *g, long long Nw, Stencil3 w) {
  const long long count = Nw * Nw;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < count;
       e += (long long)gridDim.x * blockDim.x) {
    const long long a = centred(e / Nw, Nw), b = centred(e % Nw, Nw);
    float v = 0.f;
    if (a >= -1 && a <= 1 && b >= -1 && b <= 1) v = w.w[(a + 1) * 3 + (b + 1)];
    g[e] = make_float2(v, 0.f);
  }
}

// g <- g^k elementwise (complex, by repeated squaring).
__global__ void cpow_kernel(float2 *g, long long count, int k) {
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < count;
       e += (long long)gridDim.x * blockDim.x) {
    float2 base = g[e], acc = make_float2(1.f, 0.f);
    for (int m = k; m > 0; m >>= 1) {
      if (m & 1) acc = cmul(acc, base);
      base = cmul(base, base);
    }
    g[e] = acc;
  }
}

// W[(k + a)(2k + 1) + (k + b)] = Re g[a mod Nw][b mod Nw], |a|, |b| <= k.
__global__ void extract_weights_kernel(float *W, const float2 *g, long long Nw, int k) {
  const long long side = 2 * k + 1, count = side * side;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < count;
       e += (long long)gridDim.x * blockDim.x) {
    const long long a = e / side - k, b = e % side - k;
    const long long ia = (a + Nw) % Nw, ib = (b + Nw) % Nw;
    W[e] = g[ia * Nw + ib].x;
  }
}

// The convolution kernel of Lemma 1 on an N x N periodic grid: w[-a mod N]
// [-b mod N] = W[k + a][k + b] for |a|, |b| <= k (W flipped and padded with
// zeros), so that (x (*) w)[i][j] = sum W[k+a][k+b] x[i+a][j+b].  W is read
// from the Nw x Nw grid of the weight computation.
__global__ void place_kernel_kernel(float2 *w, long long N, const float2 *g, long long Nw,
                                    int k) {
  const long long count = N * N;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < count;
       e += (long long)gridDim.x * blockDim.x) {
    const long long a = -centred(e / N, N), b = -centred(e % N, N);
    float v = 0.f;
    if (a >= -k && a <= k && b >= -k && b <= k) v = g[((a + Nw) % Nw) * Nw + (b + Nw) % Nw].x;
    w[e] = make_float2(v, 0.f);
  }
}

// Tile (r, c) of the side x side grid A as the N x N complex array whose
// top-left (B + 2k) x (B + 2k) block is the window A[rB - k .. rB + B + k)
// [cB - k .. cB + B + k) (zero outside A) and whose other entries are 0: the
// input of output block (r, c) of B x B points.  B = k is Lemma 1's tile
// A'_{r,c} (3k x 3k); the plan takes B = N - 2k, the largest block whose
// window still fits N without wrapping.  Blocks of 32 x 8 threads, one per
// tile (blockIdx.x) and chunk of kRowChunk tile rows (blockIdx.y): rows by
// threadIdx.y, column pairs by threadIdx.x (one 16-byte store of two complex
// values: N is even, so every pair is 16-byte aligned), so reads of A and
// writes of the tile are contiguous along the columns.
constexpr int kRowChunk = 32;

__global__ void gather_tiles_kernel(float2 *tiles, const float *A, long long side, int k,
                                    int N, int B, long long tpr) {
  const long long t = blockIdx.x;
  const long long r0 = (t / tpr) * B - k, c0 = (t % tpr) * B - k;
  const int win = B + 2 * k;
  float4 *dst = reinterpret_cast<float4 *>(tiles + t * N * N);
  const int i1 = min(N, (int)(blockIdx.y + 1) * kRowChunk);
  for (int i = blockIdx.y * kRowChunk + threadIdx.y; i < i1; i += blockDim.y) {
    const long long gi = r0 + i;
    const bool row_in = i < win && gi >= 0 && gi < side;
    for (int j = 2 * threadIdx.x; j < N; j += 2 * blockDim.x) {
      const long long gj = c0 + j;
      float v0 = 0.f, v1 = 0.f;
      if (row_in && j < win && gj >= 0 && gj < side) v0 = __ldg(A + gi * side + gj);
      if (row_in && j + 1 < win && gj + 1 >= 0 && gj + 1 < side)
        v1 = __ldg(A + gi * side + gj + 1);
      __stcs(dst + ((long long)i * N + j) / 2, make_float4(v0, 0.f, v1, 0.f));
    }
  }
}

// A_k[rB + i][cB + j] = Re tile_{r,c}[k + i][k + j] for i, j < B inside the
// grid (the last blocks of a row or column may be cut): one thread block per
// tile and chunk of kRowChunk block rows, contiguous along the columns.
__global__ void extract_tiles_kernel(float *Ak, const float2 *tiles, long long side, int k,
                                     int N, int B, long long tpr) {
  const long long t = blockIdx.x;
  const long long r0 = (t / tpr) * B, c0 = (t % tpr) * B;
  const float2 *src = tiles + t * N * N + (long long)k * N + k;
  const int i1 = min(B, (int)(blockIdx.y + 1) * kRowChunk);
  for (int i = blockIdx.y * kRowChunk + threadIdx.y; i < i1 && r0 + i < side; i += blockDim.y)
    for (int j = threadIdx.x; j < B && c0 + j < side; j += blockDim.x)
      Ak[(r0 + i) * side + c0 + j] = __ldcs(src + (long long)i * N + j).x;
}

// out[b][j][i] = in[b][i][j] for n1 x n2 arrays: 32 x 32 tiles through
// shared memory (a column of 33 for conflict-free reads of the transposed
// tile), blocks of 32 x 8 threads; both the read of `in` and the write of
// `out` run along contiguous rows of 32 complex values.  The grid walks
// every (array, tile) pair.
constexpr int kTile = 32;

__global__ void transpose_kernel(float2 *out, const float2 *in, long long batch, long long n1,
                                 long long n2) {
  __shared__ float2 t[kTile][kTile + 1];
  const long long ti = (n1 + kTile - 1) / kTile, tj = (n2 + kTile - 1) / kTile;
  const long long total = batch * ti * tj;
  for (long long tile = blockIdx.x; tile < total; tile += gridDim.x) {
    const long long b = tile / (ti * tj), rem = tile % (ti * tj);
    const long long i0 = (rem / tj) * kTile, j0 = (rem % tj) * kTile;
    const float2 *src = in + b * n1 * n2;
    float2 *dst = out + b * n1 * n2;
    for (int y = threadIdx.y; y < kTile; y += blockDim.y) {
      const long long i = i0 + y, j = j0 + threadIdx.x;
      if (i < n1 && j < n2) t[y][threadIdx.x] = __ldcs(src + i * n2 + j);
    }
    __syncthreads();
    for (int y = threadIdx.y; y < kTile; y += blockDim.y) {
      const long long j = j0 + y, i = i0 + threadIdx.x;
      if (i < n1 && j < n2) __stcs(dst + j * n1 + i, t[threadIdx.x][y]);
    }
    __syncthreads();
  }
}

// x[b][e] *= spec[e] for every array b of n complex values.
__global__ void spectrum_product_kernel(float2 *x, const float2 *spec, long long batch,
                                        long long n) {
  const long long count = batch * n;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < count;
       e += (long long)gridDim.x * blockDim.x)
    x[e] = cmul(x[e], __ldg(spec + e % n));
}

unsigned grid_for(long long count, int num_sms) {
  long long blocks = (count + kBlock - 1) / kBlock;
  const long long cap = (long long)num_sms * 8;  // 8 resident 256-thread blocks per SM
  if (blocks > cap) blocks = cap;
  return (unsigned)(blocks < 1 ? 1 : blocks);
}

}  // namespace

cudaError_t launch_place_poly(float2 *g, long long Nw, const Stencil3 &w, int num_sms,
                              cudaStream_t st) {
  place_poly_kernel<<<grid_for(Nw * Nw, num_sms), kBlock, 0, st>>>(g, Nw, w);
  return cudaGetLastError();
}

cudaError_t launch_cpow(float2 *g, long long count, int k, int num_sms, cudaStream_t st) {
  cpow_kernel<<<grid_for(count, num_sms), kBlock, 0, st>>>(g, count, k);
  return cudaGetLastError();
}

cudaError_t launch_extract_weights(float *W, const float2 *g, long long Nw, int k,
                                   int num_sms, cudaStream_t st) {
  const long long side = 2 * k + 1;
  extract_weights_kernel<<<grid_for(side * side, num_sms), kBlock, 0, st>>>(W, g, Nw, k);
  return cudaGetLastError();
}

cudaError_t launch_place_kernel(float2 *w, long long N, const float2 *g, long long Nw, int k,
                                int num_sms, cudaStream_t st) {
  place_kernel_kernel<<<grid_for(N * N, num_sms), kBlock, 0, st>>>(w, N, g, Nw, k);
  return cudaGetLastError();
}

cudaError_t launch_transpose(float2 *out, const float2 *in, long long batch, long long n1,
                             long long n2, int num_sms, cudaStream_t st) {
  const long long tiles = batch * ((n1 + kTile - 1) / kTile) * ((n2 + kTile - 1) / kTile);
  const long long cap = (long long)num_sms * 8;
  const unsigned grid = (unsigned)(tiles < cap ? tiles : cap);
  transpose_kernel<<<grid, dim3(kTile, 8), 0, st>>>(out, in, batch, n1, n2);
  return cudaGetLastError();
}

cudaError_t launch_spectrum_product(float2 *x, const float2 *spec, long long batch,
                                    long long n, int num_sms, cudaStream_t st) {
  spectrum_product_kernel<<<grid_for(batch * n, num_sms), kBlock, 0, st>>>(x, spec, batch, n);
  return cudaGetLastError();
}

cudaError_t launch_gather_tiles(float2 *tiles, const float *A, long long side, int k,
                                long long N, int B, int num_sms, cudaStream_t st) {
  const long long tpr = (side + B - 1) / B;
  const dim3 grid((unsigned)(tpr * tpr), (unsigned)((N + kRowChunk - 1) / kRowChunk));
  gather_tiles_kernel<<<grid, dim3(32, 8), 0, st>>>(tiles, A, side, k, (int)N, B, tpr);
  return cudaGetLastError();
}

cudaError_t launch_extract_tiles(float *Ak, const float2 *tiles, long long side, int k,
                                 long long N, int B, int num_sms, cudaStream_t st) {
  const long long tpr = (side + B - 1) / B;
  const dim3 grid((unsigned)(tpr * tpr), (unsigned)((B + kRowChunk - 1) / kRowChunk));
  extract_tiles_kernel<<<grid, dim3(32, 8), 0, st>>>(Ak, tiles, side, k, (int)N, B, tpr);
  return cudaGetLastError();
}

}  // namespace tcu

// ---------------------------------------------------------- mixed radix
// The q-point pass of a mixed-radix transform n = q R^k (q = 2 .. 16, any
// integer): the four-step split n = q x n2 with the q-point DFTs over the
// stride-n2 columns done on the CUDA cores -- for q <= 16 a tensor-core
// product would be mostly padding -- straight from the definition
// y_k = sum_a x_a w_q^{a k}, then the inter-pass twiddle w_n^{k v} from the
// two-level tables A[k][vl], B[vh][k] (v = vh 256 + vl).  One thread per
// column (b, v), v fastest: every load and store is coalesced.
namespace tcu {
namespace {

template <int Q>
__global__ void radix_q_kernel(const float2 *x, float2 *out, long long batch, int log2n2,
                               const float2 *twA, const float2 *twB, RootsQ roots) {
  const long long n2 = 1ll << log2n2, n = Q * n2, count = batch * n2;
  const int log2vl = log2n2 > 8 ? 8 : log2n2;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < count;
       e += (long long)gridDim.x * blockDim.x) {
    const long long b = e >> log2n2, v = e & (n2 - 1);
    const float2 *src = x + b * n + v;
    float2 a[Q];
#pragma unroll
    for (int i = 0; i < Q; ++i) a[i] = __ldcs(src + i * n2);
    const long long vl = v & ((1ll << log2vl) - 1), vh = v >> log2vl;
    float2 *dst = out + b * n + v;
#pragma unroll
    for (int k = 0; k < Q; ++k) {
      float2 y = a[0];
#pragma unroll
      for (int i = 1; i < Q; ++i) {
        const float2 w = roots.w[(i * k) % Q];
        y.x = fmaf(a[i].x, w.x, fmaf(-a[i].y, w.y, y.x));
        y.y = fmaf(a[i].x, w.y, fmaf(a[i].y, w.x, y.y));
      }
      float2 tw = __ldg(twA + ((long long)k << log2vl) + vl);
      if (log2n2 > 8) tw = cmul(tw, __ldg(twB + vh * Q + k));
      __stcs(dst + k * n2, cmul(y, tw));
    }
  }
}

}  // namespace

cudaError_t launch_radix_q(int q, const float2 *x, float2 *out, long long batch, int log2n2,
                           const float2 *twA, const float2 *twB, const RootsQ &roots,
                           int num_sms, cudaStream_t st) {
  const unsigned grid = grid_for(batch << log2n2, num_sms);
  switch (q) {
    case 2: radix_q_kernel<2><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 3: radix_q_kernel<3><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 4: radix_q_kernel<4><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 5: radix_q_kernel<5><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 6: radix_q_kernel<6><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 7: radix_q_kernel<7><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 8: radix_q_kernel<8><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 9: radix_q_kernel<9><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 10: radix_q_kernel<10><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 11: radix_q_kernel<11><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 12: radix_q_kernel<12><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 13: radix_q_kernel<13><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 14: radix_q_kernel<14><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 15: radix_q_kernel<15><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    case 16: radix_q_kernel<16><<<grid, kBlock, 0, st>>>(x, out, batch, log2n2, twA, twB, roots); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace tcu
