/*
 * Oracle for the batched complex DFT -- TEST INFRASTRUCTURE ONLY.
 *
 * This file is the plain, slow, fp64 CPU statement of what the GPU path
 * computes.  It shares no code, header, table or constant with the CUDA
 * library: it is built on its own (gcc) and only tests/, the smoke check and
 * the CPU-baseline leg of the benchmark may load it.
 *
 * What it computes (arXiv 1908.06649, Sec. 4.5):
 *   The DFT of an n-vector x is the product y = x^T W with the symmetric
 *   Fourier matrix W[r][c] = exp(-(2 pi i / n) r c).  So, entry by entry,
 *       y_k = sum_{j<n} x_j exp(sign * 2 pi i * j k / n),  sign = -1 (forward).
 *   The paper defines only the forward transform.  The inverse used here is
 *   the usual one: sign = +1 and a factor 1/n (applied by the caller through
 *   the `scale` argument).
 *
 * Two independent routes are provided:
 *   oracle_dft_direct : the definition written out, O(n^2); the angle index
 *                       (j*k) is reduced mod n before cos/sin, in fp64.
 *   oracle_fft_radix2 : a recursive decimation-in-time radix-2 FFT (the
 *                       textbook even/odd split), fp64, with every twiddle
 *                       taken from cos/sin of 2 pi t / m directly (no
 *                       recurrence).  It is NOT the paper's radix-sqrt(m)
 *                       algorithm, so the two oracles and the GPU path share
 *                       no decomposition either.
 *
 * Data: interleaved complex128 (re, im) arrays, transform-major
 * (x[2*(b*n + j)] = Re, x[2*(b*n + j) + 1] = Im).
 *
 * Parity pins: see tests/test_oracle.py (closed forms, Parseval, linearity,
 * Hermitian symmetry, inverse round trip, shift theorem, brute force on tiny
 * n, agreement of the two routes, numpy's pocketfft as a library special
 * case, and hand-derived golden vectors).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifndef M_PI
#define M_PI 3.14159265358979323846
#endif

/* ---- direct definition (Sec. 4.5: y = x^T W, W[r][c] = e^{-2 pi i rc/n}) ---- */
static void dft_direct_one(const double *x, double *y, int64_t n, int sign,
                           double scale) {
  for (int64_t k = 0; k < n; ++k) {
    double acc_re = 0.0, acc_im = 0.0;
    for (int64_t j = 0; j < n; ++j) {
      /* j*k < n^2 <= 2^48 for every n this oracle is asked for */
      int64_t m = (j * k) % n;
      double ang = (double)sign * 2.0 * M_PI * (double)m / (double)n;
      double c = cos(ang), s = sin(ang);
      double xr = x[2 * j], xi = x[2 * j + 1];
      acc_re += xr * c - xi * s;
      acc_im += xr * s + xi * c;
    }
    y[2 * k] = acc_re * scale;
    y[2 * k + 1] = acc_im * scale;
  }
}

/* ---- independent route: recursive radix-2 decimation in time ----
 * DFT_m(x)[k]       = E[k] + w_m^k O[k]
 * DFT_m(x)[k + m/2] = E[k] - w_m^k O[k],   k < m/2,
 * with E, O the DFTs of the even- and odd-indexed halves and
 * w_m = exp(sign * 2 pi i / m). */
static void fft_rec(const double *x, int64_t stride, double *y, int64_t m,
                    int sign) {
  if (m == 1) {
    y[0] = x[0];
    y[1] = x[1];
    return;
  }
  int64_t h = m / 2;
  fft_rec(x, 2 * stride, y, h, sign);               /* evens -> y[0, h)  */
  fft_rec(x + 2 * stride, 2 * stride, y + 2 * h, h, sign); /* odds -> y[h, m) */
  for (int64_t k = 0; k < h; ++k) {
    double ang = (double)sign * 2.0 * M_PI * (double)k / (double)m;
    double c = cos(ang), s = sin(ang);
    double er = y[2 * k], ei = y[2 * k + 1];
    double orr = y[2 * (k + h)], oi = y[2 * (k + h) + 1];
    double tr = orr * c - oi * s, ti = orr * s + oi * c;
    y[2 * k] = er + tr;
    y[2 * k + 1] = ei + ti;
    y[2 * (k + h)] = er - tr;
    y[2 * (k + h) + 1] = ei - ti;
  }
}

static void fft_radix2_one(const double *x, double *y, int64_t n, int sign,
                           double scale) {
  fft_rec(x, 1, y, n, sign);
  if (scale != 1.0)
    for (int64_t i = 0; i < 2 * n; ++i) y[i] *= scale;
}

/* ---- batch driver: transforms split across pthreads ---- */
typedef struct {
  const double *x;
  double *y;
  int64_t n, b0, b1;
  int sign, route;
  double scale;
} job_t;

static void *run_job(void *arg) {
  job_t *j = (job_t *)arg;
  for (int64_t b = j->b0; b < j->b1; ++b) {
    const double *xb = j->x + 2 * b * j->n;
    double *yb = j->y + 2 * b * j->n;
    if (j->route == 0)
      dft_direct_one(xb, yb, j->n, j->sign, j->scale);
    else
      fft_radix2_one(xb, yb, j->n, j->sign, j->scale);
  }
  return NULL;
}

static int is_pow2(int64_t n) { return n > 0 && (n & (n - 1)) == 0; }

/* route 0 = direct definition, 1 = radix-2 FFT.  Returns the number of
 * threads used, or -1 on bad arguments. */
static int run_batch(const double *x, double *y, int64_t n, int64_t batch,
                     int sign, double scale, int threads, int route) {
  if (n < 1 || batch < 0 || (sign != 1 && sign != -1)) return -1;
  if (route == 1 && !is_pow2(n)) return -1;
  if (x == y) return -1; /* out-of-place only */
  if (threads < 1) threads = 1;
  if (threads > batch) threads = (int)(batch > 0 ? batch : 1);
  if (threads > 256) threads = 256;
  job_t jobs[256];
  pthread_t tid[256];
  int64_t per = batch / threads, rem = batch % threads, b = 0;
  for (int t = 0; t < threads; ++t) {
    int64_t cnt = per + (t < rem ? 1 : 0);
    jobs[t] = (job_t){x, y, n, b, b + cnt, sign, route, scale};
    b += cnt;
  }
  if (threads == 1) {
    run_job(&jobs[0]);
    return 1;
  }
  int started = 0;
  for (int t = 0; t < threads; ++t) {
    if (pthread_create(&tid[t], NULL, run_job, &jobs[t]) != 0) {
      run_job(&jobs[t]); /* could not spawn: do it inline */
      tid[t] = 0;
    } else {
      ++started;
    }
  }
  for (int t = 0; t < threads; ++t)
    if (tid[t]) pthread_join(tid[t], NULL);
  return started > 0 ? started : 1;
}

int oracle_dft_direct(const double *x, double *y, int64_t n, int64_t batch,
                      int sign, double scale, int threads) {
  return run_batch(x, y, n, batch, sign, scale, threads, 0);
}

int oracle_fft_radix2(const double *x, double *y, int64_t n, int64_t batch,
                      int sign, double scale, int threads) {
  return run_batch(x, y, n, batch, sign, scale, threads, 1);
}

/* Per-transform relative L2 error ||a - b|| / ||b||, accumulated in fp64.
 * a: complex64 (interleaved float), b: complex128 (interleaved double). */
void oracle_rel_l2(const float *a, const double *b, int64_t n, int64_t batch,
                   double *err_out) {
  for (int64_t t = 0; t < batch; ++t) {
    double num = 0.0, den = 0.0;
    const float *at = a + 2 * t * n;
    const double *bt = b + 2 * t * n;
    for (int64_t i = 0; i < 2 * n; ++i) {
      double d = (double)at[i] - bt[i];
      num += d * d;
      den += bt[i] * bt[i];
    }
    err_out[t] = den > 0.0 ? sqrt(num / den) : sqrt(num);
  }
}
