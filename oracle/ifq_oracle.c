/*
 * ifq_oracle.c -- plain, slow CPU oracle for the IFQ-Net quantized substructure
 * (Gao et al., "IFQ-Net: Integrated Fixed-point Quantization Networks for
 * Embedded Vision", arXiv:1911.08076).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the reference that the CUDA path is
 * checked against.  Only the test suite, the package smoke test and the
 * CPU-baseline leg of the benchmark may load it.  It shares no code, header,
 * table or constant with the GPU library, and the GPU library never calls it.
 *
 * Everything here follows the paper's equations in their own order, in double
 * precision, with no blocking, fusion or reordering:
 *   ifqo_float_chain  Eq. (1) conv scale + bias, Eq. (2) batch norm, Eq. (3)
 *                     k-bit uniform quantizer (thresholds of the compact form
 *                     thr_i = i*base + offset, Sec. 3.2 / Eq. (8)).
 *   ifqo_fold         Eq. (6)-(7) composition of alpha, BN and the quantizer
 *                     into accumulator-domain thresholds, then the floor of
 *                     Sec. 3.2 ("integrated fixed-point conversion").
 *   ifqo_int_chain    Eq. (7)/(8) applied to the integer accumulator.
 *   ifqo_conv_acc     the integer core W_b (x) X_q of Eq. (1) (cross-correlation,
 *                     zero padding = code 0).
 *   ifqo_maxpool_acc  Sec. 2.1: max pooling on Y^conv, before BN / quantizer.
 *   ifqo_maxpool_codes  pooling on codes: plain max, or with a per-channel sign
 *                     the max/min that equals quantize(max over Y^conv).
 *   ifqo_separated_chain  the separated fixed-point conversion of Sec. 2.2 (each
 *                     float floored at scale Q_m = 2^m on its own), for comparison.
 *
 * Readings of the paper used here (where it is silent or assumes more):
 *   - BN is the general affine form z = gamma*(y - mean)/sqrt(var + eps) + beta;
 *     the paper's sigma is sqrt(var + eps) and its BN has gamma = 1, beta = 0.
 *   - A negative BN scale (gamma < 0) reverses the inequality of Eq. (7); the
 *     fold then thresholds -A against floor(-tau) and reports sign = -1.
 *   - gamma == 0 makes the code constant; thresholds are set to the ends of the
 *     achievable accumulator range [-3K, 3K] (2^k - 1 in place of 3 for k bits).
 *   - Thresholds are clamped to [-Amax-1, Amax] with Amax = (2^k - 1)*K, which
 *     leaves every code of an achievable accumulator unchanged.
 */
#include <math.h>
#include <stdint.h>
#include <stddef.h>

#define ORC_OK 0
#define ORC_EINVAL 1

static int64_t floor_scaled(double x, double q) { return (int64_t)floor(x * q); }

/* Uniform quantizer level i (1-based), Sec. 3.2: thr_i = i*base + offset. */
static double level(int i, double q_base, double q_offset) { return (double)i * q_base + q_offset; }

/*
 * Float chain, Eq. (1)-(3), for an M x cout matrix of accumulators A = W_b (x) X_q
 * (row-major, channel fastest).  For channel n:
 *   y = alpha[n] * delta_in * A + bias[n]                   Eq. (1)
 *   z = gamma[n] * (y - mean[n]) / sqrt(var[n] + eps) + beta[n]   Eq. (2)
 *   code = number of levels i in 1..L with z > thr_i         Eq. (3)
 * Eq. (3) gives code 0 for z <= thr_1, i for thr_i < z <= thr_{i+1} and L for
 * z > thr_L, which is that count for ascending thresholds.
 * If gap is not NULL, gap[m*cout+n] receives min_i |z - thr_i| (tie detector).
 */
int ifqo_float_chain(long M, int cout, const int32_t* A, int L, const double* alpha, double delta_in,
                     const double* bias, const double* gamma, const double* beta, const double* mean,
                     const double* var, double eps, double q_base, double q_offset, uint8_t* codes, double* gap) {
  if (M < 0 || cout <= 0 || L <= 0 || L > 255) return ORC_EINVAL;
  for (long m = 0; m < M; ++m) {
    for (int n = 0; n < cout; ++n) {
      double a = (double)A[m * cout + n];
      double b = bias ? bias[n] : 0.0;
      double y = alpha[n] * delta_in * a + b;
      double z = gamma[n] * (y - mean[n]) / sqrt(var[n] + eps) + beta[n];
      int code = 0;
      double g = INFINITY;
      for (int i = 1; i <= L; ++i) {
        double t = level(i, q_base, q_offset);
        if (z > t) code += 1;
        if (fabs(z - t) < g) g = fabs(z - t);
      }
      codes[m * cout + n] = (uint8_t)code;
      if (gap) gap[m * cout + n] = g;
    }
  }
  return ORC_OK;
}

/*
 * Integrated fixed-point conversion, Eq. (6)-(7) and the floor of Sec. 3.2.
 * K is the reduction length of the layer (kh*kw*cin), so |A| <= Amax = (2^k-1)*K.
 * For channel n and level i the accumulator-domain threshold of Eq. (7) is
 *   tau_i = ((thr_i - beta) * sqrt(var + eps) / gamma + mean - bias) / (alpha * delta_in)
 * (the paper's (thr_i*sigma + theta - b)/(alpha*beta) with the affine BN).
 *   gamma > 0: z > thr_i  <=>  A > tau_i   <=>  A > floor(tau_i);   sign = +1
 *   gamma < 0: z > thr_i  <=>  A < tau_i   <=> -A > floor(-tau_i);  sign = -1
 *   gamma = 0: z = beta for every A; T_i = -Amax-1 if beta > thr_i else Amax.
 * T is [cout][L] int32; sign is [cout].
 */
int ifqo_fold(int cout, long K, int L, const double* alpha, double delta_in, const double* bias,
              const double* gamma, const double* beta, const double* mean, const double* var, double eps,
              double q_base, double q_offset, int32_t* T, int8_t* sign) {
  if (cout <= 0 || K <= 0 || L <= 0 || L > 255) return ORC_EINVAL;
  if (!(delta_in > 0.0) || !(q_base > 0.0)) return ORC_EINVAL;
  double amax = (double)L * (double)K;
  for (int n = 0; n < cout; ++n) {
    if (!(alpha[n] > 0.0) || !(var[n] + eps > 0.0)) return ORC_EINVAL;
    double b = bias ? bias[n] : 0.0;
    double sA = alpha[n] * delta_in;
    double sd = sqrt(var[n] + eps);
    sign[n] = (int8_t)(gamma[n] < 0.0 ? -1 : 1);
    for (int i = 1; i <= L; ++i) {
      double thr = level(i, q_base, q_offset);
      double t;
      if (gamma[n] == 0.0) {
        t = (beta[n] > thr) ? -amax - 1.0 : amax;
      } else {
        double tau = ((thr - beta[n]) * sd / gamma[n] + mean[n] - b) / sA;
        t = gamma[n] > 0.0 ? floor(tau) : floor(-tau);
        if (!(t >= -amax - 1.0)) t = -amax - 1.0;  /* also catches NaN */
        if (t > amax) t = amax;
      }
      T[n * L + (i - 1)] = (int32_t)t;
    }
  }
  return ORC_OK;
}

/* Eq. (7)/(8) on the integer accumulator: code = #{ i : sign*A > T_i }. */
int ifqo_int_chain(long M, int cout, const int32_t* A, int L, const int32_t* T, const int8_t* sign, uint8_t* codes) {
  if (M < 0 || cout <= 0 || L <= 0) return ORC_EINVAL;
  for (long m = 0; m < M; ++m) {
    for (int n = 0; n < cout; ++n) {
      long v = (long)sign[n] * (long)A[m * cout + n];
      int code = 0;
      for (int i = 0; i < L; ++i)
        if (v > (long)T[n * L + i]) code += 1;
      codes[m * cout + n] = (uint8_t)code;
    }
  }
  return ORC_OK;
}

/*
 * Integer core of Eq. (1): A[b][oy][ox][n] = sum_{dy,dx,c} w[n][dy][dx][c] * x[b][oy*s+dy-p][ox*s+dx-p][c],
 * with x outside the image read as code 0.  x is NHWC uint8 codes, w is int8
 * (+1/-1) [cout][kh][kw][cin], A is int32 NHWC [nb][ho][wo][cout].
 * Output size ho = (h + 2p - kh)/s + 1 (floor), likewise wo.
 */
int ifqo_conv_acc(int nb, int h, int w, int cin, int cout, int kh, int kw, int stride, int pad,
                  const uint8_t* x, const int8_t* wt, int32_t* A) {
  if (nb < 0 || h <= 0 || w <= 0 || cin <= 0 || cout <= 0 || kh <= 0 || kw <= 0 || stride <= 0 || pad < 0)
    return ORC_EINVAL;
  int ho = (h + 2 * pad - kh) / stride + 1;
  int wo = (w + 2 * pad - kw) / stride + 1;
  if (ho <= 0 || wo <= 0) return ORC_EINVAL;
  for (int b = 0; b < nb; ++b)
    for (int oy = 0; oy < ho; ++oy)
      for (int ox = 0; ox < wo; ++ox)
        for (int n = 0; n < cout; ++n) {
          long acc = 0;
          for (int dy = 0; dy < kh; ++dy)
            for (int dx = 0; dx < kw; ++dx) {
              int iy = oy * stride + dy - pad;
              int ix = ox * stride + dx - pad;
              if (iy < 0 || iy >= h || ix < 0 || ix >= w) continue; /* code 0 */
              for (int c = 0; c < cin; ++c) {
                long xv = x[(((long)b * h + iy) * w + ix) * cin + c];
                long wv = wt[(((long)n * kh + dy) * kw + dx) * cin + c];
                acc += wv * xv;
              }
            }
          A[(((long)b * ho + oy) * wo + ox) * cout + n] = (int32_t)acc;
        }
  return ORC_OK;
}

/*
 * Pooling geometry (both pools): windows of k x k starting at (oy*s, ox*s);
 * `pad` extra cells at the bottom and right, which hold no value and are
 * skipped.  ho = (h + pad - k)/s + 1.
 */

/* Sec. 2.1: max pooling of Y^conv, placed before BN and the quantizer.  A is int32 NHWC. */
int ifqo_maxpool_acc(int nb, int h, int w, int c, int k, int stride, int pad, const int32_t* A, int32_t* out) {
  if (nb < 0 || h <= 0 || w <= 0 || c <= 0 || k <= 0 || stride <= 0 || pad < 0) return ORC_EINVAL;
  int ho = (h + pad - k) / stride + 1;
  int wo = (w + pad - k) / stride + 1;
  if (ho <= 0 || wo <= 0) return ORC_EINVAL;
  for (int b = 0; b < nb; ++b)
    for (int oy = 0; oy < ho; ++oy)
      for (int ox = 0; ox < wo; ++ox)
        for (int ch = 0; ch < c; ++ch) {
          long best = 0;
          int any = 0;
          for (int dy = 0; dy < k; ++dy)
            for (int dx = 0; dx < k; ++dx) {
              int iy = oy * stride + dy, ix = ox * stride + dx;
              if (iy >= h || ix >= w) continue;
              long v = A[(((long)b * h + iy) * w + ix) * c + ch];
              if (!any || v > best) best = v;
              any = 1;
            }
          out[(((long)b * ho + oy) * wo + ox) * c + ch] = (int32_t)best;
        }
  return ORC_OK;
}

/*
 * Pooling on codes.  With sign == NULL: plain max of the codes (pooling after
 * the quantizer).  With a sign per channel: max of the codes where sign = +1
 * and min where sign = -1.  Because the quantizer composed with the affine
 * conv/BN map is non-decreasing in A for sign +1 and non-increasing for sign -1,
 * this equals quantize(max of A over the window), the order of Sec. 2.1.
 */
int ifqo_maxpool_codes(int nb, int h, int w, int c, int k, int stride, int pad, const uint8_t* x,
                       const int8_t* sign, uint8_t* out) {
  if (nb < 0 || h <= 0 || w <= 0 || c <= 0 || k <= 0 || stride <= 0 || pad < 0) return ORC_EINVAL;
  int ho = (h + pad - k) / stride + 1;
  int wo = (w + pad - k) / stride + 1;
  if (ho <= 0 || wo <= 0) return ORC_EINVAL;
  for (int b = 0; b < nb; ++b)
    for (int oy = 0; oy < ho; ++oy)
      for (int ox = 0; ox < wo; ++ox)
        for (int ch = 0; ch < c; ++ch) {
          int use_min = sign && sign[ch] < 0;
          int best = 0, any = 0;
          for (int dy = 0; dy < k; ++dy)
            for (int dx = 0; dx < k; ++dx) {
              int iy = oy * stride + dy, ix = ox * stride + dx;
              if (iy >= h || ix >= w) continue;
              int v = x[(((long)b * h + iy) * w + ix) * c + ch];
              if (!any || (use_min ? v < best : v > best)) best = v;
              any = 1;
            }
          out[(((long)b * ho + oy) * wo + ox) * c + ch] = (uint8_t)best;
        }
  return ORC_OK;
}

/*
 * Separated fixed-point conversion, Sec. 2.2 (Fig. 3a), for comparison with the
 * integrated conversion.  With Q = 2^m, every float is floored at its own scale:
 *   a = floor(alpha*Q), d = floor(delta_in*Q), bq = floor(bias*Q^2)
 *   Y^conv = (a*d*A + bq) / Q^2                         (the paper's separated conv)
 *   BN, Eq. (2) with the paper's theta = mean and sigma = sqrt(var + eps)/gamma (the
 *   divisor of the affine BN), plus the shift beta: th = floor(mean*Q),
 *   sg = floor(sigma*Q), be = floor(beta*Q):
 *   Y^BN = (Y^conv - th/Q) / (sg/Q) + be/Q
 *   code = #{ i : Y^BN > floor(thr_i*Q)/Q }             Eq. (3)
 * evaluated exactly in 64-bit integers: with N = a*d*A + bq (= Y^conv * Q^2) and
 * t_i = floor(thr_i*Q),  Y^BN > t_i/Q  <=>  (N - th*Q) / sg > t_i - be, i.e.
 * N - th*Q > (t_i - be)*sg for sg > 0 and N - th*Q < (t_i - be)*sg for sg < 0.
 * gamma = 0 (sigma infinite) gives Y^BN = be/Q for every A.  sg = 0 (|sigma| < 1/Q)
 * has no fixed-point divisor and is rejected, as is m outside 1..20 (int64 range).
 */
int ifqo_separated_chain(long M, int cout, const int32_t* A, int L, int m, const double* alpha, double delta_in,
                         const double* bias, const double* gamma, const double* beta, const double* mean,
                         const double* var, double eps, double q_base, double q_offset, uint8_t* codes) {
  if (M < 0 || cout <= 0 || L <= 0 || L > 255 || m < 1 || m > 20) return ORC_EINVAL;
  const double Q = ldexp(1.0, m);
  const int64_t Qi = (int64_t)1 << m;
  const int64_t d = floor_scaled(delta_in, Q);
  for (int n = 0; n < cout; ++n) {
    const int64_t a = floor_scaled(alpha[n], Q);
    const int64_t bq = (int64_t)floor((bias ? bias[n] : 0.0) * Q * Q);
    const int64_t th = floor_scaled(mean[n], Q), be = floor_scaled(beta[n], Q);
    int64_t sg = 0;
    if (gamma[n] != 0.0) {
      sg = floor_scaled(sqrt(var[n] + eps) / gamma[n], Q);
      if (sg == 0) return ORC_EINVAL;
    }
    for (long r = 0; r < M; ++r) {
      const int64_t N = a * d * (int64_t)A[r * cout + n] + bq;
      int code = 0;
      for (int i = 1; i <= L; ++i) {
        const int64_t t = floor_scaled(level(i, q_base, q_offset), Q);
        int above;
        if (gamma[n] == 0.0) above = be > t;                          /* Y^BN = be/Q */
        else if (sg > 0) above = N - th * Qi > (t - be) * sg;
        else above = N - th * Qi < (t - be) * sg;
        code += above;
      }
      codes[r * cout + n] = (uint8_t)code;
    }
  }
  return ORC_OK;
}

/*
 * Separated fixed-point conversion of a NON-quantized substructure's output, Sec. 2.2
 * (the linear detection conv of a YOLO head, AlexNet's substructure 7): with Q = 2^m,
 *   a = floor(alpha*Q), d = floor(delta_in*Q), bq = floor(bias*Q^2)
 *   Y^conv = (a*d*A + bq) / Q^2                                  (Eq. (1), each float floored)
 * and the output kept at Q's scale, m fractional bits:
 *   y = floor(Y^conv * Q) = floor((a*d*A + bq) / Q)
 * evaluated exactly in 128-bit integers, then saturated to the int32 range.  m in 1..24.
 */
static int32_t sat32(__int128 v) {
  if (v > (__int128)INT32_MAX) return INT32_MAX;
  if (v < (__int128)INT32_MIN) return INT32_MIN;
  return (int32_t)v;
}

int ifqo_fixed_output(long M, int cout, const int32_t* A, int m, const double* alpha, double delta_in,
                      const double* bias, int32_t* out) {
  if (M < 0 || cout <= 0 || m < 1 || m > 24) return ORC_EINVAL;
  const double Q = ldexp(1.0, m);
  const int64_t Qi = (int64_t)1 << m;
  const int64_t d = floor_scaled(delta_in, Q);
  for (int n = 0; n < cout; ++n) {
    const int64_t a = floor_scaled(alpha[n], Q);
    const int64_t bq = (int64_t)floor((bias ? bias[n] : 0.0) * Q * Q);
    for (long r = 0; r < M; ++r) {
      const __int128 N = (__int128)a * d * A[r * cout + n] + bq;
      __int128 y = N / Qi;                              /* C division truncates toward zero */
      if (N % Qi != 0 && N < 0) y -= 1;                 /* floor */
      out[r * cout + n] = sat32(y);
    }
  }
  return ORC_OK;
}
