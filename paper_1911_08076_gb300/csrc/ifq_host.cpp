// Host-only parts of the C ABI: the integrated fixed-point fold (Sec. 3.2,
// Eq. (6)-(7) + floor), packed sizes, output shapes and status strings.
// Compiled with -ffp-contract=off so the double arithmetic of the fold is
// rounded exactly in the order written.
#include <cmath>
#include <cstddef>
#include <cstdint>

#include "ifq.h"

extern "C" const char* ifq_status_str(int s) {
  switch (s) {
    case IFQ_OK: return "ok";
    case IFQ_EINVAL: return "invalid argument";
    case IFQ_ESHAPE: return "invalid or unsupported shape";
    case IFQ_EALIGN: return "misaligned pointer";
    case IFQ_ERANGE: return "size out of supported range";
    case IFQ_ECUDA: return "CUDA runtime error";
    case IFQ_ETIMEOUT: return "bounded device wait ran out";
    case IFQ_EUNSUPPORTED: return "unsupported configuration";
    case IFQ_EWORKSPACE: return "workspace missing or too small";
    default: return "unknown status";
  }
}

extern "C" int ifq_version(void) { return 301; }   // 3.1: graphs with the input and result copies

// Eq. (3)'s uniform level i (1-based) in the compact form of Sec. 3.2.
static inline double level(int i, double q_base, double q_offset) { return (double)i * q_base + q_offset; }

extern "C" int ifq_fold_layer(int cout, int K, int kbits, const float* alpha, float delta_in, const float* bias,
                              const float* gamma, const float* beta, const float* mean, const float* var, float eps,
                              float q_base, float q_offset, int32_t* thr_out, int8_t* sign_out) {
  if (cout < 1 || K < 1 || kbits < 1 || kbits > 8) return IFQ_EINVAL;
  if (!alpha || !gamma || !beta || !mean || !var || !thr_out || !sign_out) return IFQ_EINVAL;
  const double din = delta_in, qb = q_base, qo = q_offset, ep = eps;
  if (!(din > 0.0) || !std::isfinite(din) || !(qb > 0.0) || !std::isfinite(qb) || !std::isfinite(qo) ||
      !std::isfinite(ep))
    return IFQ_EINVAL;
  const int L = (1 << kbits) - 1;
  const double amax = (double)L * (double)K;
  // validate everything before writing anything
  for (int n = 0; n < cout; ++n) {
    const double a = alpha[n], g = gamma[n], be = beta[n], mu = mean[n], v = var[n];
    const double b = bias ? (double)bias[n] : 0.0;
    if (!(a > 0.0) || !std::isfinite(a) || !std::isfinite(g) || !std::isfinite(be) || !std::isfinite(mu) ||
        !std::isfinite(v) || !std::isfinite(b) || !(v + ep > 0.0))
      return IFQ_EINVAL;
  }
  for (int n = 0; n < cout; ++n) {
    const double a = alpha[n], g = gamma[n], be = beta[n], mu = mean[n], v = var[n];
    const double b = bias ? (double)bias[n] : 0.0;
    const double s_acc = a * din;          // alpha * beta of Eq. (1): scale of the integer accumulator
    const double sigma = std::sqrt(v + ep);  // BN denominator of Eq. (2)
    sign_out[n] = (int8_t)(g < 0.0 ? -1 : 1);
    for (int i = 1; i <= L; ++i) {
      const double thr = level(i, qb, qo);
      double t;
      if (g == 0.0) {
        // constant output beta: every accumulator is above (or not above) level i
        t = (be > thr) ? -amax - 1.0 : amax;
      } else {
        // Eq. (7): z > thr_i  <=>  A > tau_i (gamma > 0)  or  A < tau_i (gamma < 0)
        const double tau = ((thr - be) * sigma / g + mu - b) / s_acc;
        t = g > 0.0 ? std::floor(tau) : std::floor(-tau);
        if (!(t >= -amax - 1.0)) t = -amax - 1.0;
        if (t > amax) t = amax;
      }
      thr_out[(size_t)n * L + (i - 1)] = (int32_t)t;
    }
  }
  return IFQ_OK;
}

// Floor division of 64-bit integers (toward -infinity), d > 0.
static int64_t floor_div64(int64_t x, int64_t d) {
  int64_t q = x / d;
  if ((x % d != 0) && (x < 0)) --q;
  return q;
}

extern "C" int ifq_fold_layer_separated(int cout, int K, int kbits, int m, const float* alpha, float delta_in,
                                        const float* bias, const float* gamma, const float* beta, const float* mean,
                                        const float* var, float eps, float q_base, float q_offset, int32_t* thr_out,
                                        int8_t* sign_out) {
  if (cout < 1 || K < 1 || kbits < 1 || kbits > 8 || m < 1 || m > 20) return IFQ_EINVAL;
  if (!alpha || !gamma || !beta || !mean || !var || !thr_out || !sign_out) return IFQ_EINVAL;
  const double din = delta_in, qb = q_base, qo = q_offset, ep = eps;
  if (!(din > 0.0) || !std::isfinite(din) || !(qb > 0.0) || !std::isfinite(qb) || !std::isfinite(qo) ||
      !std::isfinite(ep))
    return IFQ_EINVAL;
  const int L = (1 << kbits) - 1;
  const int64_t amax = (int64_t)L * K;
  const double Q = std::ldexp(1.0, m);
  const int64_t Qi = (int64_t)1 << m;
  // the fixed-point constants, each floored at its own scale (Sec. 2.2)
  auto fx = [&](double x) { return (int64_t)std::floor(x * Q); };
  for (int n = 0; n < cout; ++n) {
    const double a = alpha[n], g = gamma[n], v = var[n], b = bias ? (double)bias[n] : 0.0;
    if (!(a > 0.0) || !std::isfinite(a) || !std::isfinite(g) || !std::isfinite((double)beta[n]) ||
        !std::isfinite((double)mean[n]) || !std::isfinite(v) || !std::isfinite(b) || !(v + ep > 0.0))
      return IFQ_EINVAL;
    if (g != 0.0 && fx(std::sqrt(v + ep) / g) == 0) return IFQ_EINVAL;   // no fixed-point BN divisor
  }
  const int64_t d = fx(din);
  for (int n = 0; n < cout; ++n) {
    const double g = gamma[n];
    const int64_t ad = fx(alpha[n]) * d;                                  // Y^conv = (ad*A + bq) / Q^2
    const int64_t bq = (int64_t)std::floor((bias ? (double)bias[n] : 0.0) * Q * Q);
    const int64_t th = fx(mean[n]), be = fx(beta[n]);
    const int64_t sg = g != 0.0 ? fx(std::sqrt((double)var[n] + ep) / g) : 0;   // sigma = sqrt(var+eps)/gamma
    sign_out[n] = (int8_t)(sg < 0 ? -1 : 1);
    for (int i = 1; i <= L; ++i) {
      const int64_t t = fx(level(i, qb, qo));
      int64_t T;
      if (g == 0.0) {
        T = be > t ? -amax - 1 : amax;   // Y^BN = be/Q for every A
      } else {
        // Y^BN > t/Q  <=>  (ad*A + bq - th*Q) / sg > t - be
        //   sg > 0:  ad*A > X;   sg < 0:  ad*A < X,  X = (t - be)*sg + th*Q - bq
        const int64_t X = (t - be) * sg + th * Qi - bq;
        if (ad == 0) {
          const bool above = sg > 0 ? 0 > X : 0 < X;
          T = above ? -amax - 1 : amax;
        } else {
          T = sg > 0 ? floor_div64(X, ad) : floor_div64(-X, ad);   // -A > floor(-X/ad) for sg < 0
        }
        if (T < -amax - 1) T = -amax - 1;
        if (T > amax) T = amax;
      }
      thr_out[(size_t)n * L + (i - 1)] = (int32_t)T;
    }
  }
  return IFQ_OK;
}

extern "C" int ifq_fold_output_separated(int cout, int m, const float* alpha, float delta_in, const float* bias,
                                         int64_t* mul_out, int64_t* add_out) {
  if (cout < 1 || m < 1 || m > 24 || !alpha || !mul_out || !add_out) return IFQ_EINVAL;
  const double din = delta_in;
  if (!(din > 0.0) || !std::isfinite(din)) return IFQ_EINVAL;
  for (int n = 0; n < cout; ++n) {
    const double a = alpha[n], b = bias ? (double)bias[n] : 0.0;
    if (!(a > 0.0) || !std::isfinite(a) || !std::isfinite(b)) return IFQ_EINVAL;
    if (std::fabs(a) * std::ldexp(1.0, m) > 9.0e15 || std::fabs(b) * std::ldexp(1.0, 2 * m) > 9.0e15) return IFQ_EINVAL;
  }
  const double Q = std::ldexp(1.0, m);
  const int64_t d = (int64_t)std::floor(din * Q);
  for (int n = 0; n < cout; ++n) {
    mul_out[n] = (int64_t)std::floor((double)alpha[n] * Q) * d;
    add_out[n] = (int64_t)std::floor((bias ? (double)bias[n] : 0.0) * Q * Q);
  }
  return IFQ_OK;
}

extern "C" int ifq_codes_bytes(int n, int h, int w, int c, int kbits, size_t* bytes) {
  if (!bytes || n < 0 || h < 0 || w < 0 || c < 0 || kbits < 1 || kbits > 32) return IFQ_EINVAL;
  const unsigned long long bits = (unsigned long long)n * h * w * c * (unsigned long long)kbits;
  *bytes = (size_t)((bits + 7) / 8);
  return IFQ_OK;
}

extern "C" int ifq_codes_storage_bytes(int n, int h, int w, int c, int kbits, size_t* bytes) {
  if (!bytes || n < 0 || h < 0 || w < 0 || c < 0 || kbits < 0) return IFQ_EINVAL;
  const int k = kbits == 0 ? 2 : kbits;
  if (k < 2 || k > 4) return IFQ_EUNSUPPORTED;
  if (c % 4 != 0) return IFQ_ESHAPE;
  const unsigned long long f = k == 2 ? 2 : 4;
  *bytes = (size_t)((unsigned long long)n * h * w * c * f / 8);
  return IFQ_OK;
}

extern "C" int ifq_conv_out_shape(const ifq_conv_desc* d, int* ho, int* wo) {
  if (!d || !ho || !wo) return IFQ_EINVAL;
  if (d->n < 0 || d->h < 1 || d->w < 1 || d->cin < 1 || d->cout < 1 || d->kh < 1 || d->kw < 1 || d->stride < 1 ||
      d->pad < 0)
    return IFQ_ESHAPE;
  const int a = d->h + 2 * d->pad - d->kh, b = d->w + 2 * d->pad - d->kw;
  if (a < 0 || b < 0) return IFQ_ESHAPE;
  int oh = a / d->stride + 1, ow = b / d->stride + 1;
  if (d->pool > 1) {   // fused p x p / stride p pool of the convolution output
    if (d->pool != 2 && d->pool != 4) return IFQ_EUNSUPPORTED;
    if (oh % d->pool != 0 || ow % d->pool != 0) return IFQ_ESHAPE;
    oh /= d->pool;
    ow /= d->pool;
  } else if (d->pool < 0) {
    return IFQ_EINVAL;
  }
  *ho = oh;
  *wo = ow;
  return IFQ_OK;
}

extern "C" int ifq_pool_out_shape(const ifq_pool_desc* d, int* ho, int* wo) {
  if (!d || !ho || !wo) return IFQ_EINVAL;
  if (d->n < 0 || d->h < 1 || d->w < 1 || d->c < 1 || d->k < 1 || d->stride < 1 || d->pad < 0) return IFQ_ESHAPE;
  const int a = d->h + d->pad - d->k, b = d->w + d->pad - d->k;
  if (a < 0 || b < 0) return IFQ_ESHAPE;
  *ho = a / d->stride + 1;
  *wo = b / d->stride + 1;
  return IFQ_OK;
}
