// gaus_device.cuh -- small device helpers shared by the kernels of the library:
// the window of a (node, restart), the standard normal CDF, bin masses and the
// exact fixed-point histogram update.
#pragma once

#include <cuda_runtime.h>

#include "gaus_internal.h"
#include "mills_ratio.h"

namespace gaus {

// Points t with |t + 1/2 - mu| <= k sigma, clipped to [0, D-2]; a = b + 1 when empty.
__device__ __forceinline__ void window(float mu, float sg, float k, int D, int &a, int &b) {
  float lo = ceilf(mu - k * sg - 0.5f), hi = floorf(mu + k * sg - 0.5f);
  lo = fminf(fmaxf(lo, 0.0f), (float)(D - 1));
  hi = fminf(fmaxf(hi, -1.0f), (float)(D - 2));
  a = (int)lo;
  b = (int)hi;
}

// Phi(z) from the Mills ratio: the upper tail Q(|z|) = exp(-z^2/2) P(|z|)/Q(|z|)
// (rational fit of mills_ratio.h, |z| <= 12), absolute error ~1e-6.  Used for
// the neighbour values of the edge terms, which only need absolute accuracy.
__device__ __forceinline__ float cdf_fast(float z) {
  const float x = fabsf(z);
  const float e = __expf(-0.5f * z * z);
  const float num = (((kMillsP[4] * x + kMillsP[3]) * x + kMillsP[2]) * x + kMillsP[1]) * x + kMillsP[0];
  const float den = ((((kMillsQ[5] * x + kMillsQ[4]) * x + kMillsQ[3]) * x + kMillsQ[2]) * x + kMillsQ[1]) * x + 1.0f;
  const float q = e * __fdividef(num, den);
  return z <= 0.f ? q : 1.0f - q;
}

// Upper tail Q(|z|) = Phi(-|z|) from the same Mills-ratio fit: relative error
// ~1e-6 on |z| <= 12 (the fit) plus the fast exponential's, so both tails of the
// bin masses keep their relative accuracy.
__device__ __forceinline__ float tail_fast(float z) {
  const float x = fabsf(z);
  const float e = __expf(-0.5f * z * z);
  const float num = (((kMillsP[4] * x + kMillsP[3]) * x + kMillsP[2]) * x + kMillsP[1]) * x + kMillsP[0];
  const float den = ((((kMillsQ[5] * x + kMillsQ[4]) * x + kMillsQ[3]) * x + kMillsQ[2]) * x + kMillsQ[1]) * x + 1.0f;
  return e * __fdividef(num, den);
}

// CDF families of the relaxation: the standard normal (Sec. 3.2) and, in its
// place (App. D), the logistic, Laplace and Cauchy CDFs with the scale matched to
// sigma -- logistic s = sigma sqrt(3)/pi and Laplace b = sigma/sqrt(2) (equal
// variance), Cauchy gamma = sigma sqrt(2 ln 2) (equal full width at half
// maximum).  In z = (x - mu)/sigma each is G(c z) for its standard CDF G, with
// c = sigma/s, sigma/b or sigma/gamma; every family is symmetric, so one upper
// tail Q(|z|) = 1 - F(|z|) gives F on both sides.  Fam<k>::tail(z) = Q(|z|),
// Fam<k>::pdf(z) = F'(z), Fam<k>::cdf(z) = F(z).
template <int kFam>
struct Fam;

template <>
struct Fam<GAUS_GAUSSIAN> {
  static __device__ __forceinline__ float tail(float z) { return tail_fast(z); }
  static __device__ __forceinline__ float pdf(float z) { return 0.3989422804014327f * __expf(-0.5f * z * z); }
  static __device__ __forceinline__ float cdf(float z) { return cdf_fast(z); }
};

template <>
struct Fam<GAUS_LOGISTIC> {
  static constexpr float kC = 1.8137993642342178f;  // pi / sqrt(3)
  // Q = e / (1 + e) with e = exp(-c |z|): relative accuracy in both tails
  static __device__ __forceinline__ float tail(float z) {
    const float e = __expf(-kC * fabsf(z));
    return __fdividef(e, 1.0f + e);
  }
  static __device__ __forceinline__ float pdf(float z) {
    const float e = __expf(-kC * fabsf(z));
    const float r = __fdividef(1.0f, 1.0f + e);
    return kC * e * r * r;
  }
  static __device__ __forceinline__ float cdf(float z) {
    const float q = tail(z);
    return z <= 0.f ? q : 1.0f - q;
  }
};

template <>
struct Fam<GAUS_LAPLACE> {
  static constexpr float kC = 1.4142135623730951f;  // sqrt(2)
  static __device__ __forceinline__ float tail(float z) { return 0.5f * __expf(-kC * fabsf(z)); }
  static __device__ __forceinline__ float pdf(float z) { return 0.5f * kC * __expf(-kC * fabsf(z)); }
  static __device__ __forceinline__ float cdf(float z) {
    const float q = tail(z);
    return z <= 0.f ? q : 1.0f - q;
  }
};

template <>
struct Fam<GAUS_CAUCHY> {
  static constexpr float kC = 0.8493218002880191f;   // 1 / sqrt(2 ln 2)
  static constexpr float kInvPi = 0.3183098861837907f;
  // Q = atan(1 / (c |z|)) / pi: the complement of 1/2 + atan(y)/pi without the
  // cancellation in the far tail; 1 / 0 = inf gives Q(0) = 1/2
  static __device__ __forceinline__ float tail(float z) { return kInvPi * atanf(1.0f / (kC * fabsf(z))); }
  static __device__ __forceinline__ float pdf(float z) {
    const float y = kC * z;
    return __fdividef(kC * kInvPi, 1.0f + y * y);
  }
  static __device__ __forceinline__ float cdf(float z) {
    const float q = tail(z);
    return z <= 0.f ? q : 1.0f - q;
  }
};

// One Adam step of a parameter (torch.optim.Adam semantics): m, v updated in
// place; inv_bc1 = 1 / (1 - beta1^t), rs_bc2 = 1 / sqrt(1 - beta2^t).
__device__ __forceinline__ float adam_update(float th, float g, float &m, float &v, float lr, float beta1,
                                             float beta2, float eps, float inv_bc1, float rs_bc2) {
  m = beta1 * m + (1.0f - beta1) * g;
  v = beta2 * v + (1.0f - beta2) * g * g;
  return th - __fdividef(lr * m * inv_bc1, sqrtf(v) * rs_bc2 + eps);
}

// Windowed CDF of a neighbour at integer point x.
__device__ __forceinline__ float cdf_at(int x, float mu, float inv_s, int a, int b) {
  if (x < a) return 0.0f;
  if (x > b) return 1.0f;
  return cdf_fast(((float)x + 0.5f - mu) * inv_s);
}

__device__ __forceinline__ int fold_bin(int d, int II) { return II > 0 ? d % II : d; }

// A restart's (mu, sigma) is usable when both are finite and sigma >= 1e-30, so
// that 1/sigma is finite.
__device__ __forceinline__ bool usable(float mu, float sg) {
  return isfinite(mu) && isfinite(sg) && sg >= 1e-30f;
}

constexpr float kInvSqrt2Pi = 0.3989422804014327f;
constexpr float kInvSqrt2 = 0.7071067811865476f;

// Bin mass of bin p of a window from the tail values (z, q = Q(|z|)) of points p
// and p - 1: P = C(a+p) - C(a+p-1), with C = 0 below the window and 1 above it,
// choosing the subtraction that keeps both tails relatively accurate.
__device__ __forceinline__ float bin_mass(bool pt, bool first, float zc, float qc, float zp, float qp) {
  const float c_cur = pt ? (zc <= 0.f ? qc : 1.0f - qc) : 1.0f;
  const float c_prev = first ? 0.0f : (zp <= 0.f ? qp : 1.0f - qp);
  float P = c_cur - c_prev;
  P = (pt && !first && zc <= 0.f) ? qc - qp : P;
  P = (pt && !first && zp > 0.f) ? qp - qc : P;
  P = (pt && !first && zp <= 0.f && zc > 0.f) ? (0.5f - qc) + (0.5f - qp) : P;
  P = (!pt && !first && zp > 0.f) ? qp : P;  // top bin: upper tail Q directly
  return P;
}

// Adds round(w P 2^32) to a histogram cell as two exact 16-bit halves, using
// 32-bit conversions only (float -> 64-bit integer conversion runs at the FP64 rate).
__device__ __forceinline__ void hist_add(unsigned *hlo, unsigned *hhi, int cell, float wP) {
  const float xs = fmaxf(wP, 0.0f) * 65536.0f;
  const float fh = floorf(xs);
  atomicAdd(&hlo[cell], __float2uint_rn((xs - fh) * 65536.0f));
  atomicAdd(&hhi[cell], (unsigned)fh);
}

}  // namespace gaus
