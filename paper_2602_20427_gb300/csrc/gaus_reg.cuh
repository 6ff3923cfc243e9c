// gaus_reg.cuh -- expected live storage (Eq. active, Sec. 3.2), folded modulo II
// for pipelined scheduling (MReg, App. B.3), and its gradient.
//
//   Reg(d) = sum_i b_i C_i(d) (1 - M_i(d)),   M_i(d) = prod_{j in succ(i)} C_j(d),
//
// with a leaf's successor a sink at step D (M_i = 0).  For a producer i and restart
// b the term is
//   * 0 below its window,
//   * b_i C_i(d) (1 - M_i(d)) on its own window,
//   * b_i (an integer) from its window's end until its last successor's window
//     starts (some successor certainly has not started) -- a range add,
//   * b_i (1 - M_i(d)) while the successors' CDFs vary, 0 after.
// 1 - M is accumulated as t <- t + (1 - t) Q_j with Q_j = 1 - C_j the accurate
// upper tail, so it keeps relative accuracy when every successor has almost
// surely started.  Histograms are exact fixed point (as for the usage).
//
// Backward, per producer: its own adjoint G(d) b_i (1 - M_i(d)) on its window,
// and for each out-edge i -> j the share of the successor, -G(d) b_i C_i(d)
// prod_{j' != j} C_j'(d), dotted with phi_j on j's window into one (dmu, dsigma)
// slot per (edge, restart) that the successor gathers through its in-edges.
#pragma once

#include <climits>
#include <cuda_runtime.h>
#include <stdint.h>

#include "gaus_device.cuh"
#include "gaus_internal.h"

namespace gaus {

struct RegArgs {
  const float *mu, *sg;  // (V, B) caller order
  int V, B, D, II, Dh, RB, G;
  float k_win;
  const int32_t *perm;
  const float *bits;
  const int32_t *out_ptr, *out_dst;  // internal CSR, successors by caller id
  const int32_t *seg;
  const unsigned *win;               // packed windows
  const float *tab;                  // the node pass's CDF table rows (V, B, W) by caller id
  int W;
  float *ptab;                       // (V, B, WP) by caller id: the successors' product P(d) for
  int WP;                            // d = max(a, Amax) .. Bm, written by the forward
  const float4 *qtab;                // the family's tail table (kTailRows x 2, k_tail_tables)
  long long *rpart;                  // blocks * Dh * RB
  // backward
  const float *Hreg;                 // (B, Dh): w_mem * softmax of (M)Reg
  float2 *gown;                      // (V, B) internal order: the own-window adjoint
  float2 *eslot;                     // (E, B) per out-edge slot (CSR position)
};

// Upper tail Q(|z|) and density of the storage terms: the normal through erfcf
// and expf, the other families through Fam<kFam>.
template <int kFam>
__device__ __forceinline__ float reg_tail(float z) {
  if constexpr (kFam == GAUS_GAUSSIAN) return 0.5f * erfcf(fabsf(z) * kInvSqrt2);
  else return Fam<kFam>::tail(z);
}
template <int kFam>
__device__ __forceinline__ float reg_pdf(float z) {
  if constexpr (kFam == GAUS_GAUSSIAN) return kInvSqrt2Pi * expf(-0.5f * z * z);
  else return Fam<kFam>::pdf(z);
}

// C and Q = 1 - C of a windowed CDF at integer point d, both tails accurate.
template <int kFam>
__device__ __forceinline__ void cdf_pair(int d, float mu, float inv_s, int a, int b, float &C, float &Q) {
  if (d < a) { C = 0.f; Q = 1.f; return; }
  if (d > b) { C = 1.f; Q = 0.f; return; }
  const float z = ((float)d + 0.5f - mu) * inv_s;
  const float q = reg_tail<kFam>(z);
  C = z <= 0.f ? q : 1.0f - q;
  Q = z <= 0.f ? 1.0f - q : q;
}

// ---------------------------------------------------------------- storage forward in float pairs
// The storage LSE's softmax at a small tau turns absolute errors of the expected
// storage into relative errors of its weights divided by tau, and a bin sums
// hundreds of contributions b_i C_i (1 - M_i) of up to 64 bits each: with fp32
// contributions (~1e-7 relative each) the gradient would carry ~1e-4 relative
// error.  The forward therefore carries the tails, the successors' product and
// each contribution as unevaluated pairs hi + lo of floats (~1e-12 absolute, FP32
// arithmetic throughout: GB300's FP64 rate is a small fraction of its FP32 rate)
// and rounds each contribution once, into the fixed-point histogram.
//
// The upper tail Q(z) = 1 - F(z), z >= 0, comes from a table of Q and of the
// density f and its first three derivatives at z0 = i / 64, 0 <= z0 <= 16, filled
// once in double (k_tail_tables), and a Taylor step of four terms to z
// (|z - z0| <= 1/128: truncation below 1e-12).  Beyond z = 16 the normal, logistic
// and Laplace tails are below 1e-10 and are taken in fp32; the Cauchy tail
// atan(1 / (c z)) / pi comes from the arctangent series in y = 1 / (c z) <= 0.074.
constexpr int kTailPerUnit = 64, kTailZmax = 16, kTailRows = kTailZmax * kTailPerUnit + 1;

struct FF {
  float h, l;
};
// h + l = a + b exactly (two-sum)
__device__ __forceinline__ FF ff_two_sum(float a, float b) {
  const float s = __fadd_rn(a, b), bb = __fsub_rn(s, a);
  return {s, __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb))};
}
// h + l = a + b exactly when |a| >= |b| or a = 0 (fast two-sum)
__device__ __forceinline__ FF ff_fast_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  return {s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ FF ff_add(FF a, FF b) {
  const FF s = ff_two_sum(a.h, b.h);
  return ff_fast_sum(s.h, s.l + (a.l + b.l));
}
__device__ __forceinline__ FF ff_mul(FF a, FF b) {
  const float p = __fmul_rn(a.h, b.h);
  return ff_fast_sum(p, fmaf(a.h, b.h, -p) + (a.h * b.l + a.l * b.h));
}
__device__ __forceinline__ FF ff_mulf(FF a, float b) {
  const float p = __fmul_rn(a.h, b);
  return ff_fast_sum(p, fmaf(a.h, b, -p) + a.l * b);
}
// 1 - a for 0 <= a <= 1
__device__ __forceinline__ FF ff_one_minus(FF a) {
  const FF s = ff_fast_sum(1.0f, -a.h);
  return ff_fast_sum(s.h, s.l - a.l);
}

// z = (d + 1/2 - mu) / sigma as a pair: the division's residual from an fma
__device__ __forceinline__ FF z_pair(int d, float mu, float sg, float inv_s) {
  const FF x = ff_two_sum((float)d + 0.5f, -mu);
  const float zh = x.h * inv_s;
  return {zh, (fmaf(-zh, sg, x.h) + x.l) * inv_s};
}

template <int kFam>
__device__ __forceinline__ FF reg_tail_pair(const float4 *__restrict__ tab, float zh, float zl) {
  if (zh >= (float)kTailZmax) {
    if constexpr (kFam == GAUS_CAUCHY) {
      constexpr double kC = 0.84932180028801904272, kInvPi = 0.31830988618379067154;
      constexpr float kCh = (float)kC, kCl = (float)(kC - (double)kCh);
      constexpr float kPh = (float)kInvPi, kPl = (float)(kInvPi - (double)kPh);
      const FF cz = ff_mul({kCh, kCl}, {zh, zl});
      const float yh = 1.0f / cz.h;
      const FF y = ff_fast_sum(yh, yh * (fmaf(-yh, cz.h, 1.0f) - yh * cz.l));
      const float y2 = yh * yh;
      const float del = y2 * (-1.0f / 3.0f + y2 * (0.2f + y2 * (-1.0f / 7.0f + y2 * (1.0f / 9.0f))));
      return ff_mul(ff_add(y, {yh * del, 0.0f}), {kPh, kPl});
    } else {
      return {Fam<kFam>::tail(zh), 0.0f};
    }
  }
  const int i = __float2int_rn(zh * (float)kTailPerUnit);
  const float hh = zh - (float)i * (1.0f / (float)kTailPerUnit);  // exact
  const float4 q = __ldg(&tab[2 * i]), t = __ldg(&tab[2 * i + 1]);
  // Q(z0 + h) = Q0 - f h - f' h^2 / 2 - f'' h^3 / 6 - f''' h^4 / 24, h = hh + zl
  const float rest = hh * hh * (t.x + hh * (t.y + hh * t.z));
  const float p = __fmul_rn(q.z, hh);
  const float pe = fmaf(q.z, hh, -p) + (q.z * zl + q.w * hh);
  const FF s = ff_two_sum(q.x, -p);
  return ff_fast_sum(s.h, s.l + (q.y - (pe + rest)));
}

// C of a windowed CDF at integer point d as a pair (0 and 1 outside [a, b])
template <int kFam>
__device__ __forceinline__ FF cdf_pair_ff(const float4 *__restrict__ tab, int d, float mu, float sg, float inv_s,
                                          int a, int b) {
  if (d < a) return {0.0f, 0.0f};
  if (d > b) return {1.0f, 0.0f};
  const FF z = z_pair(d, mu, sg, inv_s);
  const bool neg = z.h <= 0.0f;
  const FF q = reg_tail_pair<kFam>(tab, neg ? -z.h : z.h, neg ? -z.l : z.l);
  return neg ? q : ff_one_minus(q);
}

// hist_add of a pair in [0, 64]: rounded once to 2^-32
__device__ __forceinline__ void hist_add_pair(unsigned *hlo, unsigned *hhi, int cell, FF v) {
  long long F = __float2ll_rn(v.h * 4294967296.0f) + __float2ll_rn(v.l * 4294967296.0f);
  F = F < 0 ? 0 : F;
  atomicAdd(&hlo[cell], (unsigned)(F & 0xFFFF));
  atomicAdd(&hhi[cell], (unsigned)(F >> 16));
}

// Adds the integer v to the (folded) bins d in [s, e] through a difference
// array (Dh + 1 rows) and a per-restart constant for whole cycles of II.
__device__ __forceinline__ void range_add(int *rdiff, int *rconst, int RB, int r, int s, int e, int v, int II) {
  if (II <= 0) {
    atomicAdd(&rdiff[s * RB + r], v);
    atomicAdd(&rdiff[(e + 1) * RB + r], -v);
    return;
  }
  const int len = e - s + 1, full = len / II, rem = len % II;
  if (full) atomicAdd(&rconst[r], full * v);
  if (!rem) return;
  const int st = s % II;
  if (st + rem <= II) {
    atomicAdd(&rdiff[st * RB + r], v);
    atomicAdd(&rdiff[(st + rem) * RB + r], -v);
  } else {
    atomicAdd(&rdiff[st * RB + r], v);
    atomicAdd(&rdiff[II * RB + r], -v);
    atomicAdd(&rdiff[0 * RB + r], v);
    atomicAdd(&rdiff[(st + rem - II) * RB + r], -v);
  }
}

// Successor bounds of a producer: A = max a_j (D for a leaf), Bm = max b_j (-1 for a leaf).
__device__ __forceinline__ void succ_bounds(const RegArgs &A, int e0, int deg, int dmax, int b, int &Amax, int &Bm) {
  Amax = deg == 0 ? A.D : INT_MIN;
  Bm = -1;
  for (int q = 0; q < dmax; ++q) {
    if (q < deg) {
      const unsigned wm = A.win[(size_t)A.out_dst[e0 + q] * A.B + b];
      Amax = max(Amax, (int)(wm & 0xFFFFu));
      Bm = max(Bm, (int)(wm >> 16) - 1);
    }
  }
}

// 1 - M_i(d): 1 when some successor certainly has not started by d.
template <int kFam>
__device__ __forceinline__ float one_minus_m(const RegArgs &A, int e0, int deg, int dmax, int b, int d, int Amax) {
  if (deg == 0 || d < Amax) return 1.0f;
  float t = 0.f;
  for (int q = 0; q < dmax; ++q) {
    if (q < deg) {
      const int jc = A.out_dst[e0 + q];
      const unsigned wm = A.win[(size_t)jc * A.B + b];
      const int aj = (int)(wm & 0xFFFFu), bj = (int)(wm >> 16) - 1;
      float C, Q;
      const float mj = (d >= aj && d <= bj) ? A.mu[(size_t)jc * A.B + b] : 0.f;
      const float ij = (d >= aj && d <= bj) ? 1.0f / A.sg[(size_t)jc * A.B + b] : 1.f;
      cdf_pair<kFam>(d, mj, ij, aj, bj, C, Q);
      t = t + (1.0f - t) * Q;
    }
  }
  return t;
}

// 1 - M_i(d) = 1 - prod_j C_j(d) as a pair (the forward's product).
template <int kFam>
__device__ __forceinline__ FF one_minus_m_pair(const RegArgs &A, int e0, int deg, int dmax, int b, int d, int Amax) {
  if (deg == 0 || d < Amax) return {1.0f, 0.0f};
  FF P = {1.0f, 0.0f};
  for (int q = 0; q < dmax; ++q) {
    if (q < deg) {
      const int jc = A.out_dst[e0 + q];
      const unsigned wm = A.win[(size_t)jc * A.B + b];
      const int aj = (int)(wm & 0xFFFFu), bj = (int)(wm >> 16) - 1;
      const bool in = d >= aj && d <= bj;
      const float mj = in ? A.mu[(size_t)jc * A.B + b] : 0.f, sj = in ? A.sg[(size_t)jc * A.B + b] : 1.f;
      P = ff_mul(P, cdf_pair_ff<kFam>(A.qtab, d, mj, sj, 1.0f / sj, aj, bj));
    }
  }
  return ff_one_minus(P);
}

template <int kFam>
__global__ void __launch_bounds__(kFwdThreads) k_reg_fwd(const RegArgs A) {
  extern __shared__ __align__(16) unsigned char smem_r[];
  constexpr int T = kFwdThreads;
  constexpr unsigned FULL = 0xffffffffu;
  const int tid = threadIdx.x, RB = A.RB, Dh = A.Dh;
  unsigned *hlo = reinterpret_cast<unsigned *>(smem_r);
  unsigned *hhi = hlo + (size_t)Dh * RB;
  int *rdiff = reinterpret_cast<int *>(hhi + (size_t)Dh * RB);  // (Dh + 1) * RB
  int *rconst = rdiff + (size_t)(Dh + 1) * RB;                   // RB
  __shared__ int s_next;
  const int blk = blockIdx.x, segi = blk / A.G, g = blk % A.G;
  const int s0 = A.seg[3 * segi], s1 = A.seg[3 * segi + 1];
  const int ncell = 2 * Dh * RB + (Dh + 1) * RB + RB;
  for (int i = tid; i < ncell; i += T) hlo[i] = 0u;
  if (tid == 0) s_next = 0;
  __syncthreads();

  const int lane = tid & 31, r = tid % RB, b = g * RB + r, npw = 32 / RB;
  for (;;) {
    int base = 0;
    if (lane == 0) base = atomicAdd(&s_next, npw);
    base = __shfl_sync(FULL, base, 0);
    if (base >= s1 - s0) break;
    const int vi = s0 + base + lane / RB;
    bool valid = b < A.B && vi < s1;
    const int vcl = valid ? vi : s0;
    const int vc = A.perm[vcl];
    const float mu = valid ? A.mu[(size_t)vc * A.B + b] : 0.f, sg = valid ? A.sg[(size_t)vc * A.B + b] : 1.f;
    valid = valid && usable(mu, sg);
    const float inv_s = valid ? 1.0f / sg : 1.0f, bits = A.bits[vcl];
    int a = 0, bw = -2;
    if (valid) window(mu, sg, A.k_win, A.D, a, bw);
    const int e0 = A.out_ptr[vcl], deg = valid ? A.out_ptr[vcl + 1] - e0 : 0;
    const int dmax = __reduce_max_sync(FULL, deg);
    int Amax, Bm;
    succ_bounds(A, e0, deg, dmax, b, Amax, Bm);
    // certainly live from the end of the own window until a successor may start
    const int ib = __float2int_rn(bits);
    if (valid && ib != 0) {
      const int s = bw + 1, e = min(Amax, A.D) - 1;
      if (s <= e) range_add(rdiff, rconst, RB, r, s, e, ib, A.II);
    }
    // own window, then the tail where the successors' product varies
    const int n_own = valid ? bw - a + 1 : 0;
    const int tail_lo = max(bw + 1, Amax);
    const int n_tail = valid ? max(0, Bm - tail_lo + 1) : 0;
    const int total = n_own + n_tail;
    const int tmax = __reduce_max_sync(FULL, total);
    // the successors' product over d0 .. Bm for the backward, when the row holds it
    const int d0 = max(a, Amax);
    const bool prow = valid && deg > 0 && Bm >= d0 && Bm - d0 + 1 <= A.WP;
    float *pr = A.ptab + ((size_t)vc * A.B + (b < A.B ? b : 0)) * A.WP;
    for (int k = 0; k < tmax; ++k) {
      const bool on = k < total;
      const bool own = k < n_own;
      const int d = own ? a + k : tail_lo + (k - n_own);
      FF Ci = {1.0f, 0.0f};
      if (on && own) Ci = cdf_pair_ff<kFam>(A.qtab, d, mu, sg, inv_s, a, bw);
      const FF L = one_minus_m_pair<kFam>(A, e0, on ? deg : 0, dmax, b, d, Amax);
      if (on && prow && d >= d0) {
        const FF P = ff_one_minus(L);
        pr[d - d0] = P.h + P.l;
      }
      if (on && bits != 0.f) hist_add_pair(hlo, hhi, fold_bin(d, A.II) * RB + r, ff_mulf(ff_mul(Ci, L), bits));
    }
    __syncwarp();
  }
  __syncthreads();
  // partials [block][bin][restart]: fixed-point window parts + 2^32 x integer range adds
  if (tid < RB) {
    long long run = 0;
    long long *dst = A.rpart + (size_t)blk * Dh * RB;
    for (int d = 0; d < Dh; ++d) {
      run += rdiff[d * RB + tid];
      const int cell = d * RB + tid;
      const long long frac = (long long)(((unsigned long long)hhi[cell] << 16) + (unsigned long long)hlo[cell]);
      dst[cell] = frac + ((run + (long long)rconst[tid]) << 32);
    }
  }
}

#ifndef GAUS_FAMILY_KERNELS_ONLY
// The tail tables of the four families (GAUS_GAUSSIAN..GAUS_CAUCHY, kTailRows rows
// each, row i at z0 = i / 64): float4 {Q hi, Q lo, f hi, f lo} and float4
// {f' / 2, f'' / 6, f''' / 24, 0}, in double from the closed forms (scales c as in
// Fam<k>: logistic pi / sqrt(3), Laplace sqrt(2), Cauchy 1 / sqrt(2 ln 2)).
__global__ void k_tail_tables(float4 *tab) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= 4 * kTailRows) return;
  const int fam = i / kTailRows;
  const double z = (double)(i % kTailRows) / kTailPerUnit;
  double Q, f, f1, f2, f3;
  if (fam == GAUS_GAUSSIAN) {
    Q = 0.5 * erfc(z * 0.70710678118654752440);
    f = 0.39894228040143267794 * exp(-0.5 * z * z);
    f1 = -z * f;
    f2 = (z * z - 1.0) * f;
    f3 = (3.0 * z - z * z * z) * f;
  } else if (fam == GAUS_LOGISTIC) {
    const double c = 1.81379936423421785059, e = exp(-c * z);
    Q = e / (1.0 + e);
    f = c * Q * (1.0 - Q);
    f1 = -c * f * (1.0 - 2.0 * Q);
    f2 = -c * (f1 * (1.0 - 2.0 * Q) + 2.0 * f * f);
    f3 = -c * (f2 * (1.0 - 2.0 * Q) + 6.0 * f * f1);
  } else if (fam == GAUS_LAPLACE) {
    const double c = 1.41421356237309504880;
    Q = 0.5 * exp(-c * z);
    f = c * Q;
    f1 = -c * f;
    f2 = c * c * f;
    f3 = -c * c * c * f;
  } else {
    const double c = 0.84932180028801904272, kp = c * 0.31830988618379067154, u = c * z, g = 1.0 / (1.0 + u * u);
    Q = 0.31830988618379067154 * atan2(1.0, u);
    f = kp * g;
    f1 = kp * c * (-2.0 * u * g * g);
    f2 = kp * c * c * (6.0 * u * u - 2.0) * g * g * g;
    f3 = kp * c * c * c * 24.0 * u * (1.0 - u * u) * g * g * g * g;
  }
  float4 a, b;
  a.x = (float)Q;
  a.y = (float)(Q - (double)a.x);
  a.z = (float)f;
  a.w = (float)(f - (double)a.z);
  b.x = (float)(f1 / 2.0);
  b.y = (float)(f2 / 6.0);
  b.z = (float)(f3 / 24.0);
  b.w = 0.0f;
  tab[2 * i] = a;
  tab[2 * i + 1] = b;
}

// Reg per (restart, bin) from every block's partials: block = (group, bin),
// threads = restarts x slices of the segment list, slices combined in order.
__global__ void __launch_bounds__(256) k_reduce_reg(const long long *rpart, long long *Ureg, int B, int Dh, int RB,
                                                    int G, int nseg) {
  __shared__ long long part[256];
  const int nsl = 256 / RB;
  const int d = blockIdx.x % Dh, g = blockIdx.x / Dh;
  const int r = threadIdx.x % RB, sl = threadIdx.x / RB, b = g * RB + r;
  long long acc = 0;
  for (int s = sl; s < nseg; s += nsl) acc += rpart[((size_t)(s * G + g) * Dh + d) * RB + r];
  part[threadIdx.x] = acc;
  __syncthreads();
  if (sl == 0 && b < B) {
    long long tot = 0;
    for (int k = 0; k < nsl; ++k) tot += part[k * RB + r];
    Ureg[(size_t)b * Dh + d] = tot;
  }
}
#endif  // GAUS_FAMILY_KERNELS_ONLY

// C_j(d) of node jc (caller id), restart b, packed window wm, for the backward: the
// node pass's table row [0, C(a), ..., C(b), 1] when the window fits it (n + 3 <= W),
// else evaluated from (mu, sigma).
template <int kFam>
__device__ __forceinline__ float reg_cdf_tab(const RegArgs &A, int jc, int b, unsigned wm, int d) {
  const int aj = (int)(wm & 0xFFFFu), bj = (int)(wm >> 16) - 1;
  if (d < aj) return 0.0f;
  if (d > bj) return 1.0f;
  const size_t ix = (size_t)jc * A.B + b;
  if (bj - aj + 4 <= A.W) return __ldg(A.tab + ix * A.W + (d - aj + 1));
  const float m = __ldg(A.mu + ix), iv = 1.0f / __ldg(A.sg + ix);
  const float z = ((float)d + 0.5f - m) * iv;
  const float q = reg_tail<kFam>(z);
  return z <= 0.f ? q : 1.0f - q;
}

// 1 - M_i(d) for the backward, from the table.
template <int kFam>
__device__ __forceinline__ float one_minus_m_tab(const RegArgs &A, int e0, int deg, int dmax, int b, int d, int Amax) {
  if (deg == 0 || d < Amax) return 1.0f;
  float P = 1.0f;
  for (int q = 0; q < dmax; ++q)
    if (q < deg) {
      const int jc = A.out_dst[e0 + q];
      P *= reg_cdf_tab<kFam>(A, jc, b, A.win[(size_t)jc * A.B + b], d);
    }
  return 1.0f - P;
}

template <int kFam>
__global__ void __launch_bounds__(kFwdThreads) k_reg_bwd(const RegArgs A) {
  extern __shared__ __align__(16) unsigned char smem_rb[];
  constexpr int T = kFwdThreads;
  constexpr unsigned FULL = 0xffffffffu;
  const int tid = threadIdx.x, RB = A.RB, Dh = A.Dh;
  float *Hs = reinterpret_cast<float *>(smem_rb);  // Dh * RB
  __shared__ int s_next;
  const int blk = blockIdx.x, segi = blk / A.G, g = blk % A.G;
  const int s0 = A.seg[3 * segi], s1 = A.seg[3 * segi + 1];
  for (int i = tid; i < Dh * RB; i += T) {
    const int t = i / RB, rr = i % RB, bb = g * RB + rr;
    Hs[i] = bb < A.B ? A.Hreg[(size_t)bb * Dh + t] : 0.f;
  }
  if (tid == 0) s_next = 0;
  __syncthreads();

  const int lane = tid & 31, r = tid % RB, b = g * RB + r, npw = 32 / RB;
  for (;;) {
    int base = 0;
    if (lane == 0) base = atomicAdd(&s_next, npw);
    base = __shfl_sync(FULL, base, 0);
    if (base >= s1 - s0) break;
    const int vi = s0 + base + lane / RB;
    bool valid = b < A.B && vi < s1;
    const int vcl = valid ? vi : s0;
    const int vc = A.perm[vcl];
    const float mu = valid ? A.mu[(size_t)vc * A.B + b] : 0.f, sg = valid ? A.sg[(size_t)vc * A.B + b] : 1.f;
    valid = valid && usable(mu, sg);
    const float inv_s = valid ? 1.0f / sg : 1.0f, bits = A.bits[vcl];
    int a = 0, bw = -2;
    if (valid) window(mu, sg, A.k_win, A.D, a, bw);
    const unsigned own_w = (unsigned)a | ((unsigned)(bw + 1) << 16);
    const int e0 = A.out_ptr[vcl], deg = valid ? A.out_ptr[vcl + 1] - e0 : 0;
    const int dmax = __reduce_max_sync(FULL, deg);
    int Amax, Bm;
    succ_bounds(A, e0, deg, dmax, b, Amax, Bm);
    // the successors' product P(d), d0 <= d <= Bm, as the forward stored it (else formed
    // here from the table); below d0 = max(a, Amax) every share and 1 - M's complement
    // vanish (C_i = 0 below a; some successor certainly not started below Amax)
    const int d0 = max(a, Amax);
    const bool prow = valid && deg > 0 && Bm >= d0 && Bm - d0 + 1 <= A.WP;
    const float *pr = A.ptab + ((size_t)vc * A.B + (b < A.B ? b : 0)) * A.WP;
    // own adjoint on the own window: dL/dC_i(d) = G(d) b_i (1 - M_i(d))
    float Ao = 0.f, Bo = 0.f;
    const int n_own = valid ? bw - a + 1 : 0;
    const int nmax = __reduce_max_sync(FULL, n_own);
    for (int k = 0; k < nmax; ++k) {
      const bool on = k < n_own;
      const int d = a + k;
      const float L = (prow && d >= d0) ? 1.0f - pr[d - d0]
                                        : one_minus_m_tab<kFam>(A, e0, on && !prow ? deg : 0, dmax, b, d, Amax);
      if (on) {
        const float z = ((float)d + 0.5f - mu) * inv_s;
        const float f = reg_pdf<kFam>(z);
        const float gg = Hs[fold_bin(d, A.II) * RB + r] * bits * L;
        Ao += gg * f;
        Bo += gg * z * f;
      }
    }
    __syncwarp();
    if (valid) A.gown[(size_t)vcl * A.B + b] = make_float2(Ao, Bo);
    // successors' shares: dL/dC_j(d) = -G(d) b_i C_i(d) prod_{j' != j} C_j'(d) on j's window
    for (int q = 0; q < dmax; ++q) {
      const bool eon = q < deg;
      const int jc = eon ? A.out_dst[e0 + q] : 0;
      const unsigned wm = eon ? A.win[(size_t)jc * A.B + b] : 0u;
      const int aj = (int)(wm & 0xFFFFu), bj = (int)(wm >> 16) - 1;
      const int lo = max(aj, d0);  // C_i(d) = 0 below the own window, the product 0 below Amax
      const int cnt = eon && bits != 0.f ? max(0, bj - lo + 1) : 0;
      const float mj = cnt ? A.mu[(size_t)jc * A.B + b] : 0.f;
      const float ij = cnt ? 1.0f / A.sg[(size_t)jc * A.B + b] : 1.f;
      const int cmax = __reduce_max_sync(FULL, cnt);
      float Aj = 0.f, Bj = 0.f;
      for (int k = 0; k < cmax; ++k) {
        const bool on = k < cnt;
        const int d = lo + k;
        const float Ci = on ? reg_cdf_tab<kFam>(A, vc, b, own_w, d) : 1.0f;
        // product of the other successors' CDFs at d: P(d) / C_j(d) (C_j > 0 on j's
        // window), or formed directly where P is not stored or C_j is below 1e-30
        float prod = 1.f;
        bool direct = !prow;
        if (on && prow) {
          const float cj = reg_cdf_tab<kFam>(A, jc, b, wm, d);
          if (cj > 1e-30f) prod = pr[d - d0] / cj;
          else direct = true;
        }
        const bool dir_any = __any_sync(FULL, on && direct);
        for (int q2 = 0; q2 < dmax && dir_any; ++q2) {
          if (on && direct && q2 < deg && q2 != q) {
            const int kc2 = A.out_dst[e0 + q2];
            prod *= reg_cdf_tab<kFam>(A, kc2, b, A.win[(size_t)kc2 * A.B + b], d);
          }
        }
        if (on) {
          const float z = ((float)d + 0.5f - mj) * ij;
          const float f = reg_pdf<kFam>(z);
          const float adj = -Hs[fold_bin(d, A.II) * RB + r] * bits * Ci * prod;
          Aj += adj * f;
          Bj += adj * z * f;
        }
      }
      __syncwarp();
      if (eon) A.eslot[(size_t)(e0 + q) * A.B + b] = make_float2(Aj, Bj);
    }
  }
}

}  // namespace gaus
