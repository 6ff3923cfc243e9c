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
    for (int k = 0; k < tmax; ++k) {
      const bool on = k < total;
      const bool own = k < n_own;
      const int d = own ? a + k : tail_lo + (k - n_own);
      float Ci = 1.f, Qi;
      if (on && own) cdf_pair<kFam>(d, mu, inv_s, a, bw, Ci, Qi);
      const float L = one_minus_m<kFam>(A, e0, on ? deg : 0, dmax, b, d, Amax);
      if (on && bits != 0.f) hist_add(hlo, hhi, fold_bin(d, A.II) * RB + r, bits * Ci * L);
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
    const int e0 = A.out_ptr[vcl], deg = valid ? A.out_ptr[vcl + 1] - e0 : 0;
    const int dmax = __reduce_max_sync(FULL, deg);
    int Amax, Bm;
    succ_bounds(A, e0, deg, dmax, b, Amax, Bm);
    // own adjoint on the own window: dL/dC_i(d) = G(d) b_i (1 - M_i(d))
    float Ao = 0.f, Bo = 0.f;
    const int n_own = valid ? bw - a + 1 : 0;
    const int nmax = __reduce_max_sync(FULL, n_own);
    for (int k = 0; k < nmax; ++k) {
      const bool on = k < n_own;
      const int d = a + k;
      const float L = one_minus_m<kFam>(A, e0, on ? deg : 0, dmax, b, d, Amax);
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
      const int lo = max(aj, a);  // C_i(d) = 0 below the own window
      const int cnt = eon && bits != 0.f ? max(0, bj - lo + 1) : 0;
      const float mj = cnt ? A.mu[(size_t)jc * A.B + b] : 0.f;
      const float ij = cnt ? 1.0f / A.sg[(size_t)jc * A.B + b] : 1.f;
      const int cmax = __reduce_max_sync(FULL, cnt);
      float Aj = 0.f, Bj = 0.f;
      for (int k = 0; k < cmax; ++k) {
        const bool on = k < cnt;
        const int d = lo + k;
        float Ci = 1.f, Qi;
        if (on) cdf_pair<kFam>(d, mu, inv_s, a, bw, Ci, Qi);
        // product of the other successors' CDFs at d
        float prod = 1.f;
        for (int q2 = 0; q2 < dmax; ++q2) {
          if (on && q2 < deg && q2 != q) {
            const int kc2 = A.out_dst[e0 + q2];
            const unsigned wm2 = A.win[(size_t)kc2 * A.B + b];
            const int a2 = (int)(wm2 & 0xFFFFu), b2 = (int)(wm2 >> 16) - 1;
            const bool in2 = d >= a2 && d <= b2;
            const float m2 = in2 ? A.mu[(size_t)kc2 * A.B + b] : 0.f;
            const float i2 = in2 ? 1.0f / A.sg[(size_t)kc2 * A.B + b] : 1.f;
            float C2, Q2;
            cdf_pair<kFam>(d, m2, i2, a2, b2, C2, Q2);
            prod *= C2;
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
