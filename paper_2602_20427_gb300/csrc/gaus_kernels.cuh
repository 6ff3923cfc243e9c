// gaus_kernels.cuh -- device code of one GauS iteration (Sec. 3.2-3.3, App. B).
//
// Work item: one (node v, restart b).  A warp row of RB (16) lanes holds RB
// restarts of the same node (lanes = b; two nodes or edges per warp), so every
// mu/sigma gather of a neighbour is one coalesced 64-byte load.  Each (node,
// restart) has its window of CDF points
//   C_v(t) = F((t + 1/2 - mu_v) / sigma_v),  t in [a_v, b_v] = points within
//   window_k * sigma_v of mu_v, with C_v(t) = 0 below and 1 above (Eq. round and
// its open end bins; F the normal CDF, or another family of App. D).
//
// k_nodes   : windows, the CDF table (C at each window point, computed once per
//             (node, restart) and read by every incident edge) and bin masses ->
//             usage histogram (shared-memory fixed point, one class per block).
// k_edges   : every edge term, once per (edge, restart), from both endpoints'
//             table rows: forward sums (exact fixed point) and each endpoint's
//             unscaled partial gradients, written to per-edge slots.
// k_reduce  : usage per (restart, class, bin) from the node pass's block partials.
// k_finalize: one block per restart -- LogSumExp (Eq. max), ReLU (Eq. relu), the
//             augmented-Lagrangian coefficients and multiplier step (Sec. 3.3).
// k_update  : usage adjoint of the node's own window, the node's edge slots
//             gathered in a fixed order, the combined gradient and (optionally)
//             the Adam step.
#pragma once

#include <climits>
#include <cuda_runtime.h>
#include <stdint.h>

#include "gaus_device.cuh"
#include "gaus_internal.h"
#include "gaus_reg.cuh"

namespace gaus {

struct IterArgs {
  const float *mu, *sg;  // (V, B) caller order
  int V, B, D, II, Dh, C, RB, G, W;  // W: points per table row
  float k_win, alpha;
  const int32_t *perm;
  const float *w;
  const int32_t *lat;
  const int32_t *in_ptr, *in_src, *in_lat;
  const int32_t *out_ptr, *out_dst;
  const int32_t *bin_ptr, *bin_src, *bin_shift;
  const int32_t *bout_ptr, *bout_dst, *bout_shift;
  const int32_t *seg;
  long long *hpart;
  int2 *hspan;
  unsigned long long *fwdtot;  // (B, 3) forward sums (dep, com, rec), 2^32 fixed point
  int32_t *nonfinite;
  unsigned *win;  // (V, B) packed windows a | (b + 1) << 16, written by k_nodes
  float *tab;     // (V, B, W) CDF values at the window points, written by k_nodes
  const int4 *ed; // edge list of the edge pass (nEt = E + NB edges; k_dep_cf: ce per block)
  int nEt, ce, E;
  unsigned long long *wstat;  // (B, 2) window points / valid items of this iteration
  float4 *eslot4; // per-edge partials [side][position][restart]: producer side at
                  // the edge's index (CSR / bout order), consumer side at its
                  // CSC / bin position (+E for back edges), offset nEt * B
};

struct RedArgs {
  int B, C, Dh, RB, G;
  const int32_t *cls_seg_ptr;
  const long long *hpart;
  const int2 *hspan;
  long long *U;       // (B, C, Dh) usage, 2^32 fixed point
};

struct FinArgs {
  int B, C, Dh, RB, G;
  const long long *Ug;   // (B, C, Dh) usage from k_reduce, 2^32 fixed point
  const long long *Ureg; // (B, Dh) storage, or NULL when the storage term is off
  float *Hreg;        // (B, Dh) storage adjoint
  unsigned terms;
  float tau, rho, alpha, w_res, w_mem;
  const int32_t *cls_seg_ptr;
  const float *limit;
  const long long *hpart;
  const int2 *hspan;
  unsigned long long *fwdtot;  // (B, 3) forward sums; read and cleared
  float *lambda;      // read; updated in place when update_lambda
  int update_lambda;
  int32_t *step;      // incremented when not NULL
  float beta1, beta2; // Adam: 1 / (1 - beta1^t), 1 / sqrt(1 - beta2^t) written to coef[2], coef[3]
  float *H, *coef, *loss, *terms_out;
  int32_t *status, *nonfinite;
  unsigned long long *wstat;  // read into thr and cleared for the next iteration
  int32_t *thr;
  int W;
};

struct UpdArgs {
  // per-edge partials of the edge pass, gathered per node: out-edges (CSR positions
  // out_ptr), in-edges (in_eslot maps CSC to CSR position), back edges out
  // (positions E + bout_ptr) and in (bin_eslot maps bin to bout position)
  const int32_t *in_ptr, *in_eslot, *out_ptr;
  const int32_t *bin_ptr, *bout_ptr;
  int E, nEt, has_back;
  const float4 *eslot4;
  const float2 *eslot;               // storage term: successor shares (NULL when off)
  const float2 *gown;                // storage term: own-window adjoint (NULL when off)
  const int32_t *thr;                // per-restart long-window threshold (k_finalize)
  float *mu, *sg;  // caller order; written when adam
  int V, B, D, II, Dh, C, RB, G;
  float k_win;
  int W;  // table row length: longer own windows are done by the whole warp
  const int32_t *perm, *cls;
  const float *w;
  const float *H, *coef;
  float *grad_mu, *grad_sg;                  // gradient mode
  float *m_mu, *v_mu, *m_sg, *v_sg;          // Adam mode
  const int32_t *step_dev;                   // per-restart step (Adam mode, iterate)
  float lr, beta1, beta2, eps, sigma_min;
};

// round(x 2^32) for a forward sum x >= 0 of one item, with 32-bit conversions only.
__device__ __forceinline__ long long to_fix(float x) {
  const float xs = fmaxf(x, 0.0f) * 65536.0f;
  const float fh = floorf(xs);
  return ((long long)(unsigned)fh << 16) + (long long)__float2uint_rn((xs - fh) * 65536.0f);
}

// Window length above which an item of restart b is done by the whole warp:
// twice the restart's mean window (over all its nodes, this iteration) plus 4,
// at least 8.  It depends on restart b alone, so the
// split -- and with it every rounding -- does not depend on the other restarts.
__device__ __forceinline__ int threshold_of(unsigned long long sum, unsigned long long c) {
  if (c == 0) return 8;
  const int mean = (int)(sum / c);
  return min(1 << 20, max(8, 2 * mean + 4));
}
__device__ __forceinline__ int long_threshold(const unsigned long long *ws, int b) {
  return threshold_of(ws[2 * b], ws[2 * b + 1]);
}

// Mean window length (points) of restart b over the nodes s0..s1 of a segment,
// from the windows table; rows threads per restart.  It sees restart b's data
// only, so the split of items between the per-lane and the cooperative path --
// and with it every rounding -- does not depend on the other restarts.  The
// caller zeroes s_sum / s_cnt and synchronises before the call.
__device__ __forceinline__ int seg_mean_window(const unsigned *win, const int32_t *perm, int s0, int s1, int b,
                                               bool bok, int B, int tid, int RB, int rows, int *s_sum, int *s_cnt) {
  int sum = 0, cnt = 0;
  if (bok)
    for (int vi = s0 + tid / RB; vi < s1; vi += rows) {
      const unsigned w = win[(size_t)perm[vi] * B + b];
      const int n = (int)(w >> 16) - (int)(w & 0xffffu);
      if (n > 0) { sum += min(n, 4096); ++cnt; }
    }
  if (cnt) {
    atomicAdd(&s_sum[tid % RB], sum);
    atomicAdd(&s_cnt[tid % RB], cnt);
  }
  __syncthreads();
  const int c = s_cnt[tid % RB];
  return c ? s_sum[tid % RB] / c : 0;
}

__device__ __forceinline__ float warp_sum(float x) {
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// A neighbour's windowed CDF C_u(x): 0 below its window, 1 above it, inside it
// the table value written by k_nodes, or -- for a window the table row cannot
// hold -- evaluated from its mean and sigma.
template <int kFam>
struct Nb {
  const float *row;  // table row of (u, b): [0, C(a), ..., C(b), 1, ...]
  int a, b;          // window points [a, b]
  bool tab;          // the row holds the window with both sentinels (b - a + 3 <= W)
  float mu, inv;
  // any window: 0 below, 1 above, the table or a direct evaluation inside
  __device__ __forceinline__ float at(int x) const {
    if (x < a) return 0.0f;
    if (x > b) return 1.0f;
    return tab ? __ldg(row + (x - a + 1)) : Fam<kFam>::cdf(((float)x + 0.5f - mu) * inv);
  }
  // a tabled window: the sentinels make the clamped index exact everywhere
  __device__ __forceinline__ float at_tab(int x) const {
    return __ldg(row + min(max(x - a + 1, 0), b - a + 2));
  }
  // a window the table row cannot hold: direct evaluation
  __device__ __forceinline__ float at_direct(int x) const {
    return x < a ? 0.0f : (x > b ? 1.0f : Fam<kFam>::cdf(((float)x + 0.5f - mu) * inv));
  }
  template <bool kTab>
  __device__ __forceinline__ float val(int x) const {
    return kTab ? at_tab(x) : at_direct(x);
  }
};

// Window, CDF table and usage histogram (Eq. round, Eq. usage).  Block = one
// segment (nodes of one class) x one restart group; lanes are restarts.  Every
// (node, restart) gets its window [a, b] of points within window_k sigma, the CDF
// values C(a..b) (from Q(|z|) = Phi(-|z|), so that both tails keep relative
// accuracy) written to its table row for the edge pass, and its bin masses added
// to the block's histogram as round(w P 2^32) in two exact 16-bit halves.  The
// span of bins the block touched goes to the partials read by k_reduce.
template <int kFam>
__global__ void __launch_bounds__(kFwdThreads) k_nodes(const IterArgs A) {
  extern __shared__ __align__(16) unsigned char smem[];
  constexpr int T = kFwdThreads;
  constexpr unsigned FULL = 0xffffffffu;
  const int tid = threadIdx.x, lane = tid & 31, RB = A.RB, Dh = A.Dh, W = A.W;
  unsigned *hlo = reinterpret_cast<unsigned *>(smem);  // [bin][restart]
  unsigned *hhi = hlo + (size_t)Dh * RB;
  __shared__ int s_lo, s_hi, s_next, s_ws[32], s_wc[32];

  const int blk = blockIdx.x, segi = blk / A.G, g = blk % A.G;
  const int s0 = A.seg[3 * segi], s1 = A.seg[3 * segi + 1];
  for (int i = tid; i < 2 * RB * Dh; i += T) hlo[i] = 0u;
  if (tid == 0) { s_lo = INT_MAX; s_hi = INT_MIN; s_next = 0; }
  if (tid < 32) { s_ws[tid] = 0; s_wc[tid] = 0; }
  __syncthreads();

  const int r = tid % RB, b = g * RB + r;
  const bool bok = b < A.B;
  int lo = INT_MAX, hi = INT_MIN;
  const int npw = 32 / RB;
  for (;;) {
    int base = 0;
    if (lane == 0) base = atomicAdd(&s_next, npw);
    base = __shfl_sync(FULL, base, 0);
    if (base >= s1 - s0) break;
    const int vi = s0 + base + lane / RB;
    const bool present = bok && vi < s1;
    const int vcl = present ? vi : s0;
    const int vc = A.perm[vcl];
    const size_t ci = (size_t)vc * A.B + (bok ? b : 0);
    const float mu = present ? A.mu[ci] : 0.f, sg = present ? A.sg[ci] : 1.f;
    const bool valid = present && usable(mu, sg);
    if (present && !valid) A.nonfinite[b] = 1;
    const float inv_s = valid ? 1.0f / sg : 1.0f, wv = A.w[vcl];
    int a = 0, bw = -1;
    if (valid) window(mu, sg, A.k_win, A.D, a, bw);
    if (present) A.win[ci] = (unsigned)a | ((unsigned)(bw + 1) << 16);
    const int n = valid ? bw - a + 1 : -1;  // points; -1: nothing to add
    if (valid) {
      atomicAdd(&s_ws[r], min(n, 4096));
      atomicAdd(&s_wc[r], 1);
    }
    // windows much longer than the warp's typical one go to the cooperative pass
    // (the results do not depend on the split: the table values are per point
    // and the histogram sums are exact)
    const int nact = __popc(__ballot_sync(FULL, valid));
    const int mean = nact ? __reduce_add_sync(FULL, max(n, 0)) / nact : 0;
    const bool is_long = valid && n > max(8, 2 * mean + 8);
    const int nl = is_long ? -1 : n;
    const int nmax = __reduce_max_sync(FULL, nl);
    // table row [0, C(a), ..., C(b), 1] when the window fits it
    float *row = A.tab + ci * W;
    const bool tabled = n >= 0 && n + 3 <= W;
    if (tabled && !is_long) row[0] = 0.0f;
    float zp = 0.f, qp = 0.f;
    for (int j = 0; j <= nmax; ++j) {
      const bool pt = j < nl;  // point a+j exists
      const float zc = ((float)(a + j) + 0.5f - mu) * inv_s;
      const float qc = pt ? Fam<kFam>::tail(zc) : 0.f;
      if (tabled && j <= nl) row[j + 1] = pt ? (zc <= 0.f ? qc : 1.0f - qc) : 1.0f;
      if (j <= nl) hist_add(hlo, hhi, fold_bin(a + j, A.II) * RB + r, wv * bin_mass(pt, j == 0, zc, qc, zp, qp));
      zp = zc;
      qp = qc;
    }
    __syncwarp();
    unsigned longmask = __ballot_sync(FULL, is_long);
    while (longmask) {
      const int src = __ffs(longmask) - 1;
      longmask &= longmask - 1;
      const int l_a = __shfl_sync(FULL, a, src), l_n = __shfl_sync(FULL, n, src);
      const int l_r = __shfl_sync(FULL, r, src), l_vc = __shfl_sync(FULL, vc, src);
      const int l_b = __shfl_sync(FULL, b, src);
      const float l_mu = __shfl_sync(FULL, mu, src), l_inv = __shfl_sync(FULL, inv_s, src);
      const float l_w = __shfl_sync(FULL, wv, src);
      float *l_row = A.tab + ((size_t)l_vc * A.B + l_b) * W;
      const bool l_tabled = l_n + 3 <= W;
      if (l_tabled && lane == 0) l_row[0] = 0.0f;
      float z_carry = 0.f, q_carry = 0.f;
      for (int p0 = 0; p0 <= l_n; p0 += 32) {
        const int p = p0 + lane;
        const bool pt = p < l_n;
        const float z = ((float)(l_a + p) + 0.5f - l_mu) * l_inv;
        const float q = pt ? Fam<kFam>::tail(z) : 0.f;
        if (l_tabled && p <= l_n) l_row[p + 1] = pt ? (z <= 0.f ? q : 1.0f - q) : 1.0f;
        float zpv = __shfl_up_sync(FULL, z, 1), qpv = __shfl_up_sync(FULL, q, 1);
        if (lane == 0) { zpv = z_carry; qpv = q_carry; }
        if (p <= l_n) hist_add(hlo, hhi, fold_bin(l_a + p, A.II) * RB + l_r, l_w * bin_mass(pt, p == 0, z, q, zpv, qpv));
        z_carry = __shfl_sync(FULL, z, 31);
        q_carry = __shfl_sync(FULL, q, 31);
      }
    }
    if (valid) {
      lo = min(lo, a);
      hi = max(hi, bw + 1);
    }
  }

  // ---- histogram rows restricted to the folded span the block touched ----
  if (lo <= hi) {
    atomicMin(&s_lo, lo);
    atomicMax(&s_hi, hi);
  }
  __syncthreads();
  // per-restart window statistics (exact integer sums, any order)
  if (tid < RB && bok && s_wc[tid]) {
    atomicAdd(&A.wstat[2 * b], (unsigned long long)s_ws[tid]);
    atomicAdd(&A.wstat[2 * b + 1], (unsigned long long)s_wc[tid]);
  }
  int flo = s_lo, fhi = s_hi;
  if (flo > fhi) {
    flo = 1;
    fhi = 0;
  } else if (A.II > 0) {
    if (fhi - flo + 1 >= A.II) {
      flo = 0;
      fhi = A.II - 1;
    } else {
      const int x = flo % A.II, y = fhi % A.II;
      if (x <= y) { flo = x; fhi = y; } else { flo = 0; fhi = A.II - 1; }
    }
  }
  if (tid == 0) A.hspan[blk] = make_int2(flo, fhi);
  const int len = fhi - flo + 1;
  if (len > 0) {
    // partials laid out [block][bin][restart]
    long long *dst = A.hpart + (size_t)blk * Dh * RB;
    for (int i = tid; i < RB * len; i += T) {
      const int cell = flo * RB + i;
      dst[cell] = (long long)(((unsigned long long)hhi[cell] << 16) + (unsigned long long)hlo[cell]);
    }
  }
}

// One (edge, restart) whose endpoint windows are not both in the table, done by
// the whole warp with lanes over the points of each endpoint (32 at a time).
// Same terms and formulas as the per-lane path, with the own values evaluated
// directly.  Returns the warp-reduced sums on every lane: the producer's and the
// consumer's partials and the edge's forward sums.
template <int kFam, bool kDep, bool kCom>
__device__ void coop_edge(const IterArgs &A, bool back, int L, const Nb<kFam> &U, const Nb<kFam> &Vn, float4 &su, float4 &sv,
                          float &fd, float &fc, float &fr) {
  const int lane = threadIdx.x & 31;
  float s[11] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};  // su, sv, fd, fc, fr
  // consumer side: own = v
  const int nv = Vn.b - Vn.a + 1;
  for (int base = 0; base == 0 || base < nv; base += 32) {
    const int pidx = base + lane;
    const bool pt = pidx < nv;
    const int t = Vn.a + pidx;
    const float z = ((float)t + 0.5f - Vn.mu) * Vn.inv;
    const float q = pt ? Fam<kFam>::tail(z) : 0.f;
    const float Cv = pt ? (z <= 0.f ? q : 1.0f - q) : 1.0f;
    const float f = pt ? Fam<kFam>::pdf(z) : 0.f;
    const float zf = z * f;
    if (!back) {
      if (pt) {
        const float c_hi = U.at(t + 1 - L);
        const float p = c_hi - U.at(t - L);
        if (kDep) { s[8] += Cv * p; s[4] += p * f; s[5] += p * zf; }
        if (kCom) {
          const float cu = (L == 1) ? c_hi : U.at(t);
          s[9] += cu * (1.0f - Cv);
          s[6] -= A.alpha * cu * f;
          s[7] -= A.alpha * cu * zf;
        }
      }
      if (kDep && base == 0 && lane == 0) s[8] += 1.0f - U.at(Vn.b + 1 - L);
    } else {
      if (pt) {
        const float p = U.at(t + 1 - L) - U.at(t - L);
        s[10] += Cv * p; s[4] += p * f; s[5] += p * zf;
      }
      if (base == 0 && lane == 0) s[10] += 1.0f - U.at(Vn.b + 1 - L);
    }
  }
  // producer side: own = u
  const int nu = U.b - U.a + 1;
  for (int base = 0; base == 0 || base < nu; base += 32) {
    const int pidx = base + lane;
    const bool pt = pidx < nu;
    const int x = U.a + pidx;
    const float z = ((float)x + 0.5f - U.mu) * U.inv;
    const float q = pt ? Fam<kFam>::tail(z) : 0.f;
    const float Cu = pt ? (z <= 0.f ? q : 1.0f - q) : 1.0f;
    const float f = pt ? Fam<kFam>::pdf(z) : 0.f;
    const float zf = z * f;
    if (!back) {
      if (pt) {
        const float c_hi = Vn.at(x + L), c_lo = Vn.at(x + L - 1);
        if (kDep) { const float p = c_hi - c_lo; s[0] -= p * f; s[1] -= p * zf; }
        if (kCom) {
          const float cw = (L == 1) ? c_lo : Vn.at(x);
          s[2] += A.alpha * (1.0f - cw) * f;
          s[3] += A.alpha * (1.0f - cw) * zf;
          if (x < Vn.a) s[9] += Cu;
        }
      }
      if (kCom && base == 0 && lane == 0) s[9] += (float)max(0, Vn.a - 1 - U.b);
    } else if (pt) {
      const float p = Vn.at(x + L) - Vn.at(x + L - 1);
      s[0] -= p * f; s[1] -= p * zf;
    }
  }
  __syncwarp();
#pragma unroll
  for (int k = 0; k < 11; ++k) s[k] = warp_sum(s[k]);
  su = make_float4(s[0], s[1], s[2], s[3]);
  sv = make_float4(s[4], s[5], s[6], s[7]);
  fd = s[8]; fc = s[9]; fr = s[10];
}

// Per-lane terms of one (edge, restart) from both endpoints: the consumer's own
// window (own = v) and then the producer's (own = u), each visiting only the own
// points where a term can be nonzero.  kTab: both rows are in the table (clamped
// reads against the sentinels); otherwise the values are evaluated directly.
// All lanes of the warp call it (warp-wide trip counts).
template <int kFam, bool kDep, bool kCom, bool kUnit, bool kTab>
__device__ __forceinline__ void edge_sides(const IterArgs &A, bool fw, bool bk, int L, const Nb<kFam> &U, const Nb<kFam> &Vn,
                                           float4 &su, float4 &sv, float &fd, float &fc, float &fr) {
  constexpr unsigned FULL = 0xffffffffu;
  const int nu = U.b - U.a + 1, nv = Vn.b - Vn.a + 1;
  const bool back = bk;
  // own point j of the consumer (v) / producer (u): C from the table, phi, z phi
  auto own = [&](const Nb<kFam> &o, int j, float &C, float &f, float &zf) {
    const float z = ((float)(o.a + j) + 0.5f - o.mu) * o.inv;
    C = kTab ? __ldg(o.row + j + 1) : Fam<kFam>::cdf(z);
    f = Fam<kFam>::pdf(z);
    zf = z * f;
  };

  // ---- consumer side (own = v):
  //   V_e = 1 - C_u(b_v + 1 - L) + sum_{t in own} C_v(t) P_u(t + 1 - L)
  //   dV_e/dC_v(t) = P_u(t + 1 - L);  L_com,e part = sum_{t in own} C_u(t) (1 - C_v(t))
  //   dL_com,e/dC_v(t) = -C_u(t)
  {
    // P_u(t+1-L) != 0 for t in [au+L-1, bu+L]; C_u(t) != 0 for t >= au
    int jlo = 0, jhi = -1;
    if (fw) {
      jlo = max(0, U.a + min(kDep ? L - 1 : 0, 0) - Vn.a);
      jhi = kCom ? nv - 1 : min(nv - 1, U.b + L - Vn.a);
    } else if (bk) {
      jlo = max(0, U.a + L - 1 - Vn.a);
      jhi = min(nv - 1, U.b + L - Vn.a);
    }
    const int cnt = jhi >= jlo ? jhi - jlo + 1 : 0;
    const int cmax = __reduce_max_sync(FULL, cnt);
    float c_lo = cnt ? U.template val<kTab>(Vn.a + jlo - L) : 0.f;
    for (int k2 = 0; k2 < cmax; ++k2) {
      if (k2 < cnt) {
        const int j = jlo + k2, t = Vn.a + j;
        const float c_hi = U.template val<kTab>(t + 1 - L);
        const float p = c_hi - c_lo;
        float Cv, f, zf;
        own(Vn, j, Cv, f, zf);
        if (back) {
          fr += Cv * p;
          sv.x += p * f;
          sv.y += p * zf;
        } else {
          if (kDep) {
            fd += Cv * p;
            sv.x += p * f;
            sv.y += p * zf;
          }
          if (kCom) {
            const float cu = (kUnit || L == 1) ? c_hi : U.template val<kTab>(t);
            fc += cu * (1.0f - Cv);
            sv.z -= A.alpha * cu * f;
            sv.w -= A.alpha * cu * zf;
          }
        }
        c_lo = c_hi;
      }
    }
    __syncwarp();
    if ((kDep && fw) || bk) {
      const float tail = 1.0f - U.template val<kTab>(Vn.b + 1 - L);
      if (back) fr += tail; else fd += tail;
    }
  }
  // ---- producer side (own = u):
  //   dV_e/dC_u(x) = -P_v(x + L), nonzero for x in [av-L, bv+1-L]
  //   dL_com,e/dC_u(x) = 1 - C_v(x), nonzero for x <= bv
  //   L_com,e part = sum_{x in own, x < a_v} C_u(x) + max(0, a_v - 1 - b_u)
  {
    int jlo = 0, jhi = -1;
    if (fw || bk) {
      jlo = max(0, Vn.a - L - U.a);
      jhi = min(nu - 1, Vn.b + 1 - L - U.a);
      if (kCom && fw) {
        jlo = 0;
        jhi = max(jhi, min(nu - 1, Vn.b - U.a));
      }
    }
    const int cnt = jhi >= jlo ? jhi - jlo + 1 : 0;
    const int cmax = __reduce_max_sync(FULL, cnt);
    float c_lo = cnt ? Vn.template val<kTab>(U.a + jlo + L - 1) : 0.f;
    for (int k2 = 0; k2 < cmax; ++k2) {
      if (k2 < cnt) {
        const int j = jlo + k2, x = U.a + j;
        const float c_hi = Vn.template val<kTab>(x + L);
        float Cu, f, zf;
        own(U, j, Cu, f, zf);
        if (back || kDep) {
          const float p = c_hi - c_lo;
          su.x -= p * f;
          su.y -= p * zf;
        }
        if (kCom && !back) {
          const float cw = (kUnit || L == 1) ? c_lo : Vn.template val<kTab>(x);
          su.z += A.alpha * (1.0f - cw) * f;
          su.w += A.alpha * (1.0f - cw) * zf;
          if (x < Vn.a) fc += Cu;
        }
        c_lo = c_hi;
      }
    }
    __syncwarp();
    if (kCom && fw) fc += (float)max(0, Vn.a - 1 - U.b);
  }
}

// Edge pass (Eq. dep, Eq. com, App. B.3).  Block = a chunk of the edge list x one
// restart group; lane = (edge, restart).  Each edge term is a dot product of one
// endpoint's window with the other endpoint's CDF shifted by the latency; both
// endpoints' CDF values come from the table written by k_nodes.  Per (edge,
// restart) the pass writes the producer's and the consumer's partials
// (dV/dmu-, dV/dsigma-type sums: Ad, Bd, Ao, Bo for a forward edge, Ar, Br for a
// back edge) to the edge's two slots, which k_update gathers per node in a fixed
// order, and adds the edge's forward sums (exact fixed point) to the block's.
// Per lane, an endpoint whose window the table row cannot hold is evaluated
// directly; an edge with an endpoint window longer than the restart's threshold
// is done by the whole warp (coop_edge).  kUnit: every edge has latency 1 (no
// back edges), so C_u(t) is the bin mass's upper value.
template <int kFam, bool kDep, bool kCom, bool kRec, bool kUnit>
__global__ void __launch_bounds__(kFwdThreads, 4) k_edges(const IterArgs A) {
  constexpr int T = kFwdThreads;
  constexpr unsigned FULL = 0xffffffffu;
  __shared__ long long s_red[3 * T];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, RB = A.RB, epw = 32 / RB;
  // block = one restart group; its warps take rows of epw edges grid-stride over
  // the group's blocks, so each warp's rows are spread over the whole edge list
  const int g = blockIdx.x % A.G, nbg = gridDim.x / A.G;
  const int r = tid % RB, b = g * RB + r;
  const bool bok = b < A.B;
  const int thr = bok ? long_threshold(A.wstat, b) : A.W;
  long long xdep = 0, xcom = 0, xrec = 0;  // forward sums, exact (order-free) fixed point
  const int nrows = (A.nEt + epw - 1) / epw, rstride = nbg * (T / 32);
  for (int row = (blockIdx.x / A.G) * (T / 32) + warp; row < nrows; row += rstride) {
    const int e = row * epw + lane / RB;
    const bool present = bok && e < A.nEt;
    const int4 ed = present ? __ldg(A.ed + e) : make_int4(0, 0, 0, 0);
    const int uc = ed.x, vc = ed.y, L = kUnit ? 1 : ed.z;
    const bool back = (ed.w & 1) != 0;
    const int cpos = (ed.w >> 1) + (back ? A.E : 0);  // consumer-side slot
    const size_t iu = (size_t)uc * A.B + (bok ? b : 0), iv = (size_t)vc * A.B + (bok ? b : 0);
    const float mu_u = present ? A.mu[iu] : 0.f, sg_u = present ? A.sg[iu] : 1.f;
    const float mu_v = present ? A.mu[iv] : 0.f, sg_v = present ? A.sg[iv] : 1.f;
    const unsigned wu = present ? __ldg(A.win + iu) : 0u, wv = present ? __ldg(A.win + iv) : 0u;
    const bool on = present && usable(mu_u, sg_u) && usable(mu_v, sg_v);
    Nb<kFam> U, Vn;
    U.a = (int)(wu & 0xFFFFu); U.b = (int)(wu >> 16) - 1; U.row = A.tab + iu * A.W;
    Vn.a = (int)(wv & 0xFFFFu); Vn.b = (int)(wv >> 16) - 1; Vn.row = A.tab + iv * A.W;
    U.mu = on ? mu_u : 0.f; U.inv = on ? __frcp_rn(sg_u) : 1.f;
    Vn.mu = on ? mu_v : 0.f; Vn.inv = on ? __frcp_rn(sg_v) : 1.f;
    const int nu = U.b - U.a + 1, nv = Vn.b - Vn.a + 1;
    U.tab = nu + 3 <= A.W;
    Vn.tab = nv + 3 <= A.W;
    const bool is_long = on && (nu > thr || nv > thr);
    const bool ps = on && !is_long;                 // per-lane path
    const bool fw = ps && !back && (kDep || kCom);  // forward edge terms
    const bool bk = kRec && ps && back;             // back edge term
    float4 su = make_float4(0.f, 0.f, 0.f, 0.f), sv = make_float4(0.f, 0.f, 0.f, 0.f);
    float fd = 0.f, fc = 0.f, fr = 0.f;

    // ---- per-lane terms: both rows in the table (branch-free reads), then, if any
    // lane needs it, the lanes with a window the table cannot hold ----
    const bool tabbed = U.tab && Vn.tab;
    edge_sides<kFam, kDep, kCom, kUnit, true>(A, fw && tabbed, bk && tabbed, L, U, Vn, su, sv, fd, fc, fr);
    if (__any_sync(FULL, (fw || bk) && !tabbed))
      edge_sides<kFam, kDep, kCom, kUnit, false>(A, fw && !tabbed, bk && !tabbed, L, U, Vn, su, sv, fd, fc, fr);

    // ---- cooperative pass over this warp's long (edge, restart) items ----
    unsigned longmask = __ballot_sync(FULL, is_long);
    while (longmask) {
      const int src = __ffs(longmask) - 1;
      longmask &= longmask - 1;
      Nb<kFam> lu, lv;
      lu.a = __shfl_sync(FULL, U.a, src); lu.b = __shfl_sync(FULL, U.b, src);
      lu.tab = __shfl_sync(FULL, (int)U.tab, src) != 0;
      lu.mu = __shfl_sync(FULL, U.mu, src); lu.inv = __shfl_sync(FULL, U.inv, src);
      lv.a = __shfl_sync(FULL, Vn.a, src); lv.b = __shfl_sync(FULL, Vn.b, src);
      lv.tab = __shfl_sync(FULL, (int)Vn.tab, src) != 0;
      lv.mu = __shfl_sync(FULL, Vn.mu, src); lv.inv = __shfl_sync(FULL, Vn.inv, src);
      const int l_uc = __shfl_sync(FULL, uc, src), l_vc = __shfl_sync(FULL, vc, src);
      const int l_b = __shfl_sync(FULL, b, src), l_L = __shfl_sync(FULL, L, src);
      const bool l_back = __shfl_sync(FULL, (int)back, src) != 0;
      lu.row = A.tab + ((size_t)l_uc * A.B + l_b) * A.W;
      lv.row = A.tab + ((size_t)l_vc * A.B + l_b) * A.W;
      float4 csu, csv;
      float cfd, cfc, cfr;
      if (!l_back) coop_edge<kFam, kDep, kCom>(A, false, l_L, lu, lv, csu, csv, cfd, cfc, cfr);
      else coop_edge<kFam, true, false>(A, true, l_L, lu, lv, csu, csv, cfd, cfc, cfr);
      if (lane == src) {
        su = csu; sv = csv;
        fd = cfd; fc = cfc; fr = cfr;
      }
    }
    if (present) {
      A.eslot4[(size_t)e * A.B + b] = su;
      A.eslot4[((size_t)A.nEt + cpos) * A.B + b] = sv;
    }
    xdep += to_fix(fd);
    xcom += to_fix(fc);
    xrec += to_fix(fr);
  }

  // ---- per-restart forward sums of this block ----
  s_red[0 * T + tid] = xdep;
  s_red[1 * T + tid] = xcom;
  s_red[2 * T + tid] = xrec;
  __syncthreads();
  if (tid < RB && bok) {
    long long acc[3] = {0, 0, 0};
    for (int row = 0; row < T / RB; ++row)
      for (int k = 0; k < 3; ++k) acc[k] += s_red[k * T + row * RB + tid];
    // per-restart totals: exact integer sums, any order
    for (int k = 0; k < 3; ++k)
      if (acc[k]) atomicAdd(&A.fwdtot[3 * b + k], (unsigned long long)acc[k]);
  }
}

#ifndef GAUS_FAMILY_KERNELS_ONLY
// Continuous dependency penalty (term GAUS_DEP_CF; a variant, not the paper's
// binned Eq. dep): per forward edge u -> v and restart, Phi(z) with
// z = m / s, m = mu_u + Lat(u) - mu_v, s = sqrt(sigma_u^2 + sigma_v^2), the
// probability that X_u + Lat(u) > X_v for the unrounded independent normals.
// Same blocks and lanes as the edge pass (a chunk of the edge list x a restart
// group, lane = (edge, restart)), run after it: it overwrites the dependency
// halves (.x, .y) of the edge's two slots in the edge pass's convention
// (dV/dmu = -A / sigma, dV/dsigma = -B / sigma of the slot's node) and adds the
// exact fixed-point sum to the restart's dependency total.
__global__ void __launch_bounds__(kFwdThreads) k_dep_cf(const IterArgs A) {
  constexpr int T = kFwdThreads;
  __shared__ long long s_red[T];
  const int tid = threadIdx.x, RB = A.RB;
  const int blk = blockIdx.x, ch = blk / A.G, g = blk % A.G;
  const int e_begin = ch * A.ce, e_end = min(A.E, e_begin + A.ce);
  const int r = tid % RB, b = g * RB + r;
  const bool bok = b < A.B;
  long long xdep = 0;
  for (int e = e_begin + tid / RB; bok && e < e_end; e += T / RB) {
    const int4 ed = __ldg(A.ed + e);
    const size_t iu = (size_t)ed.x * A.B + b, iv = (size_t)ed.y * A.B + b;
    const float mu_u = A.mu[iu], sg_u = A.sg[iu], mu_v = A.mu[iv], sg_v = A.sg[iv];
    float2 pu = make_float2(0.f, 0.f), pv = make_float2(0.f, 0.f);
    if (usable(mu_u, sg_u) && usable(mu_v, sg_v)) {
      const float m = mu_u + (float)ed.z - mu_v;
      const float rs = rsqrtf(sg_u * sg_u + sg_v * sg_v);
      const float z = m * rs;
      const float q = tail_fast(z);
      xdep += to_fix(z <= 0.f ? q : 1.0f - q);
      const float f = kInvSqrt2Pi * __expf(-0.5f * z * z);
      // dPhi/dmu_u = f / s, dPhi/dmu_v = -f / s, dPhi/dsigma_x = -f m sigma_x / s^3
      pu = make_float2(-sg_u * f * rs, f * z * sg_u * sg_u * rs * rs);
      pv = make_float2(sg_v * f * rs, f * z * sg_v * sg_v * rs * rs);
    }
    *reinterpret_cast<float2 *>(&A.eslot4[(size_t)e * A.B + b]) = pu;
    *reinterpret_cast<float2 *>(&A.eslot4[((size_t)A.nEt + (ed.w >> 1)) * A.B + b]) = pv;
  }
  s_red[tid] = xdep;
  __syncthreads();
  if (tid < RB && bok) {
    long long acc = 0;
    for (int row = 0; row < T / RB; ++row) acc += s_red[row * RB + tid];
    if (acc) atomicAdd(&A.fwdtot[3 * b], (unsigned long long)acc);
  }
}

// Usage per (restart, class, bin) from the partials of every block of the class:
// block = (group g, class c, bin d).  The class's segment spans are staged in
// shared memory first, so that every thread then issues its partial loads
// independently (restarts x slices of the segment list); slices are combined in a
// fixed order (exact int64 sums, kept in 2^32 fixed point).
__global__ void __launch_bounds__(256) k_reduce(const RedArgs A) {
  __shared__ long long part[256];
  __shared__ int2 s_sp[kReduceSpans];
  const int RB = A.RB, Dh = A.Dh, nsl = 256 / RB;
  int x = blockIdx.x;
  const int d = x % Dh; x /= Dh;
  const int c = x % A.C, g = x / A.C;
  const int r = threadIdx.x % RB, sl = threadIdx.x / RB, b = g * RB + r;
  const int s_beg = A.cls_seg_ptr[c], s_end = A.cls_seg_ptr[c + 1];
  long long acc = 0;
  for (int t0 = s_beg; t0 < s_end; t0 += kReduceSpans) {
    const int t1 = min(s_end, t0 + kReduceSpans);
    __syncthreads();
    for (int s = t0 + threadIdx.x; s < t1; s += 256) s_sp[s - t0] = A.hspan[s * A.G + g];
    __syncthreads();
#pragma unroll 8
    for (int s = t0 + sl; s < t1; s += nsl) {
      const int2 sp = s_sp[s - t0];
      if (d >= sp.x && d <= sp.y) acc += __ldcg(A.hpart + ((size_t)(s * A.G + g) * Dh + d) * RB + r);
    }
  }
  part[threadIdx.x] = acc;
  __syncthreads();
  if (sl == 0 && b < A.B) {
    long long tot = 0;
    for (int k = 0; k < nsl; ++k) tot += part[k * RB + r];
    A.U[((size_t)b * A.C + c) * Dh + d] = tot;
  }
}
#endif  // GAUS_FAMILY_KERNELS_ONLY

// exp((U - m) / tau) of an exact 2^32 fixed-point difference du = U - m <= 0 (the
// softmax weight of Eq. max), with the exponent kept as a pair of floats: du 2^-32
// is hi + a + b exactly (hi its integer part, a and b the top 24 and the low 8 bits
// of its fraction), x = (hi + a + b) / tau = xh + xl with the division's remainder
// taken through an FMA, and exp(x) = exp(xh) (1 + xl).  Rounding du to one float
// first would cost |x| ulps of relative error, large for a small tau.
__device__ __forceinline__ float soft_exp(long long du, float tau) {
  const int hi = (int)(du >> 32);
  const unsigned lo = (unsigned)((unsigned long long)du & 0xffffffffull);
  const float a = (float)(lo >> 8) * 5.9604644775390625e-08f;    // 2^-24
  const float b = (float)(lo & 255u) * 2.3283064365386963e-10f;  // 2^-32
  const float fh = (float)hi;
  const float s = fh + a;  // two-sum: s + e1 = fh + a exactly
  const float bv = s - fh;
  const float e1 = (fh - (s - bv)) + (a - bv);
  const float xh = s / tau;
  const float xl = (fmaf(-xh, tau, s) + (e1 + b)) / tau;
  return expf(xh) * (1.0f + xl);
}

// Deterministic block reductions over 256 threads: a fixed xor-shuffle tree per
// warp, then the 8 warp results in order.
__device__ __forceinline__ float block_sum_f(float x, float *sh) {
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = x;
  __syncthreads();
  float t = 0.f;
  for (int w = 0; w < 8; ++w) t += sh[w];
  __syncthreads();
  return t;
}
__device__ __forceinline__ long long block_sum_i64(long long x, long long *sh) {
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = x;
  __syncthreads();
  long long t = 0;
  for (int w = 0; w < 8; ++w) t += sh[w];
  __syncthreads();
  return t;
}
__device__ __forceinline__ long long block_max_ll(long long x, long long *sh) {
  for (int o = 16; o > 0; o >>= 1) x = max(x, (long long)__shfl_xor_sync(0xffffffffu, x, o));
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = x;
  __syncthreads();
  long long t = sh[0];
  for (int w = 1; w < 8; ++w) t = max(t, sh[w]);
  __syncthreads();
  return t;
}

#ifndef GAUS_FAMILY_KERNELS_ONLY
// One block (256 threads) per restart; kSmem: the restart's usage and storage rows
// are staged in shared memory (else read in place: long horizons, many classes).
// Usage and storage stay exact 2^32 fixed point (max and ReLU excess in integers);
// the softmax runs in fp32 on exact differences from the max, and only thread 0
// assembles the loss in fp64.
template <bool kSmem>
__global__ void __launch_bounds__(256) k_finalize(const FinArgs A) {
  extern __shared__ __align__(16) unsigned char smem_f[];
  long long *U = reinterpret_cast<long long *>(smem_f);  // (C + 1) * Dh
  __shared__ long long s_m[kMaxClasses + 1], s_R[kMaxClasses];
  __shared__ float s_s[kMaxClasses + 1];
  const int b = blockIdx.x, tid = threadIdx.x, Dh = A.Dh;
  const float kInvFixF = 2.3283064365386963e-10f;

  // the restart's scalars, all loaded before any store (the stores below could
  // alias them): forward sums of the edge pass, multipliers, window statistics,
  // nonfinite flag, Adam step
  __shared__ float s_f3[3];
  __shared__ unsigned long long s_fw[3], s_ws[2];
  __shared__ float s_lam[GAUS_K];
  __shared__ int s_bad, s_step;
  if (tid < 3) s_fw[tid] = A.fwdtot[3 * b + tid];
  if (tid >= 32 && tid < 32 + GAUS_K) s_lam[tid - 32] = A.lambda[(size_t)b * GAUS_K + tid - 32];
  if (tid >= 64 && tid < 66) s_ws[tid - 64] = A.wstat[2 * b + tid - 64];
  if (tid == 96) s_bad = A.nonfinite[b];
  if (tid == 128) s_step = A.step ? A.step[b] : 0;
  // the restart's usage rows (then the storage row) in shared memory when they fit,
  // else read from global memory where they are used (long horizons, many classes)
  const long long *Ug = A.Ug + (size_t)b * A.C * Dh, *Ur = A.Ureg ? A.Ureg + (size_t)b * Dh : nullptr;
  auto uget = [&](int c, int t) -> long long {
    return kSmem ? U[c * Dh + t] : (c < A.C ? Ug[c * Dh + t] : Ur[t]);
  };
  if (kSmem) {
    for (int i = tid; i < A.C * Dh; i += 256) U[i] = Ug[i];
    if (A.Ureg)
      for (int t = tid; t < Dh; t += 256) U[A.C * Dh + t] = Ur[t];
  }
  if (tid < A.C) {
    const float R = A.limit[tid];
    // limits in fixed point; an infinite or huge limit never binds
    s_R[tid] = (isfinite(R) && R < 1.0e9f) ? (long long)R * 4294967296LL +
                                                   (long long)((R - floorf(R)) * 4294967296.0f)
                                           : LLONG_MAX;
  }
  __syncthreads();


  // per class: the max (Eq. max, max shifted out) and the exact ReLU excess over
  // finite limits (Eq. relu) in one pass, then the sums of exp; every class is
  // warp-reduced first and the warps are combined in order after one barrier
  const int nh = A.C + (A.Ureg ? 1 : 0);
  const int lane = tid & 31, wid = tid >> 5;
  __shared__ long long s_wm[kMaxClasses + 1][8], s_wx[8], s_ex;
  __shared__ float s_wsum[kMaxClasses + 1][8];
  long long ex = 0;
  for (int c = 0; c < nh; ++c) {
    const long long R = c < A.C ? s_R[c] : LLONG_MAX;
    long long m = LLONG_MIN;
    for (int t = tid; t < Dh; t += 256) {
      const long long u = uget(c, t);
      m = max(m, u);
      if (R != LLONG_MAX && u > R) ex += u - R;
    }
    for (int o = 16; o > 0; o >>= 1) m = max(m, (long long)__shfl_xor_sync(0xffffffffu, m, o));
    if (lane == 0) s_wm[c][wid] = m;
  }
  for (int o = 16; o > 0; o >>= 1) ex += __shfl_xor_sync(0xffffffffu, ex, o);
  if (lane == 0) s_wx[wid] = ex;
  __syncthreads();
  if (tid < 3) {
    s_f3[tid] = (float)((double)(long long)s_fw[tid] * kInvFix);
    A.fwdtot[3 * b + tid] = 0ull;
  }
  if (tid < nh) {
    long long m = LLONG_MIN;
    for (int w = 0; w < 8; ++w) m = max(m, s_wm[tid][w]);
    s_m[tid] = m;
  }
  if (tid == 32) {
    long long e = 0;
    for (int w = 0; w < 8; ++w) e += s_wx[w];
    s_ex = e;
  }
  __syncthreads();
  for (int c = 0; c < nh; ++c) {
    const long long m = s_m[c];
    float sacc = 0.f;
    for (int t = tid; t < Dh; t += 256) sacc += soft_exp(uget(c, t) - m, A.tau);
    sacc = warp_sum(sacc);
    if (lane == 0) s_wsum[c][wid] = sacc;
  }
  __syncthreads();
  if (tid < nh) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += s_wsum[tid][w];
    s_s[tid] = t;
  }
  __syncthreads();
  const float vdep = s_f3[0], lcom = s_f3[1], vrec = s_f3[2];
  ex = s_ex;

  const bool on_dep = A.terms & (GAUS_DEP | GAUS_DEP_CF), on_com = A.terms & GAUS_COM;
  const bool on_robj = A.terms & GAUS_RES_OBJ, on_rv = A.terms & GAUS_RES_VIOL;
  const bool on_rec = A.terms & GAUS_REC;
  const float *lam = s_lam;
  const double vres = (double)ex * kInvFix;
  const float c_res = on_rv ? (float)((double)lam[GAUS_K_RES] + (double)A.rho * vres) : 0.f;
  if (tid == 0) {
    double lse_sum = 0.0;
    for (int c = 0; c < A.C; ++c) lse_sum += (double)s_m[c] * kInvFix + (double)A.tau * (double)logf(s_s[c]);
    const double reg_lse = A.Ureg ? (double)s_m[A.C] * kInvFix + (double)A.tau * (double)logf(s_s[A.C]) : 0.0;
    double L = 0.0;
    if (on_robj) L += (double)A.w_res * lse_sum;
    if (on_com) L += (double)A.alpha * (double)lcom;
    if (A.Ureg) L += (double)A.w_mem * reg_lse;
    const double Vk[3] = {on_dep ? (double)vdep : 0.0, on_rv ? vres : 0.0, on_rec ? (double)vrec : 0.0};
    const bool act[3] = {on_dep, on_rv, on_rec};
    for (int k = 0; k < 3; ++k)
      if (act[k]) L += (double)lam[k] * Vk[k] + 0.5 * (double)A.rho * Vk[k] * Vk[k];
    float *T = A.terms_out + (size_t)b * GAUS_NT;
    T[GAUS_T_RES] = on_robj ? (float)lse_sum : 0.f;
    T[GAUS_T_COM] = on_com ? lcom : 0.f;
    T[GAUS_T_REG] = A.Ureg ? (float)reg_lse : 0.f;
    T[GAUS_T_VDEP] = (float)Vk[0];
    T[GAUS_T_VRES] = (float)Vk[1];
    T[GAUS_T_VREC] = (float)Vk[2];
    A.loss[b] = (float)L;
    A.coef[b * 4 + 0] = on_dep ? (float)((double)lam[GAUS_K_DEP] + (double)A.rho * Vk[0]) : 0.f;
    A.coef[b * 4 + 1] = on_rec ? (float)((double)lam[GAUS_K_REC] + (double)A.rho * Vk[2]) : 0.f;
    A.thr[b] = threshold_of(s_ws[0], s_ws[1]);
    A.wstat[2 * b] = 0ull;
    A.wstat[2 * b + 1] = 0ull;
    const int bad = s_bad;
    if (A.status) A.status[b] = bad ? GAUS_ENONFINITE : GAUS_OK;
    A.nonfinite[b] = 0;
    if (A.update_lambda) {
      float *lw = A.lambda + (size_t)b * GAUS_K;
      for (int k = 0; k < 3; ++k)
        if (act[k]) lw[k] = (float)((double)lam[k] + (double)A.rho * Vk[k]);
    }
    if (A.step) {
      const int st = s_step + 1;
      A.step[b] = st;
      // Adam bias corrections of this step (torch.optim.Adam): 1 / (1 - beta1^t)
      // and 1 / sqrt(1 - beta2^t)
      A.coef[b * 4 + 2] = 1.0f / (1.0f - powf(A.beta1, (float)st));
      A.coef[b * 4 + 3] = 1.0f / sqrtf(1.0f - powf(A.beta2, (float)st));
    }
  }
  // usage adjoint dL/dU_c(t) = w_res softmax_c(t) + c_res [U_c(t) > R_c], [class][bin][restart]
  for (int i = tid; i < A.C * Dh; i += 256) {
    const int c = i / Dh;
    const long long u = uget(c, i - c * Dh);
    float h = 0.f;
    if (on_robj) h += A.w_res * soft_exp(u - s_m[c], A.tau) / s_s[c];
    if (on_rv && s_R[c] != LLONG_MAX && u > s_R[c]) h += c_res;
    A.H[(size_t)i * A.B + b] = h;
  }
  if (A.Ureg)
    for (int t = tid; t < Dh; t += 256)
      A.Hreg[(size_t)b * Dh + t] = A.w_mem * soft_exp(uget(A.C, t) - s_m[A.C], A.tau) / s_s[A.C];
  (void)kInvFixF;
}
#endif  // GAUS_FAMILY_KERNELS_ONLY

// Gradient and Adam step (Sec. 3.3).  Warp-item = 32 / RB internal nodes x one
// restart group (lanes are restarts), taken grid-stride.  Per (node, restart):
// the usage adjoint over the own window, dL/dC_v(t) = w_v (H(t) - H(t+1)); the
// node's edge partials from the edge pass in a fixed order (out-edges, in-edges,
// back edges out and in, all contiguous per node); the combined gradient
//   dL/dmu = -(c_dep Ad + Ao + c_rec Ar + Ah) / sigma, same with B.. for sigma,
// and, in Adam mode, the Adam step with the per-restart bias corrections.
// Windows longer than the restart's threshold are done by the whole warp.
template <int kFam, bool kAdam, bool kHist>
__global__ void __launch_bounds__(kUpdThreads) k_update(const UpdArgs A) {
  constexpr unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31, RB = A.RB, npw = 32 / RB, Dh = A.Dh;
  const int r = lane % RB;
  const int nwi = (A.V + npw - 1) / npw * A.G;
  const int wstride = gridDim.x * (kUpdThreads / 32);
  const size_t nP = (size_t)A.nEt * A.B;  // consumer-side slots follow the producer side
  for (int wi = blockIdx.x * (kUpdThreads / 32) + (threadIdx.x >> 5); wi < nwi; wi += wstride) {
    const int g = wi % A.G, vi = (wi / A.G) * npw + lane / RB, b = g * RB + r;
    const bool valid = b < A.B && vi < A.V;
    const int vcl = valid ? vi : 0, bs = valid ? b : 0;
    const int vc = A.perm[vcl];
    const size_t ci = (size_t)vc * A.B + bs, gi = (size_t)vcl * A.B + bs;
    const float mu = valid ? A.mu[ci] : 0.f, sg = valid ? A.sg[ci] : 1.f;
    const bool ok = valid && usable(mu, sg);
    float Ah = 0.f, Bh = 0.f;
    if (kHist) {
      const float *Hc = A.H + (size_t)A.cls[vcl] * Dh * A.B;  // [bin][restart]
      const float inv_s = ok ? 1.0f / sg : 1.0f, wv = A.w[vcl];
      int a = 0, bw = -1;
      if (ok) window(mu, sg, A.k_win, A.D, a, bw);
      const int nfull = bw - a + 1;
      const bool is_long = ok && nfull > A.thr[bs];
      const int n = is_long ? 0 : nfull;
      const int nmax = __reduce_max_sync(FULL, n);
      for (int j = 0; j < nmax; ++j) {
        if (j < n) {
          const int t = a + j;
          const float z = ((float)t + 0.5f - mu) * inv_s;
          const float f = Fam<kFam>::pdf(z);
          const float gh = wv * (Hc[(size_t)fold_bin(t, A.II) * A.B + b] - Hc[(size_t)fold_bin(t + 1, A.II) * A.B + b]);
          Ah += gh * f;
          Bh += gh * z * f;
        }
      }
      __syncwarp();
      unsigned longmask = __ballot_sync(FULL, is_long);
      while (longmask) {
        const int src = __ffs(longmask) - 1;
        longmask &= longmask - 1;
        const int l_a = __shfl_sync(FULL, a, src), l_n = __shfl_sync(FULL, nfull, src);
        const int l_b = __shfl_sync(FULL, b, src);
        const float l_mu = __shfl_sync(FULL, mu, src), l_inv = __shfl_sync(FULL, inv_s, src);
        const float l_w = __shfl_sync(FULL, wv, src);
        const float *l_H = A.H + (size_t)A.cls[__shfl_sync(FULL, vcl, src)] * Dh * A.B;
        float pa = 0.f, pb = 0.f;
        for (int base = 0; base < l_n; base += 32) {
          const int j = base + lane;
          if (j < l_n) {
            const int t = l_a + j;
            const float z = ((float)t + 0.5f - l_mu) * l_inv;
            const float f = Fam<kFam>::pdf(z);
            const float gh = l_w * (l_H[(size_t)fold_bin(t, A.II) * A.B + l_b] -
                                    l_H[(size_t)fold_bin(t + 1, A.II) * A.B + l_b]);
            pa += gh * f;
            pb += gh * z * f;
          }
        }
        pa = warp_sum(pa);
        pb = warp_sum(pb);
        if (lane == src) { Ah = pa; Bh = pb; }
      }
    }
    if (!valid) continue;
    // the node's edge partials in a fixed order: out-edges, in-edges, back edges
    float Ad = 0.f, Bd = 0.f, Ao = 0.f, Bo = 0.f, Ar = 0.f, Br = 0.f;
    if (ok) {
#pragma unroll 8
      for (int e = A.out_ptr[vi]; e < A.out_ptr[vi + 1]; ++e) {
        const float4 s = A.eslot4[(size_t)e * A.B + b];
        Ad += s.x; Bd += s.y; Ao += s.z; Bo += s.w;
      }
#pragma unroll 4
      for (int e = A.in_ptr[vi]; e < A.in_ptr[vi + 1]; ++e) {
        const float4 s = A.eslot4[nP + (size_t)e * A.B + b];
        Ad += s.x; Bd += s.y; Ao += s.z; Bo += s.w;
      }
      if (A.has_back) {
        for (int e = A.bout_ptr[vi]; e < A.bout_ptr[vi + 1]; ++e) {
          const float4 s = A.eslot4[(size_t)(A.E + e) * A.B + b];
          Ar += s.x; Br += s.y;
        }
        for (int e = A.bin_ptr[vi]; e < A.bin_ptr[vi + 1]; ++e) {
          const float4 s = A.eslot4[nP + (size_t)(A.E + e) * A.B + b];
          Ar += s.x; Br += s.y;
        }
      }
      if (A.gown) {
        const float2 s = A.gown[gi];
        Ao += s.x; Bo += s.y;
      }
    }
    const float c_dep = A.coef[b * 4 + 0], c_rec = A.coef[b * 4 + 1];
    float Asum = c_dep * Ad + Ao + c_rec * Ar + Ah;
    float Bsum = c_dep * Bd + Bo + c_rec * Br + Bh;
    if (A.eslot && ok)
      for (int e = A.in_ptr[vi]; e < A.in_ptr[vi + 1]; ++e) {
        const float2 sh = A.eslot[(size_t)A.in_eslot[e] * A.B + b];
        Asum += sh.x;
        Bsum += sh.y;
      }
    // dC/dmu = -phi/sigma, dC/dsigma = -z phi/sigma
    const float rs = ok ? __frcp_rn(sg) : 0.f;
    const float gm = -Asum * rs, gs = -Bsum * rs;
    if (!kAdam) {
      A.grad_mu[ci] = gm;
      A.grad_sg[ci] = gs;
    } else {
      const float inv_bc1 = A.coef[b * 4 + 2], rs_bc2 = A.coef[b * 4 + 3];
      float m1 = A.m_mu[ci], v1 = A.v_mu[ci], m2 = A.m_sg[ci], v2 = A.v_sg[ci];
      const float nmu = adam_update(mu, gm, m1, v1, A.lr, A.beta1, A.beta2, A.eps, inv_bc1, rs_bc2);
      const float nsg = adam_update(sg, gs, m2, v2, A.lr, A.beta1, A.beta2, A.eps, inv_bc1, rs_bc2);
      A.m_mu[ci] = m1; A.v_mu[ci] = v1; A.m_sg[ci] = m2; A.v_sg[ci] = v2;
      A.mu[ci] = nmu;
      A.sg[ci] = fmaxf(nsg, A.sigma_min);
    }
  }
}

}  // namespace gaus
