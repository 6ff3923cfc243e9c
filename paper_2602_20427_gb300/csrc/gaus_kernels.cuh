// gaus_kernels.cuh -- device code of one GauS iteration (Sec. 3.2-3.3, App. B).
//
// Work item: one (node v, restart b).  Threads of a warp are restarts of the same
// node (lanes = b), so every mu/sigma gather of a neighbour is one coalesced
// 128-byte load.  Each thread keeps its own window of CDF points
//   C_v(t) = Phi((t + 1/2 - mu_v) / sigma_v),  t in [a_v, b_v] = points within
//   window_k * sigma_v of mu_v, with C_v(t) = 0 below and 1 above (Eq. round and
// its open end bins), and evaluates each neighbour's CDF at the points it needs.
//
// k_fwd     : bin masses -> usage histogram (shared-memory int64 fixed point, one
//             class per block, no global atomics) and every edge term from both
//             endpoints (gathered through CSC as consumer and CSR as producer):
//             forward sums and the unscaled partial gradients.
// k_finalize: one block per restart -- usage per class, LogSumExp (Eq. max),
//             ReLU (Eq. relu), the augmented-Lagrangian coefficients (Sec. 3.3).
// k_update  : usage adjoint of the node's own window, the combined gradient and
//             (optionally) the Adam step.
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
  int V, B, D, II, Dh, C, RB, G, kc;
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
  long long *fwd;
  float *gpart;
  int32_t *nonfinite;
  const unsigned *win;  // (V, B) packed windows: a | (b + 1) << 16
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
  const long long *fwd;
  float *lambda;      // read; updated in place when update_lambda
  int update_lambda;
  int32_t *step;      // incremented when not NULL
  float beta1, beta2; // Adam, for the bias corrections written to coef[2], coef[3]
  float *H, *coef, *loss, *terms_out;
  int32_t *status, *nonfinite;
};

struct UpdArgs {
  const int32_t *in_ptr, *in_eslot;  // storage term: successor shares gathered per in-edge
  const float2 *eslot;               // NULL when the storage term is off
  float *mu, *sg;  // caller order; written when adam
  int V, B, D, II, Dh, C, RB, G;
  float k_win;
  const int32_t *perm;
  const unsigned *win;  // (V, B) packed windows of the state being updated
  const float *w;
  const int32_t *seg;
  const float *gpart;
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

// One (node, restart) item whose window is long, processed by the whole warp with
// lanes over its points (32 at a time).  Same terms and formulas as the per-lane
// path; the warp-reduced sums are returned in out[0..8] on every lane:
// Ad, Bd, Ao, Bo, Ar, Br, fdep, fcom, frec.
template <bool kDep, bool kCom, bool kRec>
__device__ void coop_item(const IterArgs &A, int vcl, int b, int r, int RB, float mu, float inv_s, int a, int bw,
                          float wv, unsigned *hlo, unsigned *hhi, float out[9]) {
  constexpr unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31, n = bw - a + 1;
  float Ad = 0.f, Bd = 0.f, Ao = 0.f, Bo = 0.f, Ar = 0.f, Br = 0.f, fdep = 0.f, fcom = 0.f, frec = 0.f;
  float z_carry = 0.f, q_carry = 0.f;
  for (int base = 0; base <= n; base += 32) {
    const int pidx = base + lane;
    const bool pt = pidx < n;
    const int t = a + pidx;
    const float z = ((float)t + 0.5f - mu) * inv_s;
    const float q = pt ? 0.5f * erfcf(fabsf(z) * kInvSqrt2) : 0.f;
    const float Cv = pt ? (z <= 0.f ? q : 1.0f - q) : 1.0f;
    const float f = pt ? kInvSqrt2Pi * expf(-0.5f * z * z) : 0.f;
    const float zf = z * f;
    float zp = __shfl_up_sync(FULL, z, 1), qp = __shfl_up_sync(FULL, q, 1);
    if (lane == 0) { zp = z_carry; qp = q_carry; }
    if (pidx <= n) hist_add(hlo, hhi, fold_bin(t, A.II) * RB + r, wv * bin_mass(pt, pidx == 0, z, q, zp, qp));
    z_carry = __shfl_sync(FULL, z, 31);
    q_carry = __shfl_sync(FULL, q, 31);
    if (kDep || kCom) {
      for (int e = A.in_ptr[vcl]; e < A.in_ptr[vcl + 1]; ++e) {  // own = consumer
        const int uc = A.in_src[e], L = A.in_lat[e];
        const float mu_u = A.mu[(size_t)uc * A.B + b], sg_u = A.sg[(size_t)uc * A.B + b];
        if (!usable(mu_u, sg_u)) continue;
        const float inv_u = 1.0f / sg_u;
        int au, bu;
        window(mu_u, sg_u, A.k_win, A.D, au, bu);
        if (pt) {
          const float c_hi = cdf_at(t + 1 - L, mu_u, inv_u, au, bu);
          const float p = c_hi - cdf_at(t - L, mu_u, inv_u, au, bu);
          if (kDep) { fdep += Cv * p; Ad += p * f; Bd += p * zf; }
          if (kCom) {
            const float cu = (L == 1) ? c_hi : cdf_at(t, mu_u, inv_u, au, bu);
            fcom += cu * (1.0f - Cv);
            Ao -= A.alpha * cu * f;
            Bo -= A.alpha * cu * zf;
          }
        }
        if (kDep && base == 0 && lane == 0) fdep += 1.0f - cdf_at(bw + 1 - L, mu_u, inv_u, au, bu);
      }
      const int L = A.lat[vcl];
      for (int e = A.out_ptr[vcl]; e < A.out_ptr[vcl + 1]; ++e) {  // own = producer
        const int wc = A.out_dst[e];
        const float mu_w = A.mu[(size_t)wc * A.B + b], sg_w = A.sg[(size_t)wc * A.B + b];
        if (!usable(mu_w, sg_w)) continue;
        const float inv_w = 1.0f / sg_w;
        int aw, bw2;
        window(mu_w, sg_w, A.k_win, A.D, aw, bw2);
        if (pt) {
          const float c_hi = cdf_at(t + L, mu_w, inv_w, aw, bw2);
          const float c_lo = cdf_at(t + L - 1, mu_w, inv_w, aw, bw2);
          if (kDep) { const float p = c_hi - c_lo; Ad -= p * f; Bd -= p * zf; }
          if (kCom) {
            const float cw = (L == 1) ? c_lo : cdf_at(t, mu_w, inv_w, aw, bw2);
            Ao += A.alpha * (1.0f - cw) * f;
            Bo += A.alpha * (1.0f - cw) * zf;
            if (t < aw) fcom += Cv;
          }
        }
        if (kCom && base == 0 && lane == 0) fcom += (float)max(0, aw - 1 - bw);
      }
    }
    if (kRec) {
      for (int e = A.bin_ptr[vcl]; e < A.bin_ptr[vcl + 1]; ++e) {  // own = consumer i
        const int jc = A.bin_src[e], L = A.bin_shift[e];
        const float mu_u = A.mu[(size_t)jc * A.B + b], sg_u = A.sg[(size_t)jc * A.B + b];
        if (!usable(mu_u, sg_u)) continue;
        const float inv_u = 1.0f / sg_u;
        int au, bu;
        window(mu_u, sg_u, A.k_win, A.D, au, bu);
        if (pt) {
          const float p = cdf_at(t + 1 - L, mu_u, inv_u, au, bu) - cdf_at(t - L, mu_u, inv_u, au, bu);
          frec += Cv * p; Ar += p * f; Br += p * zf;
        }
        if (base == 0 && lane == 0) frec += 1.0f - cdf_at(bw + 1 - L, mu_u, inv_u, au, bu);
      }
      for (int e = A.bout_ptr[vcl]; e < A.bout_ptr[vcl + 1]; ++e) {  // own = producer j
        const int ic = A.bout_dst[e], L = A.bout_shift[e];
        const float mu_w = A.mu[(size_t)ic * A.B + b], sg_w = A.sg[(size_t)ic * A.B + b];
        if (!usable(mu_w, sg_w)) continue;
        const float inv_w = 1.0f / sg_w;
        int aw, bw2;
        window(mu_w, sg_w, A.k_win, A.D, aw, bw2);
        if (pt) {
          const float p = cdf_at(t + L, mu_w, inv_w, aw, bw2) - cdf_at(t + L - 1, mu_w, inv_w, aw, bw2);
          Ar -= p * f; Br -= p * zf;
        }
      }
    }
  }
  __syncwarp();
  out[0] = warp_sum(Ad); out[1] = warp_sum(Bd); out[2] = warp_sum(Ao); out[3] = warp_sum(Bo);
  out[4] = warp_sum(Ar); out[5] = warp_sum(Br);
  out[6] = warp_sum(fdep); out[7] = warp_sum(fcom); out[8] = warp_sum(frec);
}

template <bool kDep, bool kCom, bool kRec>
__global__ void __launch_bounds__(kFwdThreads) k_fwd(const IterArgs A) {
  // Shared memory: usage histogram as two u32 halves [bin][restart] (conflict-free
  // for any bins the lanes of a warp touch), then the own-window cache.
  extern __shared__ __align__(16) unsigned char smem[];
  constexpr int T = kFwdThreads;
  const int tid = threadIdx.x, RB = A.RB, Dh = A.Dh, kc = A.kc;
  unsigned *hlo = reinterpret_cast<unsigned *>(smem);
  unsigned *hhi = hlo + (size_t)Dh * RB;
  float *cC = reinterpret_cast<float *>(hhi + (size_t)Dh * RB);
  float *cF = cC + (size_t)kc * T;
  float *cZ = cF + (size_t)kc * T;
  __shared__ int s_lo, s_hi, s_next, s_wsum[32], s_wcnt[32];

  const int blk = blockIdx.x, segi = blk / A.G, g = blk % A.G;
  const int s0 = A.seg[3 * segi], s1 = A.seg[3 * segi + 1];
  for (int i = tid; i < 2 * RB * Dh; i += T) hlo[i] = 0u;
  if (tid == 0) { s_lo = INT_MAX; s_hi = INT_MIN; s_next = 0; }
  if (tid < 32) { s_wsum[tid] = 0; s_wcnt[tid] = 0; }
  __syncthreads();

  const int r = tid % RB, b = g * RB + r, rows = T / RB;
  const bool bok = b < A.B;
  // long-window threshold of this restart in this segment
  const int long_min = min(kc, max(8, 3 * seg_mean_window(A.win, A.perm, s0, s1, b, bok, A.B, tid, RB, rows,
                                                           s_wsum, s_wcnt) + 8));
  const size_t VB = (size_t)A.V * A.B;
  constexpr unsigned FULL = 0xffffffffu;
  long long xdep = 0, xcom = 0, xrec = 0;  // forward sums, exact (order-free) fixed point
  int lo = INT_MAX, hi = INT_MIN;
  // Control flow is kept warp-uniform: each warp claims the next group of
  // 32 / RB nodes of the segment from a shared counter (so warps finish
  // together), and every loop runs to the warp's maximum trip count with a
  // per-lane predicate, so the warp never splits around the shared atomics.
  const int npw = 32 / RB;
  for (;;) {
    int base = 0;
    if ((tid & 31) == 0) base = atomicAdd(&s_next, npw);
    base = __shfl_sync(FULL, base, 0);
    if (base >= s1 - s0) break;
    const int vi = s0 + base + (tid & 31) / RB;
    float fdep = 0.f, fcom = 0.f, frec = 0.f;  // this item's forward sums
    bool valid = bok && vi < s1;
    const int vcl = valid ? vi : s0;
    const int vc = A.perm[vcl];
    const size_t gi = (size_t)vcl * A.B + (bok ? b : 0);
    const float mu = valid ? A.mu[(size_t)vc * A.B + b] : 0.f;
    const float sg = valid ? A.sg[(size_t)vc * A.B + b] : 1.f;
    if (valid && !usable(mu, sg)) {
      A.nonfinite[b] = 1;
      for (int k = 0; k < 6; ++k) A.gpart[k * VB + gi] = 0.f;
      valid = false;
    }
    const float inv_s = valid ? 1.0f / sg : 1.0f, wv = A.w[vcl];
    int a = 0, bw = -2;
    if (valid) window(mu, sg, A.k_win, A.D, a, bw);
    const int nfull = bw - a + 1;                  // points; -1 for an idle lane
    // Windows much longer than this restart's typical one in the segment (or
    // than the cache) go to the cooperative path after this per-lane pass.
    const bool is_long = valid && nfull > long_min;
    const int n = is_long ? -1 : nfull;            // per-lane points
    const bool vs = valid && !is_long;
    const int nmax = __reduce_max_sync(FULL, n);

    // ---- own points: cache C, phi, z*phi; bin masses into the usage histogram ----
    // P(d) for d in [a, b+1] from Q(|z|) = Phi(-|z|) so that both tails keep
    // relative accuracy: C = Q when z <= 0, 1 - Q otherwise.  Each mass enters
    // the histogram as round(w P 2^32), split into 16-bit halves (exact sums).
    float zp = 0.f, qp = 0.f;
    for (int j = 0; j <= nmax; ++j) {
      const bool pt = j < n;                       // point a+j exists
      const float zc = ((float)(a + j) + 0.5f - mu) * inv_s;
      const float qc = pt ? 0.5f * erfcf(fabsf(zc) * kInvSqrt2) : 0.f;
      if (pt && j < kc) {
        const float f = kInvSqrt2Pi * expf(-0.5f * zc * zc);
        cC[j * T + tid] = zc <= 0.f ? qc : 1.0f - qc;
        cF[j * T + tid] = f;
        cZ[j * T + tid] = zc * f;
      }
      if (j <= n) hist_add(hlo, hhi, fold_bin(a + j, A.II) * RB + r, wv * bin_mass(pt, j == 0, zc, qc, zp, qp));
      zp = zc;
      qp = qc;
    }
    __syncwarp();
    if (valid) {
      lo = min(lo, a);
      hi = max(hi, bw + 1);
    }

    // own point j: C, phi, z*phi (recomputed beyond the cache)
    auto own = [&](int j, float &C, float &f, float &zf) {
      if (j < kc) {
        C = cC[j * T + tid];
        f = cF[j * T + tid];
        zf = cZ[j * T + tid];
      } else {
        const float z = ((float)(a + j) + 0.5f - mu) * inv_s;
        const float q = 0.5f * erfcf(fabsf(z) * kInvSqrt2);
        C = z <= 0.f ? q : 1.0f - q;
        f = kInvSqrt2Pi * expf(-0.5f * z * z);
        zf = z * f;
      }
    };

    float Ad = 0.f, Bd = 0.f, Ao = 0.f, Bo = 0.f, Ar = 0.f, Br = 0.f;
    // ---- edges: every edge term is a dot product of the own window with the
    // neighbour's CDF shifted by a latency; only the own points where the
    // neighbour's values vary (or, for communication, are a constant 1) are
    // visited, and the neighbour's mean and sigma are read only then. ----
    // in-edges u -> v (own = consumer), latency L = Lat(u):
    //   V_e = 1 - C_u(b_v + 1 - L) + sum_{t in own} C_v(t) P_u(t + 1 - L)
    //   dV_e/dC_v(t) = P_u(t + 1 - L);  L_com,e part = sum_{t in own} C_u(t) (1 - C_v(t))
    //   dL_com,e/dC_v(t) = -C_u(t)
    if (kDep || kCom) {
      const int e0 = A.in_ptr[vcl], deg = vs ? A.in_ptr[vcl + 1] - e0 : 0;
      const int dmax = __reduce_max_sync(FULL, deg);
      for (int q = 0; q < dmax; ++q) {
        const bool eon = q < deg;
        const int uc = eon ? A.in_src[e0 + q] : 0, L = eon ? A.in_lat[e0 + q] : 0;
        const unsigned wm = eon ? A.win[(size_t)uc * A.B + b] : 0u;
        const int au = (int)(wm & 0xFFFFu), bu = (int)(wm >> 16) - 1;
        // P_u(t+1-L) != 0 for t in [au+L-1, bu+L]; C_u(t) != 0 for t >= au
        const int jlo = max(0, au + min(kDep ? L - 1 : 0, 0) - a);
        const int jhi = kCom ? n - 1 : min(n - 1, bu + L - a);
        const int x0 = bw + 1 - L;
        const int cnt = eon && jhi >= jlo ? jhi - jlo + 1 : 0;
        const bool need = cnt > 0 || (kDep && eon && x0 >= au && x0 <= bu);
        const float mu_u = need ? A.mu[(size_t)uc * A.B + b] : 0.f;
        const float inv_u = need ? 1.0f / A.sg[(size_t)uc * A.B + b] : 1.f;
        const int cmax = __reduce_max_sync(FULL, cnt);
        float c_lo = cnt ? cdf_at(a + jlo - L, mu_u, inv_u, au, bu) : 0.f;
        for (int k2 = 0; k2 < cmax; ++k2) {
          if (k2 < cnt) {
            const int j = jlo + k2, t = a + j;
            const float c_hi = cdf_at(t + 1 - L, mu_u, inv_u, au, bu);
            const float p = c_hi - c_lo;
            float Cv, f, zf;
            own(j, Cv, f, zf);
            if (kDep) {
              fdep += Cv * p;
              Ad += p * f;
              Bd += p * zf;
            }
            if (kCom) {
              const float cu = (L == 1) ? c_hi : cdf_at(t, mu_u, inv_u, au, bu);
              fcom += cu * (1.0f - Cv);
              Ao -= A.alpha * cu * f;
              Bo -= A.alpha * cu * zf;
            }
            c_lo = c_hi;
          }
        }
        __syncwarp();
        if (kDep && eon) fdep += 1.0f - cdf_at(x0, mu_u, inv_u, au, bu);
      }
    }
    // out-edges v -> w (own = producer), latency L = Lat(v):
    //   dV_e/dC_v(x) = -P_w(x + L), nonzero for x in [aw-L, bw+1-L]
    //   dL_com,e/dC_v(x) = 1 - C_w(x), nonzero for x <= bw
    //   L_com,e part = sum_{x in own, x < a_w} C_v(x) + max(0, a_w - 1 - b_v)
    if (kDep || kCom) {
      const int L = A.lat[vcl];
      const int e0 = A.out_ptr[vcl], deg = vs ? A.out_ptr[vcl + 1] - e0 : 0;
      const int dmax = __reduce_max_sync(FULL, deg);
      for (int q = 0; q < dmax; ++q) {
        const bool eon = q < deg;
        const int wc = eon ? A.out_dst[e0 + q] : 0;
        const unsigned wm = eon ? A.win[(size_t)wc * A.B + b] : 0u;
        const int aw = (int)(wm & 0xFFFFu), bw2 = (int)(wm >> 16) - 1;
        int jlo = max(0, aw - L - a), jhi = min(n - 1, bw2 + 1 - L - a);
        if (kCom) {
          jlo = 0;
          jhi = max(jhi, min(n - 1, bw2 - a));
        }
        const int cnt = eon && jhi >= jlo ? jhi - jlo + 1 : 0;
        const float mu_w = cnt ? A.mu[(size_t)wc * A.B + b] : 0.f;
        const float inv_w = cnt ? 1.0f / A.sg[(size_t)wc * A.B + b] : 1.f;
        const int cmax = __reduce_max_sync(FULL, cnt);
        float c_lo = cnt ? cdf_at(a + jlo + L - 1, mu_w, inv_w, aw, bw2) : 0.f;
        for (int k2 = 0; k2 < cmax; ++k2) {
          if (k2 < cnt) {
            const int j = jlo + k2, x = a + j;
            const float c_hi = cdf_at(x + L, mu_w, inv_w, aw, bw2);
            float Cv, f, zf;
            own(j, Cv, f, zf);
            if (kDep) {
              const float p = c_hi - c_lo;
              Ad -= p * f;
              Bd -= p * zf;
            }
            if (kCom) {
              const float cw = (L == 1) ? c_lo : cdf_at(x, mu_w, inv_w, aw, bw2);
              Ao += A.alpha * (1.0f - cw) * f;
              Bo += A.alpha * (1.0f - cw) * zf;
              if (x < aw) fcom += Cv;
            }
            c_lo = c_hi;
          }
        }
        __syncwarp();
        if (kCom && eon) fcom += (float)max(0, aw - 1 - bw);
      }
    }
    // back edges (App. B.3): a dependency with latency Lat(j) - k II
    if (kRec) {
      {  // own = consumer i
        const int e0 = A.bin_ptr[vcl], deg = vs ? A.bin_ptr[vcl + 1] - e0 : 0;
        const int dmax = __reduce_max_sync(FULL, deg);
        for (int q = 0; q < dmax; ++q) {
          const bool eon = q < deg;
          const int jc = eon ? A.bin_src[e0 + q] : 0, L = eon ? A.bin_shift[e0 + q] : 0;
          const unsigned wm = eon ? A.win[(size_t)jc * A.B + b] : 0u;
          const int au = (int)(wm & 0xFFFFu), bu = (int)(wm >> 16) - 1;
          const int jlo = max(0, au + L - 1 - a), jhi = min(n - 1, bu + L - a);
          const int x0 = bw + 1 - L;
          const int cnt = eon && jhi >= jlo ? jhi - jlo + 1 : 0;
          const bool need = cnt > 0 || (eon && x0 >= au && x0 <= bu);
          const float mu_u = need ? A.mu[(size_t)jc * A.B + b] : 0.f;
          const float inv_u = need ? 1.0f / A.sg[(size_t)jc * A.B + b] : 1.f;
          const int cmax = __reduce_max_sync(FULL, cnt);
          float c_lo = cnt ? cdf_at(a + jlo - L, mu_u, inv_u, au, bu) : 0.f;
          for (int k2 = 0; k2 < cmax; ++k2) {
            if (k2 < cnt) {
              const int j = jlo + k2;
              const float c_hi = cdf_at(a + j + 1 - L, mu_u, inv_u, au, bu);
              const float p = c_hi - c_lo;
              float Cv, f, zf;
              own(j, Cv, f, zf);
              frec += Cv * p;
              Ar += p * f;
              Br += p * zf;
              c_lo = c_hi;
            }
          }
          __syncwarp();
          if (eon) frec += 1.0f - cdf_at(x0, mu_u, inv_u, au, bu);
        }
      }
      {  // own = producer j
        const int e0 = A.bout_ptr[vcl], deg = vs ? A.bout_ptr[vcl + 1] - e0 : 0;
        const int dmax = __reduce_max_sync(FULL, deg);
        for (int q = 0; q < dmax; ++q) {
          const bool eon = q < deg;
          const int ic = eon ? A.bout_dst[e0 + q] : 0, L = eon ? A.bout_shift[e0 + q] : 0;
          const unsigned wm = eon ? A.win[(size_t)ic * A.B + b] : 0u;
          const int aw = (int)(wm & 0xFFFFu), bw2 = (int)(wm >> 16) - 1;
          const int jlo = max(0, aw - L - a), jhi = min(n - 1, bw2 + 1 - L - a);
          const int cnt = eon && jhi >= jlo ? jhi - jlo + 1 : 0;
          const float mu_w = cnt ? A.mu[(size_t)ic * A.B + b] : 0.f;
          const float inv_w = cnt ? 1.0f / A.sg[(size_t)ic * A.B + b] : 1.f;
          const int cmax = __reduce_max_sync(FULL, cnt);
          float c_lo = cnt ? cdf_at(a + jlo + L - 1, mu_w, inv_w, aw, bw2) : 0.f;
          for (int k2 = 0; k2 < cmax; ++k2) {
            if (k2 < cnt) {
              const int j = jlo + k2;
              const float c_hi = cdf_at(a + j + L, mu_w, inv_w, aw, bw2);
              const float p = c_hi - c_lo;
              float Cv, f, zf;
              own(j, Cv, f, zf);
              Ar -= p * f;
              Br -= p * zf;
              c_lo = c_hi;
            }
          }
          __syncwarp();
        }
      }
    }
    // ---- cooperative pass over the long windows of this warp ----
    unsigned longmask = __ballot_sync(FULL, is_long);
    while (longmask) {
      const int src = __ffs(longmask) - 1;
      longmask &= longmask - 1;
      const int l_v = __shfl_sync(FULL, vcl, src), l_b = __shfl_sync(FULL, b, src);
      const int l_r = __shfl_sync(FULL, r, src), l_a = __shfl_sync(FULL, a, src);
      const int l_bw = __shfl_sync(FULL, bw, src);
      const float l_mu = __shfl_sync(FULL, mu, src), l_inv = __shfl_sync(FULL, inv_s, src);
      const float l_w = __shfl_sync(FULL, wv, src);
      float sums[9];
      coop_item<kDep, kCom, kRec>(A, l_v, l_b, l_r, RB, l_mu, l_inv, l_a, l_bw, l_w, hlo, hhi, sums);
      if ((threadIdx.x & 31) == src) {
        Ad = sums[0]; Bd = sums[1]; Ao = sums[2]; Bo = sums[3]; Ar = sums[4]; Br = sums[5];
        fdep += sums[6]; fcom += sums[7]; frec += sums[8];
      }
    }
    xdep += to_fix(fdep);
    xcom += to_fix(fcom);
    xrec += to_fix(frec);
    if (valid) {
      A.gpart[0 * VB + gi] = Ad;
      A.gpart[1 * VB + gi] = Bd;
      A.gpart[2 * VB + gi] = Ao;
      A.gpart[3 * VB + gi] = Bo;
      A.gpart[4 * VB + gi] = Ar;
      A.gpart[5 * VB + gi] = Br;
    }
  }

  // ---- per-restart forward sums of this block (fixed order), reusing the cache ----
  if (lo <= hi) {
    atomicMin(&s_lo, lo);
    atomicMax(&s_hi, hi);
  }
  __syncthreads();
  long long *red = reinterpret_cast<long long *>(cC);
  red[0 * T + tid] = xdep;
  red[1 * T + tid] = xcom;
  red[2 * T + tid] = xrec;
  __syncthreads();
  if (tid < RB) {
    long long acc[3] = {0, 0, 0};
    for (int row = 0; row < rows; ++row)
      for (int k = 0; k < 3; ++k) acc[k] += red[k * T + row * RB + tid];
    for (int k = 0; k < 3; ++k) A.fwd[((size_t)blk * RB + tid) * 3 + k] = acc[k];
  }
  // ---- histogram rows restricted to the folded span the block touched ----
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

// Usage per (restart, class, bin) from the partials of every block of the class:
// block = (group g, class c, bin d); threads = restarts x slices of the segment
// list (four independent loads in flight per thread); slices are combined in a
// fixed order (exact int64 sums, kept in 2^32 fixed point).
__global__ void __launch_bounds__(256) k_reduce(const RedArgs A) {
  __shared__ long long part[256];
  const int RB = A.RB, Dh = A.Dh, nsl = 256 / RB;
  int x = blockIdx.x;
  const int d = x % Dh; x /= Dh;
  const int c = x % A.C, g = x / A.C;
  const int r = threadIdx.x % RB, sl = threadIdx.x / RB, b = g * RB + r;
  const int s_end = A.cls_seg_ptr[c + 1];
  long long acc = 0;
  for (int s = A.cls_seg_ptr[c] + sl; s < s_end; s += 4 * nsl) {
    long long v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int ss = s + u * nsl;
      v[u] = 0;
      if (ss < s_end) {
        const int blk = ss * A.G + g;
        const int2 sp = A.hspan[blk];
        if (d >= sp.x && d <= sp.y) v[u] = A.hpart[((size_t)blk * Dh + d) * RB + r];
      }
    }
    acc += v[0] + v[1] + v[2] + v[3];
  }
  part[threadIdx.x] = acc;
  __syncthreads();
  if (sl == 0 && b < A.B) {
    long long tot = 0;
    for (int k = 0; k < nsl; ++k) tot += part[k * RB + r];
    A.U[((size_t)b * A.C + c) * Dh + d] = tot;
  }
}

// Window of every (node, restart): a | (b + 1) << 16 with the points [a, b] of
// window(); an unusable mean/sigma gets the empty window at the horizon start.
__global__ void k_windows(const float *mu, const float *sg, unsigned *win, size_t n, float k, int D) {
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    int a = 0, b = -1;
    const float m = mu[i], s = sg[i];
    if (usable(m, s)) window(m, s, k, D, a, b);
    win[i] = (unsigned)a | ((unsigned)(b + 1) << 16);
  }
}

// x * 2^-32 of a 2^32 fixed-point value as float, through two 32-bit halves
// (64-bit integer to floating-point conversions run at the FP64 rate).
__device__ __forceinline__ float fix_to_float(long long x) {
  const int hi = (int)(x >> 32);
  const unsigned lo = (unsigned)((unsigned long long)x & 0xffffffffull);
  return (float)hi + (float)lo * 2.3283064365386963e-10f;
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

// One block (256 threads) per restart.  Usage and storage stay exact 2^32 fixed
// point (max and ReLU excess in integers); the softmax runs in fp32 on exact
// differences from the max, and only thread 0 assembles the loss in fp64.
__global__ void __launch_bounds__(256) k_finalize(const FinArgs A) {
  extern __shared__ __align__(16) unsigned char smem_f[];
  long long *U = reinterpret_cast<long long *>(smem_f);  // (C + 1) * Dh
  __shared__ long long shl[8];
  __shared__ float shf[8];
  __shared__ long long s_m[kMaxClasses + 1], s_R[kMaxClasses];
  __shared__ float s_s[kMaxClasses + 1];
  const int b = blockIdx.x, g = b / A.RB, r = b % A.RB, tid = threadIdx.x, Dh = A.Dh;
  const float kInvFixF = 2.3283064365386963e-10f;

  for (int i = tid; i < A.C * Dh; i += 256) U[i] = A.Ug[(size_t)b * A.C * Dh + i];
  if (A.Ureg)
    for (int t = tid; t < Dh; t += 256) U[A.C * Dh + t] = A.Ureg[(size_t)b * Dh + t];
  if (tid < A.C) {
    const float R = A.limit[tid];
    // limits in fixed point; an infinite or huge limit never binds
    s_R[tid] = (isfinite(R) && R < 1.0e9f) ? (long long)R * 4294967296LL +
                                                   (long long)((R - floorf(R)) * 4294967296.0f)
                                           : LLONG_MAX;
  }
  __syncthreads();

  // forward sums of the edge terms over every block of this restart group
  long long f3[3] = {0, 0, 0};
  const int nseg = A.cls_seg_ptr[A.C];
  for (int s = tid; s < nseg; s += 256)
    for (int k = 0; k < 3; ++k) f3[k] += A.fwd[((size_t)(s * A.G + g) * A.RB + r) * 3 + k];
  const float vdep = (float)((double)block_sum_i64(f3[0], shl) * kInvFix);
  const float lcom = (float)((double)block_sum_i64(f3[1], shl) * kInvFix);
  const float vrec = (float)((double)block_sum_i64(f3[2], shl) * kInvFix);

  // ReLU excess over finite limits (Eq. relu), exact
  long long ex = 0;
  for (int i = tid; i < A.C * Dh; i += 256) {
    const long long R = s_R[i / Dh];
    if (R != LLONG_MAX && U[i] > R) ex += U[i] - R;
  }
  ex = block_sum_i64(ex, shl);

  // LogSumExp per class (Eq. max) and of the storage, max shifted out
  const int nh = A.C + (A.Ureg ? 1 : 0);
  for (int c = 0; c < nh; ++c) {
    long long m = LLONG_MIN;
    for (int t = tid; t < Dh; t += 256) m = max(m, U[c * Dh + t]);
    m = block_max_ll(m, shl);
    float sacc = 0.f;
    for (int t = tid; t < Dh; t += 256) sacc += expf(fix_to_float(U[c * Dh + t] - m) / A.tau);
    sacc = block_sum_f(sacc, shf);
    if (tid == 0) { s_m[c] = m; s_s[c] = sacc; }
  }
  __syncthreads();

  const bool on_dep = A.terms & GAUS_DEP, on_com = A.terms & GAUS_COM;
  const bool on_robj = A.terms & GAUS_RES_OBJ, on_rv = A.terms & GAUS_RES_VIOL;
  const bool on_rec = A.terms & GAUS_REC;
  const float *lam = A.lambda + (size_t)b * GAUS_K;
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
    const int bad = A.nonfinite[b];
    if (A.status) A.status[b] = bad ? GAUS_ENONFINITE : GAUS_OK;
    A.nonfinite[b] = 0;
    if (A.update_lambda) {
      float *lw = A.lambda + (size_t)b * GAUS_K;
      for (int k = 0; k < 3; ++k)
        if (act[k]) lw[k] = (float)((double)lw[k] + (double)A.rho * Vk[k]);
    }
    if (A.step) {
      const int st = A.step[b] + 1;
      A.step[b] = st;
      // Adam bias corrections of this step (torch.optim.Adam)
      A.coef[b * 4 + 2] = 1.0f - powf(A.beta1, (float)st);
      A.coef[b * 4 + 3] = 1.0f - powf(A.beta2, (float)st);
    }
  }
  // usage adjoint dL/dU_c(t) = w_res softmax_c(t) + c_res [U_c(t) > R_c], [class][bin][restart]
  for (int i = tid; i < A.C * Dh; i += 256) {
    const int c = i / Dh;
    float h = 0.f;
    if (on_robj) h += A.w_res * expf(fix_to_float(U[i] - s_m[c]) / A.tau) / s_s[c];
    if (on_rv && s_R[c] != LLONG_MAX && U[i] > s_R[c]) h += c_res;
    A.H[(size_t)i * A.B + b] = h;
  }
  if (A.Ureg)
    for (int t = tid; t < Dh; t += 256)
      A.Hreg[(size_t)b * Dh + t] = A.w_mem * expf(fix_to_float(U[A.C * Dh + t] - s_m[A.C]) / A.tau) / s_s[A.C];
  (void)kInvFixF;
}

template <bool kAdam, bool kHist>
__global__ void __launch_bounds__(kThreads) k_update(const UpdArgs A) {
  constexpr unsigned FULL = 0xffffffffu;
  const int tid = threadIdx.x, RB = A.RB, Dh = A.Dh;
  const int blk = blockIdx.x, segi = blk / A.G, g = blk % A.G;
  const int s0 = A.seg[3 * segi], s1 = A.seg[3 * segi + 1], c = A.seg[3 * segi + 2];
  const float *Hc = A.H + (size_t)c * Dh * A.B;  // usage adjoint of this class, [bin][restart]
  const int r = tid % RB, b = g * RB + r, rows = kThreads / RB;
  const bool bok = b < A.B;
  __shared__ int s_wsum[32], s_wcnt[32];
  int long_min = 0;
  if (kHist) {
    if (tid < 32) { s_wsum[tid] = 0; s_wcnt[tid] = 0; }
    __syncthreads();
    long_min = max(8, 2 * seg_mean_window(A.win, A.perm, s0, s1, b, bok, A.B, tid, RB, rows, s_wsum, s_wcnt) + 8);
  }
  const size_t VB = (size_t)A.V * A.B;
  const int bs = bok ? b : 0;
  const float c_dep = A.coef[bs * 4 + 0], c_rec = A.coef[bs * 4 + 1];
  const float bc1 = kAdam ? A.coef[bs * 4 + 2] : 1.f, bc2 = kAdam ? A.coef[bs * 4 + 3] : 1.f;
  const int n_items = (s1 - s0 + rows - 1) / rows;
  for (int it = 0; it < n_items; ++it) {
    const int vi = s0 + tid / RB + it * rows;
    const bool valid = bok && vi < s1;
    const int vcl = valid ? vi : s0;
    const int vc = A.perm[vcl];
    const size_t ci = (size_t)vc * A.B + bs, gi = (size_t)vcl * A.B + bs;
    const float mu = valid ? A.mu[ci] : 0.f, sg = valid ? A.sg[ci] : 1.f;
    const bool ok = valid && usable(mu, sg);
    float Ah = 0.f, Bh = 0.f;
    if (kHist) {
      // dL/dC_v(t) = w_v (H(t) - H(t+1)) for the own points (P = C(t) - C(t-1));
      // windows much longer than the warp's typical one are done by the whole warp
      const float inv_s = ok ? 1.0f / sg : 1.0f, wv = A.w[vcl];
      int a = 0, bw = -1;
      if (ok) window(mu, sg, A.k_win, A.D, a, bw);
      const int nfull = bw - a + 1;
      const bool is_long = ok && nfull > long_min;
      const int n = is_long ? 0 : nfull;
      const int nmax = __reduce_max_sync(FULL, n);
      for (int j = 0; j < nmax; ++j) {
        if (j < n) {
          const int t = a + j;
          const float z = ((float)t + 0.5f - mu) * inv_s;
          const float f = kInvSqrt2Pi * expf(-0.5f * z * z);
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
        float pa = 0.f, pb = 0.f;
        for (int base = 0; base < l_n; base += 32) {
          const int j = base + (threadIdx.x & 31);
          if (j < l_n) {
            const int t = l_a + j;
            const float z = ((float)t + 0.5f - l_mu) * l_inv;
            const float f = kInvSqrt2Pi * expf(-0.5f * z * z);
            const float gh = l_w * (Hc[(size_t)fold_bin(t, A.II) * A.B + l_b] -
                                    Hc[(size_t)fold_bin(t + 1, A.II) * A.B + l_b]);
            pa += gh * f;
            pb += gh * z * f;
          }
        }
        pa = warp_sum(pa);
        pb = warp_sum(pb);
        if ((threadIdx.x & 31) == src) { Ah = pa; Bh = pb; }
      }
    }
    if (!valid) continue;
    float Asum = c_dep * A.gpart[0 * VB + gi] + A.gpart[2 * VB + gi] + c_rec * A.gpart[4 * VB + gi] + Ah;
    float Bsum = c_dep * A.gpart[1 * VB + gi] + A.gpart[3 * VB + gi] + c_rec * A.gpart[5 * VB + gi] + Bh;
    if (A.eslot && ok)
      for (int e = A.in_ptr[vi]; e < A.in_ptr[vi + 1]; ++e) {
        const float2 sh = A.eslot[(size_t)A.in_eslot[e] * A.B + b];
        Asum += sh.x;
        Bsum += sh.y;
      }
    // dC/dmu = -phi/sigma, dC/dsigma = -z phi/sigma
    const float gm = ok ? -Asum / sg : 0.f, gs = ok ? -Bsum / sg : 0.f;
    if (!kAdam) {
      A.grad_mu[ci] = gm;
      A.grad_sg[ci] = gs;
    } else {
      const float m1 = A.beta1 * A.m_mu[ci] + (1.0f - A.beta1) * gm;
      const float v1 = A.beta2 * A.v_mu[ci] + (1.0f - A.beta2) * gm * gm;
      const float m2 = A.beta1 * A.m_sg[ci] + (1.0f - A.beta1) * gs;
      const float v2 = A.beta2 * A.v_sg[ci] + (1.0f - A.beta2) * gs * gs;
      A.m_mu[ci] = m1; A.v_mu[ci] = v1; A.m_sg[ci] = m2; A.v_sg[ci] = v2;
      const float nmu = mu - A.lr * (m1 / bc1) / (sqrtf(v1 / bc2) + A.eps);
      const float nsg = sg - A.lr * (m2 / bc1) / (sqrtf(v2 / bc2) + A.eps);
      A.mu[ci] = nmu;
      A.sg[ci] = fmaxf(nsg, A.sigma_min);
    }
  }
}

}  // namespace gaus
