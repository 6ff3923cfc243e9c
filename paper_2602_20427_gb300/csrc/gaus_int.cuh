// gaus_int.cuh -- integer kernels: rounding (Sec. 3.3 Sampling), legalization
// (App. A, Alg. 1 and Alg. 2) and the discrete verifier (Sec. 2.1).  Bit-exact
// by construction: integer arithmetic only, and both legalizations compute a
// result that does not depend on the order of their updates.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "gaus_device.cuh"
#include "gaus_internal.h"

namespace gaus {

struct LegArgs {
  const float *mu;
  int32_t *s, *status;
  int V, B, D, II, nlvl;
  const int32_t *lvl_ptr, *lvl_nodes;
  const int32_t *pred_ptr, *pred_src, *lat;
  const int32_t *back_ptr, *back_src, *back_shift;
  const int32_t *asap, *alap;
  // predecessors of the node at each level-order position q: producer, Lat(producer)
  const int32_t *lq_ptr, *lq_src, *lq_lat;
};

// s = floor(mu + 1/2), evaluated exactly in double for every fp32 mu.
__device__ __forceinline__ int round_half_up(float m, bool &bad) {
  if (!isfinite(m)) { bad = true; return 0; }
  double x = floor((double)m + 0.5);
  x = fmin(fmax(x, -1073741824.0), 1073741824.0);
  return (int)x;
}

__global__ void k_round(const float *mu, int32_t *s, size_t n) {
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    bool bad = false;
    s[i] = round_half_up(mu[i], bad);
  }
}

// Block = 32 restarts (lanes) x 8 node rows.  Alg. 1: clamp to [ASAP, ALAP], then
// one forward pass level by level: s_v <- max(s_v, max_u s_u + Lat(u)).  The
// result is the least legal schedule above the clamped input, whatever the
// order inside a level, so it equals the sequential algorithm bit for bit.
__global__ void __launch_bounds__(256) k_legalize_regular(const LegArgs A) {
  const int lane = threadIdx.x & 31, row = threadIdx.x >> 5;
  const int b = blockIdx.x * 32 + lane;
  __shared__ int bad_lane[32];
  if (row == 0) bad_lane[lane] = 0;
  __syncthreads();
  const bool bok = b < A.B;
  if (bok)
    for (int v = row; v < A.V; v += 8) {
      bool bad = false;
      int x = round_half_up(A.mu[(size_t)v * A.B + b], bad);
      if (bad) bad_lane[lane] = 1;
      x = max(x, A.asap[v]);
      x = min(x, A.alap[v]);
      A.s[(size_t)v * A.B + b] = x;
    }
  __syncthreads();
  for (int l = 1; l < A.nlvl; ++l) {
    if (bok)
      for (int q = A.lvl_ptr[l] + row; q < A.lvl_ptr[l + 1]; q += 8) {
        const int v = A.lvl_nodes[q];
        int x = A.s[(size_t)v * A.B + b];
        for (int e = A.pred_ptr[v]; e < A.pred_ptr[v + 1]; ++e) {
          const int u = A.pred_src[e];
          x = max(x, A.s[(size_t)u * A.B + b] + A.lat[u]);
        }
        A.s[(size_t)v * A.B + b] = x;
      }
    __syncthreads();
  }
  if (row == 0 && bok) A.status[b] = bad_lane[lane] ? GAUS_ENONFINITE : GAUS_OK;
}

// Alg. 1 with one restart per block and its whole schedule in shared memory
// (4 |V| bytes): the same clamp and level-by-level forward pass, each level's
// nodes in parallel, predecessors read from the level-ordered lists.  Same
// fixed point, so the same result bit for bit.
__global__ void __launch_bounds__(512) k_legalize_regular_smem(const LegArgs A) {
  extern __shared__ int s_sched[];  // V, caller order
  __shared__ int bad;
  const int b = blockIdx.x, tid = threadIdx.x, nt = blockDim.x;
  if (tid == 0) bad = 0;
  __syncthreads();
  for (int v = tid; v < A.V; v += nt) {
    bool bd = false;
    int x = round_half_up(A.mu[(size_t)v * A.B + b], bd);
    if (bd) bad = 1;
    x = max(x, A.asap[v]);
    x = min(x, A.alap[v]);
    s_sched[v] = x;
  }
  __syncthreads();
  for (int l = 1; l < A.nlvl; ++l) {
    const int q1 = A.lvl_ptr[l + 1];
    for (int q = A.lvl_ptr[l] + tid; q < q1; q += nt) {
      const int v = A.lvl_nodes[q], e1 = A.lq_ptr[q + 1];
      int x = s_sched[v];
      for (int e = A.lq_ptr[q]; e < e1; ++e) x = max(x, s_sched[A.lq_src[e]] + A.lq_lat[e]);
      s_sched[v] = x;
    }
    __syncthreads();
  }
  for (int v = tid; v < A.V; v += nt) A.s[(size_t)v * A.B + b] = s_sched[v];
  if (tid == 0) A.status[b] = bad ? GAUS_ENONFINITE : GAUS_OK;
}

// Alg. 2: sweeps in topological (level) order of
//   s_v <- max(s_v, 0, max_u s_u + Lat(u), max_{(j -> v, k)} s_j + Lat(j) - k II)
// until a sweep changes nothing, at most |V| sweeps.  The updates only raise
// values and the iteration is bounded by the least fixed point above the
// rounded input, which it reaches within |V| sweeps whenever the recurrences are
// feasible, so the converged result is order independent.
__global__ void __launch_bounds__(256) k_legalize_modulo(const LegArgs A) {
  const int lane = threadIdx.x & 31, row = threadIdx.x >> 5;
  const int b = blockIdx.x * 32 + lane;
  __shared__ int bad_lane[32], changed[32], done[32];
  __shared__ int any_changed;
  if (row == 0) { bad_lane[lane] = 0; done[lane] = 0; }
  __syncthreads();
  const bool bok = b < A.B;
  if (bok)
    for (int v = row; v < A.V; v += 8) {
      bool bad = false;
      const int x = round_half_up(A.mu[(size_t)v * A.B + b], bad);
      if (bad) bad_lane[lane] = 1;
      A.s[(size_t)v * A.B + b] = x;
    }
  __syncthreads();
  for (int sweep = 0; sweep < A.V; ++sweep) {
    if (row == 0) changed[lane] = 0;
    if (threadIdx.x == 0) any_changed = 0;
    __syncthreads();
    for (int l = 0; l < A.nlvl; ++l) {
      if (bok)
        for (int q = A.lvl_ptr[l] + row; q < A.lvl_ptr[l + 1]; q += 8) {
          const int v = A.lvl_nodes[q];
          int t = 0;
          for (int e = A.pred_ptr[v]; e < A.pred_ptr[v + 1]; ++e) {
            const int u = A.pred_src[e];
            t = max(t, A.s[(size_t)u * A.B + b] + A.lat[u]);
          }
          for (int e = A.back_ptr[v]; e < A.back_ptr[v + 1]; ++e)
            t = max(t, A.s[(size_t)A.back_src[e] * A.B + b] + A.back_shift[e]);
          if (t > A.s[(size_t)v * A.B + b]) {
            A.s[(size_t)v * A.B + b] = t;
            changed[lane] = 1;
          }
        }
      __syncthreads();
    }
    if (row == 0 && bok) {
      if (!changed[lane]) done[lane] = 1;
      else atomicOr(&any_changed, 1);
    }
    __syncthreads();
    if (!any_changed) break;
  }
  if (row == 0 && bok)
    A.status[b] = bad_lane[lane] ? GAUS_ENONFINITE : (done[lane] ? GAUS_OK : GAUS_ENOTCONV);
}

struct VerArgs {
  const int32_t *s;
  gaus_report *rep;
  int V, E, NB, B, C, D, II, Dh;
  int RB, G;  // restarts per warp row, restart groups (pass 1)
  const int32_t *e_src, *e_dst, *lat, *cls, *dem, *bits;
  const int32_t *b_src, *b_dst, *b_dist;
  const int32_t *succ_ptr, *succ_dst;
  const float *limit;
  // zeroed before pass 1: per restart the counts (dep, com, lat, rec), the usage
  // counts (B, C, Dh) and the storage difference array (B, D + 1), exact int64
  unsigned long long *vacc, *vcnt, *vdiff;
  long long *vmm;  // (B, Dh) folded storage when pass 2 cannot stage it in shared memory
  int vsmem;       // 1: pass 2 stages its rows in shared memory
};

// Verifier pass 1 (Sec. 2.1 definitions; L_com of App. B.1): items are the edges,
// the nodes and the back edges; lanes are restarts (32 / RB items per warp, rows
// grid-stride over the blocks of the restart group), so every read of a schedule
// is coalesced over restarts.  Per (item, restart): the dependency / latency /
// recurrence violation and L_com counts in registers, then per restart in shared
// memory and once per block in global memory; usage counts and the storage
// difference array as global integer atomics (exact, order-free).
__global__ void __launch_bounds__(256) k_verify_scan(const VerArgs A) {
  __shared__ unsigned long long s_acc[4][32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, RB = A.RB, ipw = 32 / RB;
  const int g = blockIdx.x % A.G, nbg = gridDim.x / A.G;
  const int r = lane % RB, b = g * RB + r;
  const bool bok = b < A.B;
  if (tid < 4 * 32) s_acc[tid / 32][tid % 32] = 0ull;
  __syncthreads();
  const int nback = A.II > 0 ? A.NB : 0;
  const long long nitems = (long long)A.E + A.V + nback;
  const long long rows = (nitems + ipw - 1) / ipw;
  long long ndep = 0, lcom = 0, nlat = 0, nrec = 0;
  for (long long row = (long long)(blockIdx.x / A.G) * 8 + warp; row < rows; row += (long long)nbg * 8) {
    const long long it = row * ipw + lane / RB;
    if (!bok || it >= nitems) continue;
    if (it < A.E) {
      const int e = (int)it, u = A.e_src[e], v = A.e_dst[e];
      const int su = A.s[(size_t)u * A.B + b], sv = A.s[(size_t)v * A.B + b];
      if ((long long)sv < (long long)su + A.lat[u]) ++ndep;
      lcom += (long long)sv - su;
    } else if (it < (long long)A.E + A.V) {
      const int v = (int)(it - A.E);
      const int sv = A.s[(size_t)v * A.B + b];
      if (sv < 0 || (long long)sv + A.lat[v] > A.D) ++nlat;
      if (sv >= 0 && sv < A.D) {
        const int t = A.II > 0 ? sv % A.II : sv;
        atomicAdd(&A.vcnt[((size_t)b * A.C + A.cls[v]) * A.Dh + t], (unsigned long long)(long long)A.dem[v]);
      }
      // Mem: live on [s_v, max over successors of s_w) (leaves: until D), within [0, D)
      long long last = A.D;
      if (A.succ_ptr[v + 1] > A.succ_ptr[v]) {
        last = LLONG_MIN;
        for (int q = A.succ_ptr[v]; q < A.succ_ptr[v + 1]; ++q)
          last = max(last, (long long)A.s[(size_t)A.succ_dst[q] * A.B + b]);
      }
      const long long lo = max((long long)sv, 0LL), hi = min(last, (long long)A.D);
      if (lo < hi && A.bits[v] != 0) {
        unsigned long long *row_d = A.vdiff + (size_t)b * (A.D + 1);
        atomicAdd(&row_d[lo], (unsigned long long)(long long)A.bits[v]);
        atomicAdd(&row_d[hi], (unsigned long long)(-(long long)A.bits[v]));
      }
    } else {
      const int q = (int)(it - A.E - A.V), j = A.b_src[q], i = A.b_dst[q];
      if ((long long)A.s[(size_t)i * A.B + b] + (long long)A.b_dist[q] * A.II <
          (long long)A.s[(size_t)j * A.B + b] + A.lat[j])
        ++nrec;
    }
  }
  if (bok) {
    if (ndep) atomicAdd(&s_acc[0][r], (unsigned long long)ndep);
    if (lcom) atomicAdd(&s_acc[1][r], (unsigned long long)lcom);
    if (nlat) atomicAdd(&s_acc[2][r], (unsigned long long)nlat);
    if (nrec) atomicAdd(&s_acc[3][r], (unsigned long long)nrec);
  }
  __syncthreads();
  if (tid < 4 * RB) {
    const int k = tid / RB, rr = tid % RB, bb = g * RB + rr;
    if (bb < A.B && s_acc[k][rr]) atomicAdd(&A.vacc[(size_t)bb * 4 + k], s_acc[k][rr]);
  }
}

// Verifier pass 2: one block (256 threads) per restart assembles its report from
// pass 1's counts: per-class peaks and limit violations, the storage scan (Mem and
// its fold modulo II).
__global__ void __launch_bounds__(256) k_verify_fin(const VerArgs A) {
  extern __shared__ __align__(16) unsigned char smem_v[];
  const int b = blockIdx.x, tid = threadIdx.x;
  // the restart's rows staged in shared memory when they fit, else used in place
  // (the folded storage then in its global scratch row)
  long long *cnt = reinterpret_cast<long long *>(A.vcnt + (size_t)b * A.C * A.Dh);
  long long *diff = reinterpret_cast<long long *>(A.vdiff + (size_t)b * (A.D + 1));
  long long *mm = A.vmm + (size_t)b * A.Dh;
  if (A.vsmem) {
    long long *s_cnt = reinterpret_cast<long long *>(smem_v);
    long long *s_diff = s_cnt + (size_t)A.C * A.Dh;
    for (int i = tid; i < A.C * A.Dh; i += 256) s_cnt[i] = cnt[i];
    for (int i = tid; i <= A.D; i += 256) s_diff[i] = diff[i];
    cnt = s_cnt;
    diff = s_diff;
    mm = s_diff + (A.D + 1);
  }
  for (int i = tid; i < A.Dh; i += 256) mm[i] = 0;
  __syncthreads();
  if (tid == 0) {
    gaus_report R;
    R.n_dep_viol = (long long)A.vacc[(size_t)b * 4 + 0];
    R.L_com = (long long)A.vacc[(size_t)b * 4 + 1];
    R.n_lat_viol = (long long)A.vacc[(size_t)b * 4 + 2];
    R.n_rec_viol = (long long)A.vacc[(size_t)b * 4 + 3];
    R.n_res_viol = 0;
    R.L_res = 0;
    for (int c = 0; c < 16; ++c) R.peak[c] = 0;
    for (int c = 0; c < A.C; ++c) {
      long long pk = 0;
      const float lim = A.limit[c];
      for (int t = 0; t < A.Dh; ++t) {
        const long long x = cnt[c * A.Dh + t];
        pk = max(pk, x);
        if (isfinite(lim) && (double)x > (double)lim) R.n_res_viol++;
      }
      R.peak[c] = pk;
      R.L_res += pk;
    }
    long long run = 0, lmem = 0;
    for (int d = 0; d < A.D; ++d) {
      run += diff[d];
      lmem = max(lmem, run);
      mm[A.II > 0 ? d % A.II : d] += run;
    }
    long long lmm = 0;
    for (int t = 0; t < A.Dh; ++t) lmm = max(lmm, mm[t]);
    R.L_mem = lmem;
    R.L_mmem = lmm;
    R.feasible = (R.n_dep_viol == 0 && R.n_lat_viol == 0 && R.n_rec_viol == 0);
    R.res_ok = R.n_res_viol == 0;
    A.rep[b] = R;
  }
}

// Elementwise Adam on (V, B) arrays (gaus_adam_step), then sigma clamp.
__global__ void k_adam(float *mu, float *sg, const float *gmu, const float *gsg, float *m1, float *v1,
                       float *m2, float *v2, size_t n, int step, float lr, float beta1, float beta2,
                       float eps, float sigma_min) {
  const float inv_bc1 = 1.0f / (1.0f - powf(beta1, (float)step));
  const float rs_bc2 = 1.0f / sqrtf(1.0f - powf(beta2, (float)step));
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    float a1 = m1[i], b1 = v1[i], a2 = m2[i], b2 = v2[i];
    const float nmu = adam_update(mu[i], gmu[i], a1, b1, lr, beta1, beta2, eps, inv_bc1, rs_bc2);
    const float nsg = adam_update(sg[i], gsg[i], a2, b2, lr, beta1, beta2, eps, inv_bc1, rs_bc2);
    m1[i] = a1; v1[i] = b1; m2[i] = a2; v2[i] = b2;
    mu[i] = nmu;
    sg[i] = fmaxf(nsg, sigma_min);
  }
}

// lambda[b, k] += rho * V_k for the active constraints (Sec. 3.3).
__global__ void k_lambda(float *lambda, const float *terms, int B, unsigned on, float rho) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const float *T = terms + (size_t)b * GAUS_NT;
  if (on & (GAUS_DEP | GAUS_DEP_CF)) lambda[b * GAUS_K + GAUS_K_DEP] += rho * T[GAUS_T_VDEP];
  if (on & GAUS_RES_VIOL) lambda[b * GAUS_K + GAUS_K_RES] += rho * T[GAUS_T_VRES];
  if (on & GAUS_REC) lambda[b * GAUS_K + GAUS_K_REC] += rho * T[GAUS_T_VREC];
}

// ---- Outer loop of Alg. GauS ----

// Initialization (Sec. 3.3): sigma = max(kappa (ALAP - ASAP), sigma_min) per node
// (in double, then rounded to float), mu = mu0 or the midpoint (ASAP + ALAP) / 2;
// Adam moments zeroed.  Caller-order (V, B) arrays.
__global__ void k_init_state(const float *mu0, float *mu, float *sg, float *sg_init, float *m1, float *v1, float *m2,
                             float *v2, const int32_t *asap, const int32_t *alap, int V, int B, double kappa,
                             float sigma_min) {
  const size_t n = (size_t)V * B;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    const int v = (int)(i / B);
    const float s0 = fmaxf((float)(kappa * (double)(alap[v] - asap[v])), sigma_min);
    mu[i] = mu0 ? mu0[i] : 0.5f * (float)(asap[v] + alap[v]);
    sg[i] = s0;
    if (sg_init) sg_init[i] = s0;
    m1[i] = 0.f; v1[i] = 0.f; m2[i] = 0.f; v2[i] = 0.f;
  }
}

__global__ void k_init_restart(float *lambda, int32_t *step, int32_t *status, double *best_score,
                               int32_t *best_iter, int B, float lambda0) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  for (int k = 0; k < GAUS_K; ++k) lambda[b * GAUS_K + k] = lambda0;
  step[b] = 0;
  status[b] = GAUS_OK;
  if (best_score) best_score[b] = __longlong_as_double(0x7ff0000000000000ll);  // +inf
  if (best_iter) best_iter[b] = -1;
}

struct OuterArgs {
  const int32_t *sched, *leg_status;
  const gaus_report *rep;
  const float *mu;
  int V, B, II, iter;
  unsigned terms;
  double w_res, alpha, w_mem;
  double *best_score;
  int32_t *best_iter, *step, *moved, *decision;
};

// Outer-step decision of one restart (block b): the nodes legalization moved
// (sched != round(mu)), the candidate's score and whether it improves the best
// (App. A: the legalized schedule, or a reset to the prior best).  decision bits:
// 1 improved, 2 illegal (reset), 4 a best existed before this step, 8 legalization
// succeeded.
__global__ void __launch_bounds__(256) k_outer_decide(const OuterArgs A) {
  __shared__ int sh[8];
  const int b = blockIdx.x, tid = threadIdx.x;
  int moved = 0;
  for (int v = tid; v < A.V; v += 256) {
    bool bad = false;
    const int r = round_half_up(A.mu[(size_t)v * A.B + b], bad);
    if (bad || r != A.sched[(size_t)v * A.B + b]) ++moved;
  }
  for (int o = 16; o > 0; o >>= 1) moved += __shfl_xor_sync(0xffffffffu, moved, o);
  if ((tid & 31) == 0) sh[tid >> 5] = moved;
  __syncthreads();
  if (tid != 0) return;
  moved = 0;
  for (int w = 0; w < 8; ++w) moved += sh[w];
  const bool leg_ok = A.leg_status[b] == GAUS_OK;
  const gaus_report &R = A.rep[b];
  const bool cand = leg_ok && R.feasible && (!(A.terms & GAUS_RES_VIOL) || R.res_ok);
  double score = 0.0;
  if (A.terms & GAUS_RES_OBJ) score += A.w_res * (double)R.L_res;
  if (A.terms & GAUS_COM) score += A.alpha * (double)R.L_com;
  if (A.terms & GAUS_REG_OBJ) score += A.w_mem * (double)(A.II > 0 ? R.L_mmem : R.L_mem);
  const bool had_best = A.best_iter[b] >= 0;
  const bool improved = cand && score < A.best_score[b];
  const bool illegal = !leg_ok || moved > 0;
  if (improved) {
    A.best_score[b] = score;
    A.best_iter[b] = A.iter;
  }
  if (illegal) A.step[b] = 0;
  A.moved[b] = leg_ok ? moved : -1;
  A.decision[b] = (improved ? 1 : 0) | (illegal ? 2 : 0) | (had_best ? 4 : 0) | (leg_ok ? 8 : 0);
}

// Outer-step update of every (node, restart), coalesced: the improved restarts'
// best schedules, and the resets of the illegal ones (mu from the legalized or the
// prior best schedule, or the midpoint; sigma from sigma_init; moments zeroed).
__global__ void k_outer_apply(const int32_t *decision, const int32_t *sched, int32_t *best_sched, float *mu,
                              float *sg, const float *sg_init, float *m1, float *v1, float *m2, float *v2,
                              const int32_t *asap, const int32_t *alap, int V, int B) {
  const size_t n = (size_t)V * B;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    const int v = (int)(i / B), b = (int)(i % B);
    const int d = decision[b];
    if (d & 1) best_sched[i] = sched[i];
    if (d & 2) {
      // the legalized schedule (Alg. GauS), unless it does not improve on a prior
      // best (App. A: then that best); the midpoint only when legalization failed
      // and there is no best
      mu[i] = ((d & 1) || ((d & 8) && !(d & 4))) ? (float)sched[i]
                                                 : ((d & 4) ? (float)best_sched[i] : 0.5f * (float)(asap[v] + alap[v]));
      sg[i] = sg_init[i];
      m1[i] = 0.f; v1[i] = 0.f; m2[i] = 0.f; v2[i] = 0.f;
    }
  }
}

}  // namespace gaus
