// gaus_fused.cuh -- the whole GauS inner loop (Sec. 3.2-3.3, App. B) as one
// persistent kernel per call: n iterations of loss, gradient, Adam and the
// multiplier update for every restart, with no kernel boundary inside.
//
// Restarts are independent, so the only synchronisation an iteration needs is
// inside a restart: the usage histogram and the forward sums are reductions over
// all of the restart's nodes and edges.  The kernel therefore splits the grid into
// restart groups (RB restarts each, lanes = restarts as in the other kernels); the
// K blocks of a group iterate together and meet at two group barriers per
// iteration, so a group never waits for another one:
//
//   phase 1  node pass: windows, the CDF table rows (C at each window point between
//            a 0 and a 1 sentinel) and the usage histogram of the block's segment,
//            flushed to the restart's histogram U as exact 2^32 fixed-point adds.
//   barrier  (U, tables and windows of the iteration complete)
//   phase 2  per restart, one warp turns U into the LogSumExp / ReLU terms (Eq. max,
//            Eq. relu) and the usage adjoint H = dL/dU; every node then evaluates
//            its own side of each incident edge (Eq. dep with latency, App. B.1 Com,
//            App. B.3 Rec) from the neighbours' table rows and keeps the partial
//            derivative sums (dependency, recurrence, objective) of its own
//            (mu, sigma); the edges' forward sums go to per-restart fixed-point
//            totals.
//   barrier  (forward sums and H complete)
//   phase 3  multiplier coefficients c_k = lambda_k + rho V_k, loss and terms
//            (Sec. 3.3), the usage adjoint over the own window, the gradient, Adam
//            and sigma's floor; lambda <- lambda + rho V.
//
// Each block owns fixed segments of nodes (one class each, level-sorted, so the
// histogram of phase 1 touches a narrow span of bins) in all three phases, so the
// state a block writes in phase 3 is the state it reads in the next phase 1.
// Every per-iteration accumulator is double-buffered by the iteration's parity and
// cleared during the iteration that does not use it.  The barriers wait on a
// per-group arrival counter with a time limit: a group whose barrier times out
// raises a device abort flag, every block leaves its loop at its next barrier and
// the restarts report GAUS_ETIMEOUT.
//
// The node-side evaluation of an edge replaces the per-edge slots of the
// multi-kernel path: the producer and the consumer each compute their own side
// (the same sums as the edge pass, split by side), so no partial is written per
// edge and no gather follows.
#pragma once

#include <climits>
#include <cuda_runtime.h>
#include <stdint.h>

#include "gaus_device.cuh"
#include "gaus_internal.h"
#include "gaus_kernels.cuh"

namespace gaus {

constexpr int kFusedThreads = 768;  // one block per SM: its warps balance the phases
constexpr int kFusedWarps = kFusedThreads / 32;
constexpr int kStage = 32;  // own window points staged per lane in phase 2 (C and density)
constexpr int kMaxRG = 64;  // restarts per group
// CDF table layout: [node][point][restart] (a warp's restarts write neighbouring
// words) or [node][restart][point] (a lane's consecutive points share a line)
constexpr bool kTabPointMajor = true;
// Table row of (node, restart) and the distance between its entries.
__device__ __forceinline__ size_t tab_row(int W, int B, int node, int b) {
  return kTabPointMajor ? (size_t)node * W * B + b : ((size_t)node * B + b) * W;
}
__device__ __forceinline__ size_t tab_stride(int B) { return kTabPointMajor ? (size_t)B : 1; }
// Phase-2 items whose own window exceeds the staging capacity, queued per block and
// done by all its warps after the block's chunks (a node's long windows would
// otherwise run one after another in one warp).
constexpr int kLongQueue = 512;
constexpr unsigned long long kBarrierTimeoutNs = 4000000000ull;  // 4 s per barrier wait
constexpr unsigned kBarrierMaxPolls = 1u << 26;                   // and at most 2^26 polls

struct FusedArgs {
  // RG restarts per group (<= 64); phases 2 and 3 process a node's RG restarts in rows
  // of RBp lanes (32 / RBp nodes per warp when RG <= 16; one node per warp and, for
  // RG > 32, two passes of 32 restarts sorted by window length); phase 1 in rows of
  // RB1 <= RBp restarts, so that its shared-memory histogram fits
  int V, B, D, II, Dh, C, RG, RBp, RB1, G, K, W, n_iters, g0, nseg;
  float k_win, alpha, tau, rho, w_res, lr, beta1, beta2, eps, sigma_min;
  unsigned terms;
  int adam;  // 1: gaus_iterate (Adam, multiplier update); 0: gaus_loss_grad (gradient out)
  // graph in internal order (class, then level)
  const int32_t *perm;  // internal -> caller id
  const float *w;       // demand r_v
  const int32_t *lat, *cls, *seg;
  // phase 2 works on chunks of a node's incident edges: finc entries (neighbour,
  // latency or shift, kind 0 in / 1 out / 2 back in / 3 back out), chunk descriptors
  // in claim order, the chunks with the most edges first (node, first entry,
  // entries, chunk index), cptr (V + 1: a node's chunk indices)
  const int4 *finc, *chunk;
  const int32_t *cptr;
  int nchunk;
  // restart order of every node for the two passes of phases 1-3 (groups of more than
  // 32 restarts), [group of the launch][V][64]: written by phase 1 from the windows
  // it computes, any permutation is valid
  signed char *ord;
  const int32_t *in_ptr;
  const int2 *fin;      // in-edges of v: (producer u, Lat(u))
  const int32_t *out_ptr;
  const int2 *fout;     // out-edges of u: (consumer v, Lat(u))
  const int32_t *bin_ptr;
  const int2 *fbin;     // back edges into i: (j, Lat(j) - k II)
  const int32_t *bout_ptr;
  const int2 *fbout;    // back edges out of j: (i, Lat(j) - k II)
  const float *limit;
  // caller arrays, (V, B) caller order / (B, K) / (B)
  float *mu, *sg, *m_mu, *v_mu, *m_sg, *v_sg;  // Adam mode: read first, written by the last iteration
  float *lambda;
  int32_t *step;
  float *grad_mu, *grad_sg;  // gradient mode
  float *loss, *terms_out;
  int32_t *status;
  // scratch, internal order (V, B)
  float2 *xs;   // (mu, sigma)
  float4 *adm;  // (m_mu, v_mu, m_sigma, v_sigma)
  unsigned *win;  // a | (b + 1) << 16, bit 31: restart unusable
  float *tab;     // (V, B, W) table rows
  float4 *part;   // (nchunk, B): (Ad, Bd, Ao, Bo), the own side of a chunk's edges
  float2 *partr;  // (nchunk, B): (Ar, Br) recurrence partials
  float *H;       // (C, B, Dh) usage adjoint: a restart's bins contiguous
  long long *U;   // [2][B][C][Dh] usage, 2^32 fixed point
  unsigned long long *fwd;  // [2][B][3] forward sums (dep, com, rec), 2^32 fixed point
  unsigned long long *wst;  // [2][B][2] window points / usable items
  int32_t *nonf;            // [2][B]
  double *rstat;            // [B][2]: sum_c LSE_tau(U_c), V_res
  unsigned *bar;            // [G] group arrival counters (zeroed before the launch)
  unsigned bar_extra;       // added to every barrier target: 0 (a test sets 1: no barrier completes)
  unsigned long long bar_limit_ns;  // a barrier wait's time limit
  unsigned *ctr;            // [2][G] phase-2 work counters of the groups, by iteration parity
  int32_t *abort_flag;
  unsigned long long *prof; // optional: globaltimer stamps [n_iters][blocks][6]: iteration start,
                            // phase 1 done, first barrier passed, phase 2 done, second barrier
                            // passed, phase 3 done
};

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ unsigned ld_acquire(const unsigned *p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Group barrier: every block of the group has arrived `target` times.  Bounded:
// after limit_ns of waiting, or kBarrierMaxPolls polls, or once another group has
// aborted, the abort flag is set and false is returned to every thread of the block.
__device__ __forceinline__ bool group_barrier(unsigned *bar, unsigned target, int32_t *abort_flag, int *s_ok,
                                              unsigned long long limit_ns) {
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    __threadfence();
    atomicAdd(bar, 1u);
    unsigned long long t0 = 0;
    for (unsigned polls = 0;; ++polls) {
      if ((int)(ld_acquire(bar) - target) >= 0) break;
      if ((polls & 255u) == 255u) {
        if (*(volatile int32_t *)abort_flag) { ok = 0; break; }
        const unsigned long long t = global_ns();
        if (t0 == 0) t0 = t;
        if (t - t0 > limit_ns || polls >= kBarrierMaxPolls) {
          atomicExch(abort_flag, 1);
          ok = 0;
          break;
        }
      }
      __nanosleep(64);
    }
    __threadfence();
    *s_ok = ok;
  }
  __syncthreads();
  return *s_ok != 0;
}

// A neighbour's windowed CDF in the fused kernel.  The table is rewritten every
// iteration, so it is read through the coherent cache path (ld.global.ca), never
// the read-only one; the barriers' fences make the writes of the previous phase
// visible.
template <int kFam>
struct FNb {
  const float *row;  // table row: [0, C(a), ..., C(b), 1, ...], entries `stride` floats apart
  int a, b;          // window points [a, b]
  int stride;        // B: the table is [node][point][restart]
  bool tab;          // the row holds the window with both sentinels
  float mu, inv;
  __device__ __forceinline__ float at(int x) const {
    if (x < a) return 0.0f;
    if (x > b) return 1.0f;
    return tab ? __ldca(row + (size_t)(x - a + 1) * stride) : Fam<kFam>::cdf(((float)x + 0.5f - mu) * inv);
  }
  __device__ __forceinline__ float at_tab(int x) const {
    return __ldca(row + (size_t)min(max(x - a + 1, 0), b - a + 2) * stride);
  }
  __device__ __forceinline__ float at_direct(int x) const {
    return x < a ? 0.0f : (x > b ? 1.0f : Fam<kFam>::cdf(((float)x + 0.5f - mu) * inv));
  }
  template <bool kTab>
  __device__ __forceinline__ float val(int x) const {
    return kTab ? at_tab(x) : at_direct(x);
  }
};

__device__ __forceinline__ unsigned pack_win(int a, int b, bool ok) {
  return (unsigned)a | ((unsigned)(b + 1) << 16) | (ok ? 0u : 0x80000000u);
}

// The own node of a phase-2 lane: window [a, b], its C and density staged in
// shared memory at st[j * 32].
struct Own {
  int a, b;
  float mu, inv;
  const float2 *st;
};

// Consumer side of an edge u -> v (own = v), Lat = L, or of a back edge j -> i
// (own = i, L = Lat(j) - k II; kBack):
//   V_e = 1 - C_u(b_v + 1 - L) + sum_{t in own} C_v(t) P_u(t + 1 - L)
//   dV_e/dC_v(t) = P_u(t + 1 - L);  L_com part sum_{t in own} C_u(t) (1 - C_v(t))
//   dL_com/dC_v(t) = -C_u(t)
// Visits only the own points where a term can be nonzero (warp-wide trip count).
// kL1: L = 1, so C_u(t) is the bin mass's upper value (no second table read).
template <int kFam, bool kCom, bool kTab, bool kBack, bool kL1>
__device__ __forceinline__ void cons_side(const Own &O, const FNb<kFam> &U, int L, bool on, bool dep, float alpha,
                                          float &Ad, float &Bd, float &Ao, float &Bo, float &fd, float &fc) {
  const int nv = O.b - O.a + 1;
  int jlo = 0, jhi = -1;
  if (on) {
    if (kBack) {
      jlo = max(0, U.a + L - 1 - O.a);
      jhi = min(nv - 1, U.b + L - O.a);
    } else {
      jlo = max(0, U.a + min(dep ? L - 1 : 0, 0) - O.a);
      jhi = kCom ? nv - 1 : min(nv - 1, U.b + L - O.a);
    }
  }
  const int cnt = jhi >= jlo ? jhi - jlo + 1 : 0;
  const int cmax = __reduce_max_sync(0xffffffffu, cnt);
  float c_lo = cnt ? U.template val<kTab>(O.a + jlo - L) : 0.f;
  const float z0 = ((float)(O.a + jlo) + 0.5f - O.mu) * O.inv;  // z of the first point; then + inv per point
  for (int k2 = 0; k2 < cmax; ++k2) {
    if (k2 < cnt) {
      const int j = jlo + k2, t = O.a + j;
      const float c_hi = U.template val<kTab>(t + 1 - L);
      const float p = c_hi - c_lo;
      const float2 cf = O.st[j * 32];
      const float z = fmaf((float)k2, O.inv, z0);
      const float f = cf.y, zf = z * f;
      if (kBack || dep) {
        fd += cf.x * p;
        Ad += p * f;
        Bd += p * zf;
      }
      if (kCom && !kBack) {
        const float cu = kL1 ? c_hi : U.template val<kTab>(t);
        fc += cu * (1.0f - cf.x);
        Ao -= alpha * cu * f;
        Bo -= alpha * cu * zf;
      }
      c_lo = c_hi;
    }
  }
  __syncwarp();
  if (on && (kBack || dep)) fd += 1.0f - U.template val<kTab>(O.b + 1 - L);
}

// Producer side of an edge u -> v (own = u, L = Lat(u)), or of a back edge (own = j;
// kBack):
//   dV_e/dC_u(x) = -P_v(x + L), nonzero for x in [a_v - L, b_v + 1 - L]
//   dL_com/dC_u(x) = 1 - C_v(x), nonzero for x <= b_v
//   L_com part sum_{x in own, x < a_v} C_u(x) + max(0, a_v - 1 - b_u)
// kL1: L = 1, so C_v(x) is the bin mass's lower value.
template <int kFam, bool kCom, bool kTab, bool kBack, bool kL1>
__device__ __forceinline__ void prod_side(const Own &O, const FNb<kFam> &Vn, int L, bool on, bool dep, float alpha,
                                          float &Ad, float &Bd, float &Ao, float &Bo, float &fc) {
  const int nu = O.b - O.a + 1;
  int jlo = 0, jhi = -1;
  if (on) {
    jlo = max(0, Vn.a - L - O.a);
    jhi = min(nu - 1, Vn.b + 1 - L - O.a);
    if (kCom && !kBack) {
      jlo = 0;
      jhi = max(jhi, min(nu - 1, Vn.b - O.a));
    }
  }
  const int cnt = jhi >= jlo ? jhi - jlo + 1 : 0;
  const int cmax = __reduce_max_sync(0xffffffffu, cnt);
  float c_lo = cnt ? Vn.template val<kTab>(O.a + jlo + L - 1) : 0.f;
  const float z0 = ((float)(O.a + jlo) + 0.5f - O.mu) * O.inv;
  for (int k2 = 0; k2 < cmax; ++k2) {
    if (k2 < cnt) {
      const int j = jlo + k2, x = O.a + j;
      const float c_hi = Vn.template val<kTab>(x + L);
      const float2 cf = O.st[j * 32];
      const float z = fmaf((float)k2, O.inv, z0);
      const float f = cf.y, zf = z * f;
      const float p = c_hi - c_lo;
      if (kBack || dep) {
        Ad -= p * f;
        Bd -= p * zf;
      }
      if (kCom && !kBack) {
        const float cw = kL1 ? c_lo : Vn.template val<kTab>(x);
        Ao += alpha * (1.0f - cw) * f;
        Bo += alpha * (1.0f - cw) * zf;
        if (x < Vn.a) fc += cf.x;
      }
      c_lo = c_hi;
    }
  }
  __syncwarp();
  if (on && kCom && !kBack) fc += (float)max(0, Vn.a - 1 - O.b);
}

// A neighbour (node ni, restart b) of a phase-2 item from its packed window w:
// window, table row and, for a window the row cannot hold, its mean and 1/sigma
// for direct evaluation.  False when the neighbour is inactive or unusable.
template <int kFam>
__device__ __forceinline__ bool make_nb(const FusedArgs &A, int ni, int b, unsigned w, bool active, FNb<kFam> &N) {
  const size_t ix = (size_t)ni * A.B + b;
  N.a = (int)(w & 0xFFFFu);
  N.b = (int)((w >> 16) & 0x7FFFu) - 1;
  N.row = A.tab + tab_row(A.W, A.B, ni, b);
  N.stride = (int)tab_stride(A.B);
  N.tab = N.b - N.a + 4 <= A.W;  // n + 3 <= W, as the node pass writes it
  N.mu = 0.f;
  N.inv = 1.f;
  const bool ok = active && !(w >> 31);
  if (ok && !N.tab) {
    const float2 x = A.xs[ix];
    N.mu = x.x;
    N.inv = 1.0f / x.y;
  }
  return ok;
}

template <int kFam>
__device__ __forceinline__ bool load_nb(const FusedArgs &A, int ni, int b, bool active, FNb<kFam> &N) {
  const unsigned w = active ? A.win[(size_t)ni * A.B + b] : 0x80000000u;
  return make_nb<kFam>(A, ni, b, w, active, N);
}

// The own side of every edge of a chunk (consumer side of in-edges and back edges
// in, producer side of out-edges and back edges out) for the phase-2 lanes of a
// warp, which all work on the same node: the entries and their kinds are
// warp-uniform.  The chunk's entries (at most kChunkEdges) and then all their
// neighbours' windows are loaded before the first edge is evaluated (two round
// trips per chunk instead of two per edge), and rotate through registers.
template <int kFam, bool kCom>
__device__ __forceinline__ void chunk_edges(const FusedArgs &A, int e0, int ne, int b, bool act, const Own &O,
                                            bool dep, bool com, bool rec, float &Ad, float &Bd, float &Ao, float &Bo,
                                            float &Ar, float &Br, float &fd, float &fc, float &fr) {
  constexpr unsigned FULL = 0xffffffffu;
  static_assert(kChunkEdges == 4, "the register pipeline holds four entries");
  if (ne <= 0) return;
  const int4 none = make_int4(0, 1, -1, 0);
  int4 en_a = __ldg(A.finc + e0);
  int4 en_b = ne > 1 ? __ldg(A.finc + e0 + 1) : none;
  int4 en_c = ne > 2 ? __ldg(A.finc + e0 + 2) : none;
  int4 en_d = ne > 3 ? __ldg(A.finc + e0 + 3) : none;
  unsigned w_a = act ? A.win[(size_t)en_a.x * A.B + b] : 0x80000000u;
  unsigned w_b = (ne > 1 && act) ? A.win[(size_t)en_b.x * A.B + b] : 0x80000000u;
  unsigned w_c = (ne > 2 && act) ? A.win[(size_t)en_c.x * A.B + b] : 0x80000000u;
  unsigned w_d = (ne > 3 && act) ? A.win[(size_t)en_d.x * A.B + b] : 0x80000000u;
  for (int q = 0; q < ne; ++q) {
    const int kind = en_a.z, L = en_a.y;
    FNb<kFam> N;
    const bool on = make_nb<kFam>(A, en_a.x, b, w_a, act, N) && act;
    const bool tb = on && N.tab, dr = on && !N.tab;
    // the entry (and so its kind and latency) is the same on every lane
    if (kind == 0 && (dep || com)) {
      if (L == 1) {
        cons_side<kFam, kCom, true, false, true>(O, N, L, tb, dep, A.alpha, Ad, Bd, Ao, Bo, fd, fc);
        if (__any_sync(FULL, dr))
          cons_side<kFam, kCom, false, false, true>(O, N, L, dr, dep, A.alpha, Ad, Bd, Ao, Bo, fd, fc);
      } else {
        cons_side<kFam, kCom, true, false, false>(O, N, L, tb, dep, A.alpha, Ad, Bd, Ao, Bo, fd, fc);
        if (__any_sync(FULL, dr))
          cons_side<kFam, kCom, false, false, false>(O, N, L, dr, dep, A.alpha, Ad, Bd, Ao, Bo, fd, fc);
      }
    } else if (kind == 1 && (dep || com)) {
      if (L == 1) {
        prod_side<kFam, kCom, true, false, true>(O, N, L, tb, dep, A.alpha, Ad, Bd, Ao, Bo, fc);
        if (__any_sync(FULL, dr))
          prod_side<kFam, kCom, false, false, true>(O, N, L, dr, dep, A.alpha, Ad, Bd, Ao, Bo, fc);
      } else {
        prod_side<kFam, kCom, true, false, false>(O, N, L, tb, dep, A.alpha, Ad, Bd, Ao, Bo, fc);
        if (__any_sync(FULL, dr))
          prod_side<kFam, kCom, false, false, false>(O, N, L, dr, dep, A.alpha, Ad, Bd, Ao, Bo, fc);
      }
    } else if (kind == 2 && rec) {
      float dummy0 = 0.f, dummy1 = 0.f, dummy2 = 0.f;
      cons_side<kFam, false, true, true, false>(O, N, L, tb, dep, A.alpha, Ar, Br, dummy0, dummy1, fr, dummy2);
      if (__any_sync(FULL, dr))
        cons_side<kFam, false, false, true, false>(O, N, L, dr, dep, A.alpha, Ar, Br, dummy0, dummy1, fr, dummy2);
    } else if (kind == 3 && rec) {
      float dummy0 = 0.f, dummy1 = 0.f, dummy2 = 0.f;
      prod_side<kFam, false, true, true, false>(O, N, L, tb, dep, A.alpha, Ar, Br, dummy0, dummy1, dummy2);
      if (__any_sync(FULL, dr))
        prod_side<kFam, false, false, true, false>(O, N, L, dr, dep, A.alpha, Ar, Br, dummy0, dummy1, dummy2);
    }
    en_a = en_b; en_b = en_c; en_c = en_d;
    w_a = w_b; w_b = w_c; w_c = w_d;
  }
}

// Phase 2 for one (node, restart) whose window is too long for the per-lane path:
// the whole warp, lanes over the own points (32 at a time), every edge of the
// chunk (entries e0 .. e0 + ne) evaluated at each lane's point.  The sums are the
// per-lane path's, reduced over the warp; every lane returns them.
template <int kFam, bool kCom>
__device__ void coop_node(const FusedArgs &A, int e0, int ne, int b, int a, int bw, float mu, float inv, bool dep,
                          bool com, bool rec, float r9[9]) {
  const int lane = threadIdx.x & 31;
  float Ad = 0.f, Bd = 0.f, Ao = 0.f, Bo = 0.f, Ar = 0.f, Br = 0.f, fd = 0.f, fc = 0.f, fr = 0.f;
  const int n = bw - a + 1;
  const float alpha = A.alpha;
  // the neighbours' windows, once for all the point batches: lane q holds entry q's
  // (the warp works on one restart); the entries themselves are L1 hits
  const unsigned my_w = lane < ne ? A.win[(size_t)__ldg(A.finc + e0 + lane).x * A.B + b] : 0x80000000u;
  for (int p0 = 0; p0 == 0 || p0 < n; p0 += 32) {
    const int j = p0 + lane;
    const bool pt = j < n;
    const int t = a + j;
    const float z = ((float)t + 0.5f - mu) * inv;
    const float q = pt ? Fam<kFam>::tail(z) : 0.f;
    const float Cv = z <= 0.f ? q : 1.0f - q;
    const float f = pt ? Fam<kFam>::pdf(z) : 0.f;
    const float zf = z * f;
    const bool first = p0 == 0 && lane == 0;
    for (int e = 0; e < ne; ++e) {
      const unsigned wn = __shfl_sync(0xffffffffu, my_w, e);
      const int4 en = __ldg(A.finc + e0 + e);
      const int kind = en.z, L = en.y;
      if (kind <= 1 && !(dep || com)) continue;
      if (kind >= 2 && !rec) continue;
      FNb<kFam> N;
      if (!make_nb<kFam>(A, en.x, b, wn, true, N)) continue;
      if (kind == 0) {
        const float hi = N.at(t + 1 - L), lo = N.at(t - L), p = hi - lo;
        if (pt) {
          if (dep) { fd += Cv * p; Ad += p * f; Bd += p * zf; }
          if (kCom) {
            const float cu = (L == 1) ? hi : N.at(t);
            fc += cu * (1.0f - Cv);
            Ao -= alpha * cu * f;
            Bo -= alpha * cu * zf;
          }
        }
        if (dep && first) fd += 1.0f - N.at(bw + 1 - L);
      } else if (kind == 1) {
        const float hi = N.at(t + L), lo = N.at(t + L - 1);
        if (pt) {
          if (dep) { Ad -= (hi - lo) * f; Bd -= (hi - lo) * zf; }
          if (kCom) {
            const float cw = (L == 1) ? lo : N.at(t);
            Ao += alpha * (1.0f - cw) * f;
            Bo += alpha * (1.0f - cw) * zf;
            if (t < N.a) fc += Cv;
          }
        }
        if (kCom && first) fc += (float)max(0, N.a - 1 - bw);
      } else if (kind == 2) {
        const float p = N.at(t + 1 - L) - N.at(t - L);
        if (pt) { fr += Cv * p; Ar += p * f; Br += p * zf; }
        if (first) fr += 1.0f - N.at(bw + 1 - L);
      } else {
        const float p = N.at(t + L) - N.at(t + L - 1);
        if (pt) { Ar -= p * f; Br -= p * zf; }
      }
    }
  }
  __syncwarp();
  r9[0] = warp_sum(Ad); r9[1] = warp_sum(Bd); r9[2] = warp_sum(Ao); r9[3] = warp_sum(Bo);
  r9[4] = warp_sum(Ar); r9[5] = warp_sum(Br);
  r9[6] = warp_sum(fd); r9[7] = warp_sum(fc); r9[8] = warp_sum(fr);
}

// Per restart, one warp: the usage terms of Eq. max and Eq. relu from the exact
// histogram U (every class's max, exact ReLU excess over finite limits, the sums of
// exp((U - m)/tau) in a fixed order), the multiplier coefficient of the resource
// constraint, and the usage adjoint H = w_res softmax + c_res [U > R].
static __device__ __noinline__ void restart_usage(const FusedArgs &A, int b, int p, float lam_res, long long *s_m, float *s_s) {
  const int lane = threadIdx.x & 31, Dh = A.Dh, C = A.C;
  const long long *Ub = A.U + ((size_t)p * A.B + b) * C * Dh;
  const bool on_robj = A.terms & GAUS_RES_OBJ, on_rv = A.terms & GAUS_RES_VIOL;
  long long ex = 0;
  for (int c = 0; c < C; ++c) {
    const float Rf = __ldg(A.limit + c);
    const long long R = (isfinite(Rf) && Rf < 1.0e9f)
                            ? (long long)Rf * 4294967296LL + (long long)((Rf - floorf(Rf)) * 4294967296.0f)
                            : LLONG_MAX;
    long long m = LLONG_MIN;
    for (int t = lane; t < Dh; t += 32) {
      const long long u = __ldcg(Ub + c * Dh + t);
      m = max(m, u);
      if (R != LLONG_MAX && u > R) ex += u - R;
    }
    for (int o = 16; o > 0; o >>= 1) m = max(m, (long long)__shfl_xor_sync(0xffffffffu, m, o));
    float s = 0.f;
    for (int t = lane; t < Dh; t += 32) s += soft_exp(__ldcg(Ub + c * Dh + t) - m, A.tau);
    s = warp_sum(s);
    if (lane == 0) {
      s_m[c] = m;
      s_s[c] = s;
    }
  }
  for (int o = 16; o > 0; o >>= 1) ex += __shfl_xor_sync(0xffffffffu, ex, o);
  __syncwarp();
  const double vres = (double)ex * kInvFix;
  const float c_res = on_rv ? (float)((double)lam_res + (double)A.rho * vres) : 0.f;
  for (int i = lane; i < C * Dh; i += 32) {
    const int c = i / Dh;
    const long long u = __ldcg(Ub + i);
    float h = 0.f;
    if (on_robj) h += A.w_res * soft_exp(u - s_m[c], A.tau) / s_s[c];
    if (on_rv) {
      const float Rf = __ldg(A.limit + c);
      if (isfinite(Rf) && Rf < 1.0e9f) {
        const long long R = (long long)Rf * 4294967296LL + (long long)((Rf - floorf(Rf)) * 4294967296.0f);
        if (u > R) h += c_res;
      }
    }
    A.H[((size_t)c * A.B + b) * Dh + (i - c * Dh)] = h;
  }
  if (lane == 0) {
    double lse = 0.0;
    for (int c = 0; c < C; ++c) lse += (double)s_m[c] * kInvFix + (double)A.tau * (double)logf(s_s[c]);
    A.rstat[2 * b] = lse;
    A.rstat[2 * b + 1] = vres;
  }
  __syncwarp();
}


// round(x 2^32) for a node's forward sum 0 <= x < 2^31 (a node sums all its incident
// edges, so the edge pass's 2^16 range of to_fix is not enough), with 32-bit
// conversions only; equal to to_fix(x) wherever that is defined.
__device__ __forceinline__ long long to_fix_node(float x) {
  x = fmaxf(x, 0.0f);
  const float xi = floorf(x);
  const float fr = (x - xi) * 65536.0f;
  const float fh = floorf(fr);
  return ((long long)(unsigned)xi << 32) + ((long long)(unsigned)fh << 16) +
         (long long)__float2uint_rn((fr - fh) * 65536.0f);
}

// Static shared memory of the fused kernel.
struct FusedShared {
  int ok, next, lo, hi;
  int ws[kMaxRG], wc[kMaxRG];                  // window statistics per restart of the group
  float lam[kMaxRG][GAUS_K], coef[kMaxRG][4];  // multipliers; c_dep, c_rec, Adam bias corrections
  int step[kMaxRG];
  unsigned long long fw[3][kMaxRG];            // the block's forward sums per restart
  long long m[kFusedWarps][kMaxClasses];       // per-warp scratch of the usage terms
  float s[kFusedWarps][kMaxClasses];
  int map[kFusedWarps][64];                    // per-warp restart order of a node (two passes)
  int nlong, qnext;                            // phase 2: long-window items queued, taken
  int4 lq[kLongQueue];                         // (node, restart, chunk, first entry | entries << 28)
};

// Orders a node's RG (33..64) restarts for two passes of 32 lanes: the 32 with the
// shortest windows first, so that each pass's per-lane loops run to a similar
// length.  Lane l holds two restarts id0, id1 (-1: none) with window lengths k0, k1.
// Writes map[0..63] = restart of each (pass, lane) slot, -1 for none.  Any order
// gives the same per-restart results: every (node, restart) item is computed by one
// lane.
__device__ __forceinline__ void split_by_window(int k0, int id0, int k1, int id1, int *map) {
  constexpr unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const unsigned lt = (1u << lane) - 1u;
  // keys clamped to 64 (longer windows all go last), absent slots after every key
  k0 = id0 < 0 ? 65 : min(k0, 64);
  k1 = id1 < 0 ? 65 : min(k1, 64);
  int lo = 0, hi = 64;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    const int c = __popc(__ballot_sync(FULL, k0 <= mid)) + __popc(__ballot_sync(FULL, k1 <= mid));
    if (c >= 32) hi = mid; else lo = mid + 1;
  }
  const int m = lo;
  const int nlt = __popc(__ballot_sync(FULL, k0 < m)) + __popc(__ballot_sync(FULL, k1 < m));
  const int need = 32 - nlt;
  const unsigned e0 = __ballot_sync(FULL, k0 == m), e1 = __ballot_sync(FULL, k1 == m);
  const int r0 = __popc(e0 & lt), r1 = __popc(e0) + __popc(e1 & lt);
  const bool in0 = k0 < m || (k0 == m && r0 < need);
  const bool in1 = k1 < m || (k1 == m && r1 < need);
  const unsigned b0 = __ballot_sync(FULL, in0), b1 = __ballot_sync(FULL, in1);
  const int p0 = in0 ? __popc(b0 & lt) : 32 + __popc(~b0 & lt);
  const int p1 = in1 ? __popc(b0) + __popc(b1 & lt) : 32 + __popc(~b0) + __popc(~b1 & lt);
  __syncwarp();
  map[p0] = id0;
  map[p1] = id1;
  __syncwarp();
}

// The restart order of node vi (group g) for two passes, as stored by phase 1: map
// (per-warp shared memory) = ord[g][vi][0..63].
__device__ __forceinline__ void load_order(const FusedArgs &A, int vi, int g, int *map) {
  const int lane = threadIdx.x & 31;
  const signed char *o = A.ord + ((size_t)(g - A.g0) * A.V + vi) * 64;
  const int x0 = o[lane], x1 = o[32 + lane];
  __syncwarp();
  map[lane] = x0;
  map[32 + lane] = x1;
  __syncwarp();
}

// Phase 2 for the lane's (node vc, restart b, state x = (mu, sigma)): stage the own window's C and
// density, evaluate the own side of every incident edge (per lane; a window
// longer than the staging capacity by the whole warp), store the partials and add
// the forward sums to the block's per-restart totals.  All lanes of the warp call
// it (warp-wide trip counts).
template <int kFam, bool kCom>
__device__ __forceinline__ void p2_lane(const FusedArgs &A, FusedShared &S, int vc, int ch, int e0, int ne, int b,
                                        int rl, bool present, float2 x, float2 *st, bool dep, bool com, bool rec) {
  constexpr unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int bs = present ? b : 0;
  const bool ok = present && usable(x.x, x.y);
  const float inv = ok ? 1.0f / x.y : 1.0f;
  int a = 0, bw = -1;
  if (ok) window(x.x, x.y, A.k_win, A.D, a, bw);
  const int n = ok ? bw - a + 1 : 0;
  const bool is_long = ok && n > kStage;
  const int nl = (ok && !is_long) ? n : 0;
  const bool act = ok && !is_long;
  float Ad = 0.f, Bd = 0.f, Ao = 0.f, Bo = 0.f, Ar = 0.f, Br = 0.f, fd = 0.f, fc = 0.f, fr = 0.f;
  if (__all_sync(FULL, nl == 0 && !is_long)) {
    // no lane has an own point (late in a run, most windows are empty): only the
    // terms that do not depend on them -- the dependency and recurrence tails
    // 1 - C_u(b_v + 1 - L) of the in-edges and the communication gaps
    // max(0, a_w - 1 - b_v) of the out-edges -- with the general path's arithmetic
    // (entries, then windows, then table values: three round trips per chunk)
    int4 en[kChunkEdges];
    unsigned w[kChunkEdges];
    float cv[kChunkEdges];
#pragma unroll
    for (int q = 0; q < kChunkEdges; ++q) {
      en[q] = q < ne ? __ldg(A.finc + e0 + q) : make_int4(0, 1, -1, 0);
      const int kind = en[q].z;
      const bool need = act && ((kind == 0 && dep) || (kind == 1 && kCom) || (kind == 2 && rec));
      if (!need) en[q].z = -1;
    }
#pragma unroll
    for (int q = 0; q < kChunkEdges; ++q) w[q] = en[q].z >= 0 ? A.win[(size_t)en[q].x * A.B + bs] : 0x80000000u;
#pragma unroll
    for (int q = 0; q < kChunkEdges; ++q) {
      FNb<kFam> N;
      const bool ok_q = make_nb<kFam>(A, en[q].x, bs, w[q], en[q].z >= 0, N);
      if (!ok_q) en[q].z = -1;
      // kind 1 keeps the neighbour's first point in cv
      cv[q] = (en[q].z == 0 || en[q].z == 2) ? N.at(a - en[q].y) : (float)N.a;
    }
#pragma unroll
    for (int q = 0; q < kChunkEdges; ++q) {
      if (en[q].z == 0) fd += 1.0f - cv[q];
      else if (en[q].z == 1) fc += (float)max(0, (int)cv[q] - a);
      else if (en[q].z == 2) fr += 1.0f - cv[q];
    }
  } else {
    const int nst = __reduce_max_sync(FULL, nl);
    for (int j = 0; j < nst; ++j)
      if (j < nl) {
        const float z = ((float)(a + j) + 0.5f - x.x) * inv;
        const float q = Fam<kFam>::tail(z);
        st[j * 32] = make_float2(z <= 0.f ? q : 1.0f - q, Fam<kFam>::pdf(z));
      }
    __syncwarp();
    Own O;
    O.a = a; O.b = act ? bw : a - 1; O.mu = x.x; O.inv = inv; O.st = st;
    chunk_edges<kFam, kCom>(A, e0, ne, bs, act, O, dep, com, rec, Ad, Bd, Ao, Bo, Ar, Br, fd, fc, fr);
  }
  // long windows: queued for the block's warps (p2_long), or, when the queue is full,
  // done here by the whole warp, one after another
  bool queued = false;
  if (is_long) {
    const int q = atomicAdd(&S.nlong, 1);
    if (q < kLongQueue) {
      S.lq[q] = make_int4(vc, b, ch, e0 | (ne << 28));
      queued = true;
    }
  }
  unsigned longmask = __ballot_sync(FULL, is_long && !queued);
  while (longmask) {
    const int src = __ffs(longmask) - 1;
    longmask &= longmask - 1;
    const int l_b = __shfl_sync(FULL, b, src);
    const int l_a = __shfl_sync(FULL, a, src), l_bw = __shfl_sync(FULL, bw, src);
    const float l_mu = __shfl_sync(FULL, x.x, src), l_inv = __shfl_sync(FULL, inv, src);
    float r9[9];
    coop_node<kFam, kCom>(A, e0, ne, l_b, l_a, l_bw, l_mu, l_inv, dep, com, rec, r9);
    if (lane == src) {
      Ad = r9[0]; Bd = r9[1]; Ao = r9[2]; Bo = r9[3]; Ar = r9[4]; Br = r9[5];
      fd = r9[6]; fc = r9[7]; fr = r9[8];
    }
  }
  if (present && !queued) {
    const size_t ci = (size_t)ch * A.B + bs;
    A.part[ci] = make_float4(Ad, Bd, Ao, Bo);
    if (rec) A.partr[ci] = make_float2(Ar, Br);
    // per-restart forward sums: exact integers, any order
    const long long xd = to_fix_node(fd), xc = to_fix_node(fc), xr = to_fix_node(fr);
    if (xd) atomicAdd(&S.fw[0][rl], (unsigned long long)xd);
    if (xc) atomicAdd(&S.fw[1][rl], (unsigned long long)xc);
    if (xr) atomicAdd(&S.fw[2][rl], (unsigned long long)xr);
  }
}

// A queued long-window item of phase 2 (node, restart, chunk), done by the whole warp:
// its own side of the chunk's edges (coop_node), partials and forward sums stored as
// the per-lane path stores them.
template <int kFam, bool kCom>
__device__ __forceinline__ void p2_long(const FusedArgs &A, FusedShared &S, int4 q, bool dep, bool com, bool rec) {
  const int lane = threadIdx.x & 31;
  const int vc = q.x, b = q.y, ch = q.z, e0 = q.w & 0x0FFFFFFF, ne = (int)((unsigned)q.w >> 28);
  const int rl = b % A.RG;
  const float2 x = A.xs[(size_t)vc * A.B + b];
  const float inv = 1.0f / x.y;
  int a, bw;
  window(x.x, x.y, A.k_win, A.D, a, bw);
  float r9[9];
  coop_node<kFam, kCom>(A, e0, ne, b, a, bw, x.x, inv, dep, com, rec, r9);
  if (lane == 0) {
    const size_t ci = (size_t)ch * A.B + b;
    A.part[ci] = make_float4(r9[0], r9[1], r9[2], r9[3]);
    if (rec) A.partr[ci] = make_float2(r9[4], r9[5]);
    const long long xd = to_fix_node(r9[6]), xc = to_fix_node(r9[7]), xr = to_fix_node(r9[8]);
    if (xd) atomicAdd(&S.fw[0][rl], (unsigned long long)xd);
    if (xc) atomicAdd(&S.fw[1][rl], (unsigned long long)xc);
    if (xr) atomicAdd(&S.fw[2][rl], (unsigned long long)xr);
  }
}

// Usage adjoint of one (node, restart) over its own window, done by the whole warp
// (lanes over the window's points): the window longer than the staging capacity.
// dL/dC_v(t) = w_v (H(t) - H(t + 1)) against the density and z density; every lane
// returns the warp's sums.
template <int kFam>
__device__ __forceinline__ float2 coop_usage(const FusedArgs &A, const float *Hrow, int a, int n, float mu, float inv,
                                             float w) {
  const int lane = threadIdx.x & 31;
  float pa = 0.f, pb = 0.f;
  for (int q = 0; q < n; q += 32) {
    const int j = q + lane;
    if (j < n) {
      const int t = a + j;
      const float z = ((float)t + 0.5f - mu) * inv;
      const float f = Fam<kFam>::pdf(z);
      const float gh = w * (__ldca(Hrow + fold_bin(t, A.II)) - __ldca(Hrow + fold_bin(t + 1, A.II)));
      pa += gh * f;
      pb += gh * z * f;
    }
  }
  return make_float2(warp_sum(pa), warp_sum(pb));
}

// Phase 3 for node vc: lane l takes the group's restarts l and l + 32, so that the
// state, the Adam moments and the chunk partials of both are loaded at once (one
// round trip) and the two items overlap.  Per item: the usage adjoint over the own
// window (dL/dC_v(t) = w_v (H(t) - H(t + 1)); a window longer than the staging
// capacity by the whole warp), the node's chunk partials summed in a fixed order,
// the gradient, and Adam with sigma's floor (or the gradient itself in gradient
// mode).  `last`: the last iteration of the call, whose state goes to the caller's
// arrays.  All lanes of the warp call it.
template <int kFam>
__device__ __forceinline__ void p3_node(const FusedArgs &A, const FusedShared &S, int vc, int g, bool hist, bool rec,
                                        bool last) {
  constexpr unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31, Dh = A.Dh, B = A.B;
  int rl[2], b[2];
  bool pres[2], ok[2];
  size_t ii[2];
  float2 x[2];
  float4 m[2], pd[2];
  float2 pr[2];
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    rl[q] = lane + 32 * q;
    b[q] = g * A.RG + rl[q];
    pres[q] = rl[q] < A.RG && b[q] < B;
    ii[q] = (size_t)vc * B + (pres[q] ? b[q] : 0);
    x[q] = pres[q] ? A.xs[ii[q]] : make_float2(0.f, 1.f);
    m[q] = (pres[q] && A.adam) ? A.adm[ii[q]] : make_float4(0.f, 0.f, 0.f, 0.f);
    pd[q] = make_float4(0.f, 0.f, 0.f, 0.f);
    pr[q] = make_float2(0.f, 0.f);
  }
  // the node's chunks in a fixed order
  const int c0 = __ldg(A.cptr + vc), c1 = __ldg(A.cptr + vc + 1);
  for (int c = c0; c < c1; ++c)
#pragma unroll
    for (int q = 0; q < 2; ++q)
      if (pres[q]) {
        const size_t ci = (size_t)c * B + b[q];
        const float4 q4 = __ldcg(A.part + ci);
        pd[q].x += q4.x; pd[q].y += q4.y; pd[q].z += q4.z; pd[q].w += q4.w;
        if (rec) {
          const float2 q2 = __ldcg(A.partr + ci);
          pr[q].x += q2.x; pr[q].y += q2.y;
        }
      }
  const int cls = __ldg(A.cls + vc);
  const float wv = __ldg(A.w + vc);
  float inv[2], Ah[2] = {0.f, 0.f}, Bh[2] = {0.f, 0.f};
  int a[2], n[2];
  bool lng[2];
  const float *Hr[2];
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    ok[q] = pres[q] && usable(x[q].x, x[q].y);
    inv[q] = ok[q] ? 1.0f / x[q].y : 1.0f;
    int aa = 0, bw = -1;
    if (ok[q]) window(x[q].x, x[q].y, A.k_win, A.D, aa, bw);
    a[q] = aa;
    n[q] = bw - aa + 1;
    lng[q] = hist && ok[q] && n[q] > kStage;
    Hr[q] = A.H + ((size_t)cls * B + (pres[q] ? b[q] : 0)) * Dh;
  }
  if (hist) {
    // both items' windows in one loop: dL/dC_v(t) = w_v (H(t) - H(t + 1)), each bin's
    // value carried to the next point
    const int n0 = lng[0] ? 0 : n[0], n1 = lng[1] ? 0 : n[1];
    const int nmax = __reduce_max_sync(FULL, max(n0, n1));
    float hl0 = n0 > 0 ? __ldca(Hr[0] + fold_bin(a[0], A.II)) : 0.f;
    float hl1 = n1 > 0 ? __ldca(Hr[1] + fold_bin(a[1], A.II)) : 0.f;
    for (int j = 0; j < nmax; ++j) {
      if (j < n0) {
        const int t = a[0] + j;
        const float z = ((float)t + 0.5f - x[0].x) * inv[0];
        const float f = Fam<kFam>::pdf(z);
        const float hh = __ldca(Hr[0] + fold_bin(t + 1, A.II));
        const float gh = wv * (hl0 - hh);
        hl0 = hh;
        Ah[0] += gh * f;
        Bh[0] += gh * z * f;
      }
      if (j < n1) {
        const int t = a[1] + j;
        const float z = ((float)t + 0.5f - x[1].x) * inv[1];
        const float f = Fam<kFam>::pdf(z);
        const float hh = __ldca(Hr[1] + fold_bin(t + 1, A.II));
        const float gh = wv * (hl1 - hh);
        hl1 = hh;
        Ah[1] += gh * f;
        Bh[1] += gh * z * f;
      }
    }
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      unsigned longmask = __ballot_sync(FULL, lng[q]);
      while (longmask) {
        const int src = __ffs(longmask) - 1;
        longmask &= longmask - 1;
        const int l_a = __shfl_sync(FULL, a[q], src), l_n = __shfl_sync(FULL, n[q], src);
        const int l_b = __shfl_sync(FULL, pres[q] ? b[q] : 0, src);
        const float l_mu = __shfl_sync(FULL, x[q].x, src), l_inv = __shfl_sync(FULL, inv[q], src);
        const float2 r = coop_usage<kFam>(A, A.H + ((size_t)cls * B + l_b) * Dh, l_a, l_n, l_mu, l_inv, wv);
        if (lane == src) { Ah[q] = r.x; Bh[q] = r.y; }
      }
    }
  }
  const int pv = __ldg(A.perm + vc);
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    if (!pres[q]) continue;
    if (!ok[q]) { pd[q] = make_float4(0.f, 0.f, 0.f, 0.f); pr[q] = make_float2(0.f, 0.f); }
    const int r = rl[q];
    const float c_dep = S.coef[r][0], c_rec = S.coef[r][1];
    const float Asum = c_dep * pd[q].x + pd[q].z + c_rec * pr[q].x + Ah[q];
    const float Bsum = c_dep * pd[q].y + pd[q].w + c_rec * pr[q].y + Bh[q];
    const float rs = ok[q] ? __frcp_rn(x[q].y) : 0.f;
    const float gm = -Asum * rs, gs = -Bsum * rs;
    const size_t ci = (size_t)pv * B + b[q];
    if (!A.adam) {
      A.grad_mu[ci] = gm;
      A.grad_sg[ci] = gs;
      continue;
    }
    float4 m4 = m[q];
    const float nmu = adam_update(x[q].x, gm, m4.x, m4.y, A.lr, A.beta1, A.beta2, A.eps, S.coef[r][2], S.coef[r][3]);
    const float nsg = fmaxf(
        adam_update(x[q].y, gs, m4.z, m4.w, A.lr, A.beta1, A.beta2, A.eps, S.coef[r][2], S.coef[r][3]), A.sigma_min);
    if (last) {
      A.mu[ci] = nmu; A.sg[ci] = nsg;
      A.m_mu[ci] = m4.x; A.v_mu[ci] = m4.y; A.m_sg[ci] = m4.z; A.v_sg[ci] = m4.w;
    } else {
      A.xs[ii[q]] = make_float2(nmu, nsg);
      A.adm[ii[q]] = m4;
    }
  }
}

// Phase 1 for the lane's (node vi, restart b, state x = (mu, sigma); rl its index in
// the group, hc its column in the histogram of cs restarts per bin): the window, the CDF table row with its 0/1
// sentinels, and the bin masses into the shared-memory histogram ([bin][restart],
// two exact 16-bit halves of 2^32 fixed point).  Windows much longer than the
// warp's typical one are done by the whole warp (the table values are per point and
// the histogram sums exact, so the results do not depend on the split).  lo / hi
// collect the span of bins touched; returns the window's points (0 if unusable).
// All lanes of the warp call it.
template <int kFam>
__device__ __forceinline__ int p1_lane(const FusedArgs &A, FusedShared &S, unsigned *hlo, int cs, int vi, int rl,
                                       int hc, int b, bool present, float2 x, int p, bool hist, int &lo, int &hi) {
  constexpr unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31, B = A.B;
  unsigned *hhi = hlo + (size_t)A.Dh * cs;
  const int bs = present ? b : 0;
  const size_t ii = (size_t)vi * B + bs;
  const float mu = x.x, sg = x.y;
  const bool valid = present && usable(mu, sg);
  if (present && !valid) A.nonf[(size_t)p * B + b] = 1;
  const float inv_s = valid ? 1.0f / sg : 1.0f, wv = __ldg(A.w + vi);
  int a = 0, bw = -1;
  if (valid) window(mu, sg, A.k_win, A.D, a, bw);
  if (present) A.win[ii] = pack_win(a, bw, valid);
  const int n = valid ? bw - a + 1 : -1;
  if (valid) {
    atomicAdd(&S.ws[rl], min(n, 4096));
    atomicAdd(&S.wc[rl], 1);
  }
  const int nact = __popc(__ballot_sync(FULL, valid));
  const int mean = nact ? __reduce_add_sync(FULL, max(n, 0)) / nact : 0;
  // long: well above the warp's typical window, or above the staging capacity (a pass
  // of the sorted order can hold many long windows, which would make every lane's
  // loop run to the longest)
  const bool is_long = valid && n > min(kStage, max(8, 2 * mean + 8));
  const int nl = is_long ? -1 : n;
  const int nmax = __reduce_max_sync(FULL, nl);
  // table row: [node][point][restart], so that a warp's restarts write and read
  // neighbouring words
  float *row = A.tab + tab_row(A.W, B, vi, bs);
  const size_t ts = tab_stride(B);
  const bool tabled = n >= 0 && n + 3 <= A.W;
  if (tabled && !is_long) row[0] = 0.0f;
  float zp = 0.f, qp = 0.f;
  for (int j = 0; j <= nmax; ++j) {
    const bool pt = j < nl;
    const float zc = ((float)(a + j) + 0.5f - mu) * inv_s;
    const float qc = pt ? Fam<kFam>::tail(zc) : 0.f;
    if (tabled && j <= nl) row[(size_t)(j + 1) * ts] = pt ? (zc <= 0.f ? qc : 1.0f - qc) : 1.0f;
    if (hist && j <= nl)
      hist_add(hlo, hhi, fold_bin(a + j, A.II) * cs + hc, wv * bin_mass(pt, j == 0, zc, qc, zp, qp));
    zp = zc;
    qp = qc;
  }
  __syncwarp();
  unsigned longmask = __ballot_sync(FULL, is_long);
  while (longmask) {
    const int src = __ffs(longmask) - 1;
    longmask &= longmask - 1;
    const int l_a = __shfl_sync(FULL, a, src), l_n = __shfl_sync(FULL, n, src);
    const int l_hc = __shfl_sync(FULL, hc, src), l_b = __shfl_sync(FULL, bs, src), l_vi = __shfl_sync(FULL, vi, src);
    const float l_mu = __shfl_sync(FULL, mu, src), l_inv = __shfl_sync(FULL, inv_s, src);
    const float l_w = __shfl_sync(FULL, wv, src);
    float *l_row = A.tab + tab_row(A.W, B, l_vi, l_b);
    const bool l_tabled = l_n + 3 <= A.W;
    if (l_tabled && lane == 0) l_row[0] = 0.0f;
    float z_carry = 0.f, q_carry = 0.f;
    for (int p0 = 0; p0 <= l_n; p0 += 32) {
      const int pp = p0 + lane;
      const bool pt = pp < l_n;
      const float z = ((float)(l_a + pp) + 0.5f - l_mu) * l_inv;
      const float q = pt ? Fam<kFam>::tail(z) : 0.f;
      if (l_tabled && pp <= l_n) l_row[(size_t)(pp + 1) * ts] = pt ? (z <= 0.f ? q : 1.0f - q) : 1.0f;
      float zpv = __shfl_up_sync(FULL, z, 1), qpv = __shfl_up_sync(FULL, q, 1);
      if (lane == 0) { zpv = z_carry; qpv = q_carry; }
      if (hist && pp <= l_n)
        hist_add(hlo, hhi, fold_bin(l_a + pp, A.II) * cs + l_hc, l_w * bin_mass(pt, pp == 0, z, q, zpv, qpv));
      z_carry = __shfl_sync(FULL, z, 31);
      q_carry = __shfl_sync(FULL, q, 31);
    }
  }
  if (valid) {
    lo = min(lo, a);
    hi = max(hi, bw + 1);
  }
  return max(n, 0);
}

// Phase 1 for one segment (nodes s0..s1 of class c) and the restarts hrow RB1 ..
// (hrow + 1) RB1 - 1 of the group: every (node, restart) through p1_lane, then the
// touched span of bins flushed to the restarts' histograms U as exact integer adds.
// With RB1 = RG (the whole group's histogram fits), a warp takes one node with all
// its restarts, in two passes ordered by window length when RG > 32; otherwise rows
// of RB1 restarts, 32 / RB1 nodes per warp.
template <int kFam>
__device__ __forceinline__ void p1_segment(const FusedArgs &A, FusedShared &S, unsigned *hlo, int *map, int g, int p,
                                           int s0, int s1, int c, int hrow, bool hist) {
  constexpr int T = kFusedThreads;
  constexpr unsigned FULL = 0xffffffffu;
  const int tid = threadIdx.x, lane = tid & 31, RB1 = A.RB1, RG = A.RG, Dh = A.Dh, B = A.B;
  const bool whole = RB1 == RG;
  const int npw = whole ? 1 : 32 / RB1;
  unsigned *hhi = hlo + (size_t)Dh * RB1;
  if (hist)
    for (int i = tid; i < 2 * RB1 * Dh; i += T) hlo[i] = 0u;
  if (tid == 0) { S.lo = INT_MAX; S.hi = INT_MIN; S.next = 0; }
  __syncthreads();
  int lo = INT_MAX, hi = INT_MIN;
  for (;;) {
    int base = 0;
    if (lane == 0) base = atomicAdd(&S.next, npw);
    base = __shfl_sync(FULL, base, 0);
    if (base >= s1 - s0) break;
    if (whole && RG > 32) {
      // the node's restarts in the order of the previous iteration's windows (each
      // lane's state picked by shuffles from the two natural-order halves, loaded
      // together with the order), then the order of this iteration's windows for the
      // next phases
      const int vi = s0 + base;
      signed char *ow = A.ord + ((size_t)(g - A.g0) * A.V + vi) * 64;
      const int oo0 = ow[lane], oo1 = ow[32 + lane];
      const float2 xn0 = g * RG + lane < B ? A.xs[(size_t)vi * B + g * RG + lane] : make_float2(0.f, 1.f);
      const float2 xn1 = (lane + 32 < RG && g * RG + lane + 32 < B) ? A.xs[(size_t)vi * B + g * RG + lane + 32]
                                                                    : make_float2(0.f, 1.f);
      int kk0 = 0, kk1 = 0;
      for (int ps = 0; ps < 2; ++ps) {
        const int rl = ps ? oo1 : oo0, b = g * RG + rl, src = rl & 31;
        const float2 xa = make_float2(__shfl_sync(FULL, xn0.x, src), __shfl_sync(FULL, xn0.y, src));
        const float2 xb = make_float2(__shfl_sync(FULL, xn1.x, src), __shfl_sync(FULL, xn1.y, src));
        const bool present = rl >= 0 && b < B;
        const int kk = p1_lane<kFam>(A, S, hlo, RB1, vi, present ? rl : 0, present ? rl : 0, b, present,
                                     rl < 32 ? xa : xb, p, hist, lo, hi);
        if (ps) kk1 = kk; else kk0 = kk;
      }
      split_by_window(kk0, oo0, kk1, oo1, map);
      ow[lane] = (signed char)map[lane];
      ow[32 + lane] = (signed char)map[32 + lane];
    } else {
      const int vi = s0 + base + (whole ? 0 : lane / RB1);
      const int rl = whole ? lane : hrow * RB1 + lane % RB1, b = g * RG + rl;
      const bool present = vi < s1 && rl < RG && b < B;
      const float2 x = present ? A.xs[(size_t)vi * B + b] : make_float2(0.f, 1.f);
      p1_lane<kFam>(A, S, hlo, RB1, present ? vi : s0, present ? rl : 0, whole ? lane : lane % RB1, b, present, x, p,
                    hist, lo, hi);
    }
  }
  if (hist) {
    if (lo <= hi) {
      atomicMin(&S.lo, lo);
      atomicMax(&S.hi, hi);
    }
    __syncthreads();
    int flo = S.lo, fhi = S.hi;
    if (flo > fhi) {
      flo = 1;
      fhi = 0;
    } else if (A.II > 0) {
      if (fhi - flo + 1 >= A.II) {
        flo = 0;
        fhi = A.II - 1;
      } else {
        const int x0 = flo % A.II, y0 = fhi % A.II;
        if (x0 <= y0) { flo = x0; fhi = y0; } else { flo = 0; fhi = A.II - 1; }
      }
    }
    const int len = fhi - flo + 1;
    unsigned long long *U = reinterpret_cast<unsigned long long *>(A.U);
    // cells of restarts (whole group) or of the row hrow RB1 + 0..RB1-1
    for (int i = tid; i < RB1 * len; i += T) {
      const int cell = flo * RB1 + i, t = cell / RB1, rr = cell % RB1;
      const int rr_l = whole ? rr : hrow * RB1 + rr, bb = g * RG + rr_l;
      const unsigned long long val = ((unsigned long long)hhi[cell] << 16) + (unsigned long long)hlo[cell];
      if (rr_l < RG && bb < B && val) atomicAdd(U + ((size_t)(p * B + bb) * A.C + c) * Dh + t, val);
    }
  }
  __syncthreads();
}

template <int kFam, bool kCom>
__global__ void __launch_bounds__(kFusedThreads, 1) k_fused(const FusedArgs A) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ FusedShared S;
  constexpr int T = kFusedThreads;
  constexpr unsigned FULL = 0xffffffffu;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int RG = A.RG, RBp = A.RBp, Dh = A.Dh, B = A.B;
  const int npw = 32 / RBp, passes = RG > 32 ? 2 : 1, nsub = A.RB1 == RG ? 1 : (RG + A.RB1 - 1) / A.RB1;
  const int g = A.g0 + (int)(blockIdx.x / (unsigned)A.K), k = (int)(blockIdx.x % (unsigned)A.K);
  const unsigned on = A.terms;
  const bool dep = on & GAUS_DEP, com = on & GAUS_COM, rec = (on & GAUS_REC) && A.II > 0;
  const bool hist = on & (GAUS_RES_OBJ | GAUS_RES_VIOL);
  unsigned *hlo = reinterpret_cast<unsigned *>(smem);  // phase 1: [bin][restart], two halves
  float2 *stage = reinterpret_cast<float2 *>(smem);    // phase 2: [warp][point][lane]
  float2 *st = stage + (size_t)warp * kStage * 32 + lane;
  int *map = S.map[warp];

  // ---- prologue: per-restart scalars, the state of the block's own nodes ----
  if (tid < RG) {
    const int bb = g * RG + tid;
    for (int q = 0; q < GAUS_K; ++q) S.lam[tid][q] = bb < B ? A.lambda[(size_t)bb * GAUS_K + q] : 0.f;
    S.step[tid] = (A.adam && bb < B) ? A.step[bb] : 0;
  }
  for (int si = k; si < A.nseg; si += A.K) {
    const int s0 = __ldg(A.seg + 3 * si), s1 = __ldg(A.seg + 3 * si + 1);
    for (int q = tid; q < (s1 - s0) * RG; q += T) {
      const int vi = s0 + q / RG, bb = g * RG + q % RG;
      if (bb >= B) continue;
      const size_t ci = (size_t)__ldg(A.perm + vi) * B + bb, ii = (size_t)vi * B + bb;
      A.xs[ii] = make_float2(A.mu[ci], A.sg[ci]);
      if (A.adam) A.adm[ii] = make_float4(A.m_mu[ci], A.v_mu[ci], A.m_sg[ci], A.v_sg[ci]);
    }
  }
  __syncthreads();

  unsigned nbar = 0;
  bool alive = true;
  const bool prof = A.prof && tid == 0;
  auto stamp = [&](int it_, int q) {
    if (prof) A.prof[((size_t)it_ * gridDim.x + blockIdx.x) * 6 + q] = global_ns();
  };
  for (int it = 0; it < A.n_iters && alive; ++it) {
    const int p = it & 1;
    const bool last = it == A.n_iters - 1;
    stamp(it, 0);

    // ================= phase 1: windows, CDF table rows, usage histogram =================
    if (tid < kMaxRG) { S.ws[tid] = 0; S.wc[tid] = 0; }
    for (int si = k; si < A.nseg; si += A.K) {
      const int s0 = __ldg(A.seg + 3 * si), s1 = __ldg(A.seg + 3 * si + 1), c = __ldg(A.seg + 3 * si + 2);
      for (int h = 0; h < nsub; ++h) p1_segment<kFam>(A, S, hlo, map, g, p, s0, s1, c, h, hist);
    }
    __syncthreads();
    if (tid < RG && g * RG + tid < B && S.wc[tid]) {
      atomicAdd(&A.wst[2 * ((size_t)p * B + g * RG + tid)], (unsigned long long)S.ws[tid]);
      atomicAdd(&A.wst[2 * ((size_t)p * B + g * RG + tid) + 1], (unsigned long long)S.wc[tid]);
    }
    stamp(it, 1);
    nbar += A.K;
    alive = group_barrier(A.bar + g, nbar + A.bar_extra, A.abort_flag, &S.ok, A.bar_limit_ns);
    if (!alive) break;
    stamp(it, 2);

    // ================= phase 2: usage terms and adjoint; the own side of every edge =================
    // clear the other parity's accumulators (last read before the previous barrier,
    // next written after the following one)
    {
      const int q = 1 - p;
      const size_t per = (size_t)A.C * Dh, cells = (size_t)RG * per;
      for (size_t i = (size_t)k * T + tid; i < cells; i += (size_t)A.K * T) {
        const int bb = g * RG + (int)(i / per);
        if (bb < B) A.U[((size_t)q * B + bb) * per + i % per] = 0;
      }
      if (k == 0 && tid < RG && g * RG + tid < B) {
        const size_t bb = (size_t)q * B + g * RG + tid;
        A.fwd[3 * bb] = 0ull; A.fwd[3 * bb + 1] = 0ull; A.fwd[3 * bb + 2] = 0ull;
        A.wst[2 * bb] = 0ull; A.wst[2 * bb + 1] = 0ull;
        A.nonf[bb] = 0;
      }
    }
    if (tid < kMaxRG) { S.fw[0][tid] = 0ull; S.fw[1][tid] = 0ull; S.fw[2][tid] = 0ull; }
    if (tid == 0) { S.nlong = 0; S.qnext = 0; }
    __syncthreads();
    // one warp per restart of the group: usage terms and adjoint
    if (hist)
      for (int rr = k + A.K * warp; rr < RG; rr += A.K * kFusedWarps)
        if (g * RG + rr < B) restart_usage(A, g * RG + rr, p, S.lam[rr][GAUS_K_RES], S.m[warp], S.s[warp]);
    {
      // warp items claimed from the group's counter over all its nodes (balances the
      // blocks); the next claim is issued before the current item is worked on
      unsigned *ctr = A.ctr + (size_t)p * A.G + (g - A.g0);
      // (every lane takes part in the claim's atomic, lane 0 adding 1: the result is
      // waited for only where the next item starts, not at a branch's reconvergence)
      const unsigned one = lane == 0 ? 1u : 0u;
      int nxt = __shfl_sync(FULL, (int)atomicAdd(ctr, one), 0);
      for (;;) {
        const int base = nxt;
        if (base >= A.nchunk) break;
        const int nn = (int)atomicAdd(ctr, one);
        const int4 cd = __ldg(A.chunk + base);
        const int vi = cd.x, ch = cd.w;
        if (passes == 1) {
          const int rl = lane, b = g * RG + rl;
          const bool present = rl < RG && b < B;
          const float2 x = present ? A.xs[(size_t)vi * B + b] : make_float2(0.f, 1.f);
          p2_lane<kFam, kCom>(A, S, vi, ch, cd.y, cd.z, b, present ? rl : 0, present, x, st, dep, com, rec);
        } else {
          // the order of this iteration's windows and the two natural-order halves of
          // the node's state, loaded together; each pass's state picked by shuffles
          const signed char *o = A.ord + ((size_t)(g - A.g0) * A.V + vi) * 64;
          const int oo0 = o[lane], oo1 = o[32 + lane];
          const float2 xn0 = g * RG + lane < B ? A.xs[(size_t)vi * B + g * RG + lane] : make_float2(0.f, 1.f);
          const float2 xn1 = (lane + 32 < RG && g * RG + lane + 32 < B) ? A.xs[(size_t)vi * B + g * RG + lane + 32]
                                                                        : make_float2(0.f, 1.f);
          for (int ps = 0; ps < 2; ++ps) {
            const int rl = ps ? oo1 : oo0, b = g * RG + rl, src = rl & 31;
            const float2 xa = make_float2(__shfl_sync(FULL, xn0.x, src), __shfl_sync(FULL, xn0.y, src));
            const float2 xb = make_float2(__shfl_sync(FULL, xn1.x, src), __shfl_sync(FULL, xn1.y, src));
            const bool present = rl >= 0 && b < B;
            p2_lane<kFam, kCom>(A, S, vi, ch, cd.y, cd.z, b, present ? rl : 0, present, rl < 32 ? xa : xb, st, dep,
                                com, rec);
          }
        }
        nxt = __shfl_sync(FULL, nn, 0);
      }
    }
    // the block's queued long-window items, one per warp at a time
    __syncthreads();
    {
      const int nq = min(S.nlong, kLongQueue);
      for (;;) {
        int qi = 0;
        if (lane == 0) qi = atomicAdd(&S.qnext, 1);
        qi = __shfl_sync(FULL, qi, 0);
        if (qi >= nq) break;
        p2_long<kFam, kCom>(A, S, S.lq[qi], dep, com, rec);
      }
    }
    __syncthreads();
    if (tid < RG && g * RG + tid < B)
      for (int q = 0; q < 3; ++q)
        if (S.fw[q][tid]) atomicAdd(&A.fwd[3 * ((size_t)p * B + g * RG + tid) + q], S.fw[q][tid]);
    stamp(it, 3);
    nbar += A.K;
    alive = group_barrier(A.bar + g, nbar + A.bar_extra, A.abort_flag, &S.ok, A.bar_limit_ns);
    if (!alive) break;
    stamp(it, 4);

    // ================= phase 3: ALM coefficients, loss, gradient, Adam =================
    // the other parity's phase-2 counter: last used before the previous second
    // barrier, next used after the following first barrier
    if (k == 0 && tid == 0) A.ctr[(size_t)(1 - p) * A.G + (g - A.g0)] = 0u;
    if (tid < RG) {
      const int bb = g * RG + tid;
      if (bb < B) {
        const unsigned long long *fw3 = A.fwd + 3 * ((size_t)p * B + bb);
        const double vdep = (double)(float)((double)(long long)__ldcg(fw3 + 0) * kInvFix);
        const double lcom = (double)(float)((double)(long long)__ldcg(fw3 + 1) * kInvFix);
        const double vrec = (double)(float)((double)(long long)__ldcg(fw3 + 2) * kInvFix);
        const bool on_dep = on & GAUS_DEP, on_rv = on & GAUS_RES_VIOL, on_rec = on & GAUS_REC;
        const double lse = hist ? __ldcg(A.rstat + 2 * bb) : 0.0, vres = hist ? __ldcg(A.rstat + 2 * bb + 1) : 0.0;
        const double Vk[3] = {on_dep ? vdep : 0.0, on_rv ? vres : 0.0, on_rec ? vrec : 0.0};
        const bool actk[3] = {on_dep, on_rv, on_rec};
        S.coef[tid][0] = on_dep ? (float)((double)S.lam[tid][GAUS_K_DEP] + (double)A.rho * Vk[0]) : 0.f;
        S.coef[tid][1] = on_rec ? (float)((double)S.lam[tid][GAUS_K_REC] + (double)A.rho * Vk[2]) : 0.f;
        if (tid % A.K == k) {
          // the loss and terms of restart bb: by one block per restart, so that no
          // block's items wait for all of them
          double L = 0.0;
          if (on & GAUS_RES_OBJ) L += (double)A.w_res * lse;
          if (on & GAUS_COM) L += (double)A.alpha * lcom;
          for (int q = 0; q < 3; ++q)
            if (actk[q]) L += (double)S.lam[tid][q] * Vk[q] + 0.5 * (double)A.rho * Vk[q] * Vk[q];
          float *Tt = A.terms_out + (size_t)bb * GAUS_NT;
          Tt[GAUS_T_RES] = (on & GAUS_RES_OBJ) ? (float)lse : 0.f;
          Tt[GAUS_T_COM] = (on & GAUS_COM) ? (float)lcom : 0.f;
          Tt[GAUS_T_REG] = 0.f;
          Tt[GAUS_T_VDEP] = (float)Vk[0];
          Tt[GAUS_T_VRES] = (float)Vk[1];
          Tt[GAUS_T_VREC] = (float)Vk[2];
          A.loss[bb] = (float)L;
          A.status[bb] = __ldcg(A.nonf + (size_t)p * B + bb) ? GAUS_ENONFINITE : GAUS_OK;
        }
        if (A.adam) {
          for (int q = 0; q < 3; ++q)
            if (actk[q]) S.lam[tid][q] = (float)((double)S.lam[tid][q] + (double)A.rho * Vk[q]);
          const int stp = ++S.step[tid];
          S.coef[tid][2] = 1.0f / (1.0f - powf(A.beta1, (float)stp));
          S.coef[tid][3] = 1.0f / sqrtf(1.0f - powf(A.beta2, (float)stp));
        }
      }
    }
    if (tid == 0) S.next = 0;
    __syncthreads();
    for (int si = k; si < A.nseg; si += A.K) {
      const int s0 = __ldg(A.seg + 3 * si), s1 = __ldg(A.seg + 3 * si + 1);
      for (;;) {
        int base = 0;
        if (lane == 0) base = atomicAdd(&S.next, 1);
        base = __shfl_sync(FULL, base, 0);
        if (base >= s1 - s0) break;
        p3_node<kFam>(A, S, s0 + base, g, hist, rec, last);
      }
      __syncthreads();
      if (tid == 0) S.next = 0;
      __syncthreads();
    }
    stamp(it, 5);
  }

  // ---- epilogue: multipliers and steps (one block per group), or the abort ----
  if (k == 0 && tid < RG && g * RG + tid < B) {
    const int bb = g * RG + tid;
    if (alive && A.adam) {
      for (int q = 0; q < GAUS_K; ++q) A.lambda[(size_t)bb * GAUS_K + q] = S.lam[tid][q];
      A.step[bb] = S.step[tid];
    }
    if (!alive) A.status[bb] = GAUS_ETIMEOUT;
  }
}

}  // namespace gaus
