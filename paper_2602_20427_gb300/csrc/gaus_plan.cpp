// gaus_plan.cpp -- host planner of gaus_create: validation, topological order,
// ASAP/ALAP (App. A, Alg. 1 input), class-sorted node order and the flat arrays the
// kernels read.  Pure C++; no CUDA calls.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <numeric>
#include <string>
#include <vector>

#include "gaus_internal.h"

namespace gaus {

static gaus_status fail(std::string *err, gaus_status st, const char *msg) {
  if (err) *err = msg;
  return st;
}

gaus_status check_hparams(const gaus_hparams *hp, std::string *err) {
  if (!hp) return fail(err, GAUS_EINVAL, "hparams is NULL");
  const float pos[] = {hp->tau, hp->lr, hp->window_k, hp->sigma_min};
  for (float x : pos)
    if (!(x > 0.0f) || !std::isfinite(x)) return fail(err, GAUS_EINVAL, "tau, lr, window_k and sigma_min must be finite and > 0");
  const float nonneg[] = {hp->rho, hp->alpha, hp->w_res, hp->w_mem, hp->eps, hp->lambda0};
  for (float x : nonneg)
    if (!(x >= 0.0f) || !std::isfinite(x)) return fail(err, GAUS_EINVAL, "rho, alpha, w_res, w_mem, eps, lambda0 must be finite and >= 0");
  if (!(hp->beta1 >= 0.0f && hp->beta1 < 1.0f && hp->beta2 >= 0.0f && hp->beta2 < 1.0f))
    return fail(err, GAUS_EINVAL, "Adam betas must lie in [0, 1)");
  if (hp->terms & ~127u) return fail(err, GAUS_EINVAL, "unknown term bits");
  if ((hp->terms & GAUS_DEP) && (hp->terms & GAUS_DEP_CF))
    return fail(err, GAUS_EINVAL, "GAUS_DEP and GAUS_DEP_CF are two forms of one constraint: choose one");
  if ((hp->terms & GAUS_DEP_CF) && hp->family != GAUS_GAUSSIAN)
    return fail(err, GAUS_EINVAL, "GAUS_DEP_CF is the normal's closed form: it needs family GAUS_GAUSSIAN");
  if (hp->family < GAUS_GAUSSIAN || hp->family > GAUS_CAUCHY) return fail(err, GAUS_EINVAL, "unknown CDF family");
  return GAUS_OK;
}

// Window half-width (in sigma) of a family: the point beyond which its tail mass
// equals the normal's beyond window_k, Q = Phi(-window_k), and at least window_k.  Logistic
// (s = sigma sqrt(3)/pi): Q = 1 / (1 + e^{k pi/sqrt 3}); Laplace (b = sigma/sqrt 2):
// Q = e^{-k sqrt 2} / 2; Cauchy (gamma = sigma sqrt(2 ln 2)):
// Q = atan(gamma / (k sigma)) / pi.  Capped at FLT_MAX (a window of every step).
float family_window_k(float window_k, int family) {
  if (family == GAUS_GAUSSIAN) return window_k;
  const double q = 0.5 * std::erfc((double)window_k / std::sqrt(2.0));
  const double pi = 3.14159265358979323846;
  double k = HUGE_VAL;
  if (q > 0.0) {
    if (family == GAUS_LOGISTIC) k = std::sqrt(3.0) / pi * std::log(1.0 / q - 1.0);
    else if (family == GAUS_LAPLACE) k = std::log(0.5 / q) / std::sqrt(2.0);
    else k = std::sqrt(2.0 * std::log(2.0)) / std::tan(pi * q);
  }
  return (std::isfinite(k) && k < 3.0e38) ? (float)std::max(k, (double)window_k) : 3.4028234663852886e38f;
}

static bool valid_csr(int V, int E, const int32_t *ptr, const int32_t *idx) {
  if (!ptr || (E > 0 && !idx)) return false;
  if (ptr[0] != 0 || ptr[V] != E) return false;
  for (int v = 0; v < V; ++v)
    if (ptr[v + 1] < ptr[v]) return false;
  for (int e = 0; e < E; ++e)
    if (idx[e] < 0 || idx[e] >= V) return false;
  return true;
}

// Segments: contiguous internal nodes of one class, sized so that the per-node
// kernels launch about target_blocks blocks over all restart groups of RB restarts.
void plan_segments(Plan &P, int target_blocks, int RB) {
  const int V = P.V, C = P.C;
  P.seg.clear();
  int G = (P.B + RB - 1) / RB;
  long want = std::max(1L, (long)target_blocks / G);
  int seglen = (int)std::max(1L, ((long)V + want - 1) / want);
  // at least one row of nodes per block pass; and few enough nodes that the
  // 16-bit halves of the shared-memory usage histogram cannot overflow:
  // segment length * max demand * ceil(D / Dh) * 2^16 < 2^32
  seglen = std::max(seglen, std::max(1, kFwdThreads / RB));
  int maxw = 1;
  for (int v = 0; v < V; ++v) maxw = std::max(maxw, P.c_dem[v]);
  const long folds = (P.D + P.Dh - 1) / P.Dh;
  const long cap = std::max(1L, 32768L / ((long)maxw * folds));
  seglen = (int)std::max(1L, std::min<long>(seglen, cap));
  // whole rows of the block: warps then claim equal shares
  const int rows = kFwdThreads / RB;
  if (seglen > rows) seglen = (seglen + rows - 1) / rows * rows;
  if (seglen > cap) seglen = (int)std::max(1L, cap >= rows ? cap - cap % rows : cap);
  P.cls_seg_ptr.assign(C + 1, 0);
  int i0 = 0;
  for (int c = 0; c < C; ++c) {
    int i1 = i0;
    while (i1 < V && P.cls[i1] == c) ++i1;
    for (int s = i0; s < i1; s += seglen) {
      P.seg.push_back(s);
      P.seg.push_back(std::min(i1, s + seglen));
      P.seg.push_back(c);
    }
    P.cls_seg_ptr[c + 1] = (int)P.seg.size() / 3;
    i0 = i1;
  }
  P.nseg = (int)P.seg.size() / 3;
}

void plan_fused_segments(Plan &P, int target_per_group, int RB) {
  const int V = P.V, C = P.C;
  const int target = std::max(1, target_per_group);
  // the 16-bit halves of the shared-memory usage histogram cannot overflow:
  // segment length * max demand * ceil(D / Dh) * 2^16 < 2^32
  int maxw = 1;
  for (int v = 0; v < V; ++v) maxw = std::max(maxw, P.c_dem[v]);
  const long folds = (P.D + P.Dh - 1) / P.Dh;
  const long cap = std::max(1L, 32768L / ((long)maxw * folds));
  // estimated work of each node in phases 1 and 3: a node without predecessors starts
  // at the horizon's lower edge, where the window's clipped mass leaves sigma little
  // gradient, and keeps a wider window through a run (about five times the others'
  // points late in a run of the logic-network workload)
  std::vector<long> wt(V);
  long total = 0;
  for (int i = 0; i < V; ++i) {
    wt[i] = P.in_ptr[i + 1] > P.in_ptr[i] ? 1 : 5;
    total += wt[i];
  }
  std::vector<int> ncls(C, 0);
  for (int i = 0; i < V; ++i) ncls[P.cls[i]]++;
  // segments of about total / target weight each, cut at class boundaries and at the
  // overflow cap; the budget grows until the segments fit one block each (unless the
  // cap forces more)
  const int npw = std::max(1, 32 / RB);
  auto cut = [&](long budget, std::vector<int32_t> *out) {
    long nseg = 0;
    int i0 = 0;
    for (int c = 0; c < C; ++c) {
      const int i1 = i0 + ncls[c];
      int s = i0;
      while (s < i1) {
        long w = 0;
        int e = s;
        while (e < i1 && (e == s || (w + wt[e] <= budget && e - s < cap))) w += wt[e++];
        // whole warp rows where the budget allows
        if (e < i1 && e - s > npw) e = s + std::max(npw, (e - s) / npw * npw);
        if (out) { out->push_back(s); out->push_back(e); out->push_back(c); }
        ++nseg;
        s = e;
      }
      i0 = i1;
    }
    return nseg;
  };
  long budget = std::max(1L, (total + target - 1) / target);
  while (cut(budget, nullptr) > target && budget < total) budget += std::max(1L, budget / 64);
  P.fseg.clear();
  cut(budget, &P.fseg);
  P.nfseg = (int)P.fseg.size() / 3;
}

gaus_status plan_problem(const gaus_problem *p, int target_blocks, Plan *out, std::string *err) {
  if (!p) return fail(err, GAUS_EINVAL, "problem is NULL");
  const int V = p->V, E = p->E, C = p->C, NB = p->n_back;
  if (V < 1 || E < 0 || NB < 0) return fail(err, GAUS_EINVAL, "V >= 1, E >= 0, n_back >= 0 required");
  if (C < 1 || C > kMaxClasses) return fail(err, GAUS_EINVAL, "C must lie in 1..16");
  if (p->D < 1 || p->II < 0 || p->B < 1) return fail(err, GAUS_EINVAL, "D >= 1, II >= 0, B >= 1 required");
  if ((int64_t)V * p->B >= (int64_t)1 << 31 || (int64_t)V * p->D >= (int64_t)1 << 31)
    return fail(err, GAUS_EINVAL, "V * B and V * D must stay below 2^31");
  if (p->D > 65536) return fail(err, GAUS_EINVAL, "D must be <= 65536");
  if (!valid_csr(V, E, p->succ_ptr, p->succ_idx)) return fail(err, GAUS_EINVAL, "invalid CSR (succ_ptr/succ_idx)");
  if (!valid_csr(V, E, p->pred_ptr, p->pred_idx)) return fail(err, GAUS_EINVAL, "invalid CSC (pred_ptr/pred_idx)");
  if (!p->latency || !p->res_class || !p->limit) return fail(err, GAUS_EINVAL, "latency, res_class and limit are required");
  if (NB > 0 && (!p->back_src || !p->back_dst || !p->back_dist)) return fail(err, GAUS_EINVAL, "back-edge arrays missing");

  // edge list from CSR; CSC must describe the same set; no duplicates or self loops
  std::vector<int64_t> ecsr(E), ecsc(E);
  for (int u = 0; u < V; ++u)
    for (int q = p->succ_ptr[u]; q < p->succ_ptr[u + 1]; ++q) {
      if (p->succ_idx[q] == u) return fail(err, GAUS_ECYCLE, "self loop");
      ecsr[q] = (int64_t)u * V + p->succ_idx[q];
    }
  for (int v = 0; v < V; ++v)
    for (int q = p->pred_ptr[v]; q < p->pred_ptr[v + 1]; ++q) ecsc[q] = (int64_t)p->pred_idx[q] * V + v;
  std::sort(ecsr.begin(), ecsr.end());
  std::sort(ecsc.begin(), ecsc.end());
  if (ecsr != ecsc) return fail(err, GAUS_EINVAL, "CSR and CSC describe different edges");
  for (int e = 1; e < E; ++e)
    if (ecsr[e] == ecsr[e - 1]) return fail(err, GAUS_EINVAL, "duplicate edge");

  Plan &P = *out;
  P = Plan();
  P.V = V; P.E = E; P.NB = NB; P.C = C; P.D = p->D; P.II = p->II; P.B = p->B;
  P.Dh = p->II > 0 ? p->II : p->D;
  for (int v = 0; v < V; ++v) {
    if (p->latency[v] < 0 || p->latency[v] > p->D) return fail(err, GAUS_EINVAL, "latency must lie in 0..D");
    if (p->res_class[v] < 0 || p->res_class[v] >= C) return fail(err, GAUS_EINVAL, "res_class out of range");
    if (p->demand && p->demand[v] < 0) return fail(err, GAUS_EINVAL, "demand must be >= 0");
    if (p->bits && p->bits[v] < 0) return fail(err, GAUS_EINVAL, "bits must be >= 0");
  }
  for (int c = 0; c < C; ++c)
    if (!(p->limit[c] >= 0.0f)) return fail(err, GAUS_EINVAL, "limit must be >= 0 or INFINITY");
  for (int q = 0; q < NB; ++q) {
    if (p->back_src[q] < 0 || p->back_src[q] >= V || p->back_dst[q] < 0 || p->back_dst[q] >= V)
      return fail(err, GAUS_EINVAL, "back edge endpoint out of range");
    if (p->back_dist[q] < 1) return fail(err, GAUS_EINVAL, "back edge distance must be >= 1");
  }

  // Kahn's algorithm and topological levels
  std::vector<int32_t> indeg(V), order;
  order.reserve(V);
  for (int v = 0; v < V; ++v) indeg[v] = p->pred_ptr[v + 1] - p->pred_ptr[v];
  for (int v = 0; v < V; ++v)
    if (!indeg[v]) order.push_back(v);
  P.level.assign(V, 0);
  for (size_t h = 0; h < order.size(); ++h) {
    int u = order[h];
    for (int q = p->succ_ptr[u]; q < p->succ_ptr[u + 1]; ++q) {
      int w = p->succ_idx[q];
      P.level[w] = std::max(P.level[w], P.level[u] + 1);
      if (--indeg[w] == 0) order.push_back(w);
    }
  }
  if ((int)order.size() != V) return fail(err, GAUS_ECYCLE, "the dependency graph has a cycle");

  // ASAP_v = max_u ASAP_u + Lat(u); CP = max ASAP_v + Lat(v); ALAP_v = min(D - Lat(v), min_w ALAP_w - Lat(v))
  P.asap.assign(V, 0);
  for (int u : order)
    for (int q = p->succ_ptr[u]; q < p->succ_ptr[u + 1]; ++q) {
      int w = p->succ_idx[q];
      P.asap[w] = std::max(P.asap[w], P.asap[u] + p->latency[u]);
    }
  P.cp = 0;
  for (int v = 0; v < V; ++v) P.cp = std::max(P.cp, P.asap[v] + p->latency[v]);
  if (P.cp > p->D) return fail(err, GAUS_EHORIZON, "critical path longer than the horizon D");
  P.alap.assign(V, 0);
  for (int h = V - 1; h >= 0; --h) {
    int v = order[h];
    int a = p->D - p->latency[v];
    for (int q = p->succ_ptr[v]; q < p->succ_ptr[v + 1]; ++q) a = std::min(a, P.alap[p->succ_idx[q]] - p->latency[v]);
    P.alap[v] = a;
  }

  // caller-order attributes
  P.c_lat.assign(p->latency, p->latency + V);
  P.c_cls.assign(p->res_class, p->res_class + V);
  P.c_dem.resize(V);
  P.c_bits.resize(V);
  for (int v = 0; v < V; ++v) {
    P.c_dem[v] = p->demand ? p->demand[v] : 1;
    P.c_bits[v] = p->bits ? p->bits[v] : 1;
  }
  P.limit.assign(p->limit, p->limit + C);
  P.e_src.resize(E);
  P.e_dst.resize(E);
  for (int u = 0; u < V; ++u)
    for (int q = p->succ_ptr[u]; q < p->succ_ptr[u + 1]; ++q) { P.e_src[q] = u; P.e_dst[q] = p->succ_idx[q]; }
  P.b_src.assign(p->back_src, p->back_src + NB);
  P.b_dst.assign(p->back_dst, p->back_dst + NB);
  P.b_dist.assign(p->back_dist, p->back_dist + NB);

  // internal order: by class, then topological level, then caller id
  P.perm.resize(V);
  std::iota(P.perm.begin(), P.perm.end(), 0);
  std::stable_sort(P.perm.begin(), P.perm.end(), [&](int a, int b) {
    if (P.c_cls[a] != P.c_cls[b]) return P.c_cls[a] < P.c_cls[b];
    return P.level[a] < P.level[b];
  });
  P.inv.resize(V);
  for (int i = 0; i < V; ++i) P.inv[P.perm[i]] = i;
  P.w.resize(V); P.bits.resize(V); P.lat.resize(V); P.cls.resize(V);
  for (int i = 0; i < V; ++i) {
    int v = P.perm[i];
    P.w[i] = (float)P.c_dem[v];
    P.bits[i] = (float)P.c_bits[v];
    P.lat[i] = P.c_lat[v];
    P.cls[i] = P.c_cls[v];
  }
  // internal CSC / CSR (neighbours stored by caller id)
  P.in_ptr.assign(V + 1, 0);
  P.out_ptr.assign(V + 1, 0);
  for (int i = 0; i < V; ++i) {
    int v = P.perm[i];
    P.in_ptr[i + 1] = P.in_ptr[i] + (p->pred_ptr[v + 1] - p->pred_ptr[v]);
    P.out_ptr[i + 1] = P.out_ptr[i] + (p->succ_ptr[v + 1] - p->succ_ptr[v]);
  }
  P.in_src.resize(E); P.in_lat.resize(E); P.out_dst.resize(E);
  for (int i = 0; i < V; ++i) {
    int v = P.perm[i];
    int o = P.in_ptr[i];
    for (int q = p->pred_ptr[v]; q < p->pred_ptr[v + 1]; ++q, ++o) {
      P.in_src[o] = p->pred_idx[q];
      P.in_lat[o] = p->latency[p->pred_idx[q]];
    }
    o = P.out_ptr[i];
    for (int q = p->succ_ptr[v]; q < p->succ_ptr[v + 1]; ++q, ++o) P.out_dst[o] = p->succ_idx[q];
  }
  // CSC position of every in-edge -> CSR position of the same edge in its
  // producer's out-list (per-edge slots written by producers, read by consumers)
  {
    std::vector<int64_t> key(E);
    std::vector<int32_t> pos(E);
    for (int i = 0; i < V; ++i)
      for (int o = P.out_ptr[i]; o < P.out_ptr[i + 1]; ++o) {
        key[o] = (int64_t)P.perm[i] * V + P.out_dst[o];
        pos[o] = o;
      }
    std::vector<int32_t> idx(E);
    std::iota(idx.begin(), idx.end(), 0);
    std::sort(idx.begin(), idx.end(), [&](int x, int y) { return key[x] < key[y]; });
    P.in_eslot.resize(E);
    for (int i = 0; i < V; ++i)
      for (int e = P.in_ptr[i]; e < P.in_ptr[i + 1]; ++e) {
        const int64_t k = (int64_t)P.in_src[e] * V + P.perm[i];
        int lo = 0, hi = E - 1;
        while (lo < hi) {
          const int mid = (lo + hi) / 2;
          if (key[idx[mid]] < k) lo = mid + 1; else hi = mid;
        }
        P.in_eslot[e] = pos[idx[lo]];
      }
  }
  // back edges: shift = Lat(j) - k II (a back edge acts as a dependency with that latency)
  P.bin_ptr.assign(V + 1, 0);
  P.bout_ptr.assign(V + 1, 0);
  for (int q = 0; q < NB; ++q) {
    P.bin_ptr[P.inv[p->back_dst[q]] + 1]++;
    P.bout_ptr[P.inv[p->back_src[q]] + 1]++;
  }
  for (int i = 0; i < V; ++i) { P.bin_ptr[i + 1] += P.bin_ptr[i]; P.bout_ptr[i + 1] += P.bout_ptr[i]; }
  P.bin_src.resize(NB); P.bin_shift.resize(NB); P.bout_dst.resize(NB); P.bout_shift.resize(NB);
  P.bin_eslot.resize(NB);
  {
    std::vector<int32_t> fi(P.bin_ptr.begin(), P.bin_ptr.end() - 1), fo(P.bout_ptr.begin(), P.bout_ptr.end() - 1);
    for (int q = 0; q < NB; ++q) {
      int j = p->back_src[q], i = p->back_dst[q];
      int shift = p->latency[j] - p->back_dist[q] * p->II;
      int a = fi[P.inv[i]]++;
      P.bin_src[a] = j; P.bin_shift[a] = shift;
      int b = fo[P.inv[j]]++;
      P.bout_dst[b] = i; P.bout_shift[b] = shift;
      P.bin_eslot[a] = b;
    }
  }
  // incident edges by internal id (fused kernel)
  P.fin.resize(2 * (size_t)E);
  P.fout.resize(2 * (size_t)E);
  for (int e = 0; e < E; ++e) {
    P.fin[2 * (size_t)e] = P.inv[P.in_src[e]];
    P.fin[2 * (size_t)e + 1] = P.in_lat[e];
  }
  for (int i = 0; i < V; ++i)
    for (int o = P.out_ptr[i]; o < P.out_ptr[i + 1]; ++o) {
      P.fout[2 * (size_t)o] = P.inv[P.out_dst[o]];
      P.fout[2 * (size_t)o + 1] = P.lat[i];
    }
  P.fbin.resize(2 * (size_t)NB);
  P.fbout.resize(2 * (size_t)NB);
  for (int q = 0; q < NB; ++q) {
    P.fbin[2 * (size_t)q] = P.inv[P.bin_src[q]];
    P.fbin[2 * (size_t)q + 1] = P.bin_shift[q];
    P.fbout[2 * (size_t)q] = P.inv[P.bout_dst[q]];
    P.fbout[2 * (size_t)q + 1] = P.bout_shift[q];
  }
  // the fused kernel's edge phase: incident-edge lists, chunks, claim order (the
  // chunks with the most edges first, so that the last items claimed are short)
  {
    P.finc.clear();
    P.chunk.clear();
    P.cptr.assign(V + 1, 0);
    auto add = [&](int nb, int L, int kind) {
      P.finc.push_back(nb); P.finc.push_back(L); P.finc.push_back(kind); P.finc.push_back(0);
    };
    for (int i = 0; i < V; ++i) {
      const int first = (int)P.finc.size() / 4;
      for (int e = P.in_ptr[i]; e < P.in_ptr[i + 1]; ++e) add(P.inv[P.in_src[e]], P.in_lat[e], 0);
      for (int o = P.out_ptr[i]; o < P.out_ptr[i + 1]; ++o) add(P.inv[P.out_dst[o]], P.lat[i], 1);
      for (int q = P.bin_ptr[i]; q < P.bin_ptr[i + 1]; ++q) add(P.inv[P.bin_src[q]], P.bin_shift[q], 2);
      for (int q = P.bout_ptr[i]; q < P.bout_ptr[i + 1]; ++q) add(P.inv[P.bout_dst[q]], P.bout_shift[q], 3);
      const int last = (int)P.finc.size() / 4;
      for (int c = first; c < last; c += kChunkEdges) {
        P.chunk.push_back(i); P.chunk.push_back(c); P.chunk.push_back(std::min(kChunkEdges, last - c));
        P.chunk.push_back(0);
      }
      P.cptr[i + 1] = (int)P.chunk.size() / 4;
    }
    P.nchunk = (int)P.chunk.size() / 4;
    P.p2ord.resize(P.nchunk);
    std::iota(P.p2ord.begin(), P.p2ord.end(), 0);
    std::stable_sort(P.p2ord.begin(), P.p2ord.end(),
                     [&](int a, int b) { return P.chunk[4 * (size_t)a + 2] > P.chunk[4 * (size_t)b + 2]; });
    // descriptors in claim order, with the chunk index (where its partials go)
    std::vector<int32_t> claim(P.chunk.size());
    for (int q = 0; q < P.nchunk; ++q) {
      const int c = P.p2ord[q];
      for (int k = 0; k < 3; ++k) claim[4 * (size_t)q + k] = P.chunk[4 * (size_t)c + k];
      claim[4 * (size_t)q + 3] = c;
    }
    P.chunk.swap(claim);
  }
  P.unit_lat = 1;
  for (int i = 0; i < V; ++i)
    if (P.out_ptr[i + 1] > P.out_ptr[i] && P.lat[i] != 1) P.unit_lat = 0;
  // edge list of the edge pass: forward edges in internal CSR order (producer,
  // consumer, Lat(producer), kind | consumer position << 1), then back edges in
  // producer order (j, i, shift, ...).  kind: 0 forward, 1 back; the consumer
  // position is the edge's place in its consumer's CSC (forward) or bin (back)
  // list, where the consumer's partial is written.
  {
    std::vector<int32_t> csc_of(E), bin_of(NB);
    for (int c = 0; c < E; ++c) csc_of[P.in_eslot[c]] = c;
    for (int a = 0; a < NB; ++a) bin_of[P.bin_eslot[a]] = a;
    P.ed.resize(4 * ((size_t)E + NB));
    for (int i = 0; i < V; ++i)
      for (int o = P.out_ptr[i]; o < P.out_ptr[i + 1]; ++o) {
        P.ed[4 * (size_t)o + 0] = P.perm[i];
        P.ed[4 * (size_t)o + 1] = P.out_dst[o];
        P.ed[4 * (size_t)o + 2] = P.lat[i];
        P.ed[4 * (size_t)o + 3] = csc_of[o] << 1;
      }
    for (int i = 0; i < V; ++i)
      for (int q = P.bout_ptr[i]; q < P.bout_ptr[i + 1]; ++q) {
        const size_t k = 4 * ((size_t)E + q);
        P.ed[k + 0] = P.perm[i];
        P.ed[k + 1] = P.bout_dst[q];
        P.ed[k + 2] = P.bout_shift[q];
        P.ed[k + 3] = 1 | (bin_of[q] << 1);
      }
  }
  // caller-order CSC / CSR / back edges for the integer kernels
  P.cpred_ptr.assign(p->pred_ptr, p->pred_ptr + V + 1);
  P.cpred_src.assign(p->pred_idx, p->pred_idx + E);
  P.csucc_ptr.assign(p->succ_ptr, p->succ_ptr + V + 1);
  P.csucc_dst.assign(p->succ_idx, p->succ_idx + E);
  P.cback_ptr.assign(V + 1, 0);
  for (int q = 0; q < NB; ++q) P.cback_ptr[p->back_dst[q] + 1]++;
  for (int v = 0; v < V; ++v) P.cback_ptr[v + 1] += P.cback_ptr[v];
  P.cback_src.resize(NB); P.cback_shift.resize(NB);
  {
    std::vector<int32_t> f(P.cback_ptr.begin(), P.cback_ptr.end() - 1);
    for (int q = 0; q < NB; ++q) {
      int a = f[p->back_dst[q]]++;
      P.cback_src[a] = p->back_src[q];
      P.cback_shift[a] = p->latency[p->back_src[q]] - p->back_dist[q] * p->II;
    }
  }
  // nodes by topological level (caller ids)
  P.nlvl = 0;
  for (int v = 0; v < V; ++v) P.nlvl = std::max(P.nlvl, P.level[v] + 1);
  P.lvl_ptr.assign(P.nlvl + 1, 0);
  for (int v = 0; v < V; ++v) P.lvl_ptr[P.level[v] + 1]++;
  for (int l = 0; l < P.nlvl; ++l) P.lvl_ptr[l + 1] += P.lvl_ptr[l];
  P.lvl_nodes.resize(V);
  {
    std::vector<int32_t> f(P.lvl_ptr.begin(), P.lvl_ptr.end() - 1);
    for (int v = 0; v < V; ++v) P.lvl_nodes[f[P.level[v]]++] = v;
  }
  P.lq_ptr.assign(V + 1, 0);
  P.lq_src.clear();
  P.lq_lat.clear();
  for (int q = 0; q < V; ++q) {
    const int v = P.lvl_nodes[q];
    for (int e = p->pred_ptr[v]; e < p->pred_ptr[v + 1]; ++e) {
      P.lq_src.push_back(p->pred_idx[e]);
      P.lq_lat.push_back(p->latency[p->pred_idx[e]]);
    }
    P.lq_ptr[q + 1] = (int32_t)P.lq_src.size();
  }

  int RB = 1;
  while (RB < P.B && RB < kMaxRB) RB <<= 1;
  plan_segments(P, target_blocks, RB);
  return GAUS_OK;
}

}  // namespace gaus
