/*
 * gaus_oracle.c -- fp64 CPU oracle for GauS (arXiv 2602.20427).
 *
 * TEST INFRASTRUCTURE.  Only the tests, the smoke check and the CPU-baseline leg
 * of the benchmark call this code; the product path never does.  It shares no
 * code with the CUDA library.
 *
 * Every expectation is evaluated over the whole horizon d = 0..D-1 (no window)
 * as the double sum the paper writes, and the gradient is the derivative of
 * that double sum taken term by term, then chained through the bin masses of
 * Eq. round to (mu, sigma).  Nothing is blocked, fused or reordered.
 *
 * Readings of the paper used here (the paper is silent or ambiguous):
 *  - Dependency edge u -> v with latency Lat(u) is violated iff s_v < s_u + Lat(u)
 *    (Sec. 2.1 Dep); Eq. dep is the Lat = 0 case (d_j < d_i).
 *  - Back edge (j -> i, k) is violated iff s_i + k*II < s_j + Lat(j) (Sec. 2.1
 *    Rec), summed over every d_i >= 0 (App. B.3 starts at d_i = 1).
 *  - Usage is counted at the start step only (Sec. 2.1 Res), one histogram per
 *    resource class c with limit R_c; classes with R_c = inf add no violation.
 *  - ReLU'(0) = 0.
 *  - A leaf's successor is a sink fixed at step D (Sec. 2.1 footnote), so its
 *    output is live until the end of the horizon.
 *  - Modulo folds use k >= 0 while t + k*II <= D-1 (App. B.3).
 *  - Alg. 1 / Alg. 2 use +Lat(u) where the paper writes +1; Alg. 2's lower
 *    bound for a node without predecessors is 0.
 */
#include "gaus_oracle.h"

#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

double orc_Phi(double z) { return 0.5 * erfc(-z / sqrt(2.0)); }
double orc_phi(double z) { return exp(-0.5 * z * z) / sqrt(2.0 * M_PI); }

/* App. D: the family's standard CDF replaces Phi in Eq. round, its scale matched
 * to N(mu, sigma^2) so that one sigma means a comparable spread:
 *   logistic  s     = sigma sqrt(3) / pi   (same variance)
 *   Laplace   b     = sigma / sqrt(2)      (same variance)
 *   Cauchy    gamma = sigma sqrt(2 ln 2)   (same full width at half maximum)
 * In z = (x - mu) / sigma each family is G(z / c) for its standard CDF G and
 * c = s / sigma, b / sigma or gamma / sigma; the density in z is g(z / c) / c. */
static double family_scale(int32_t fam) {
  switch (fam) {
    case ORC_LOGISTIC: return sqrt(3.0) / M_PI;
    case ORC_LAPLACE: return 1.0 / sqrt(2.0);
    case ORC_CAUCHY: return sqrt(2.0 * log(2.0));
    default: return 1.0;
  }
}

double orc_F(int32_t fam, double z) {
  const double y = z / family_scale(fam);
  switch (fam) {
    case ORC_LOGISTIC: {  /* 1 / (1 + e^-y), written with e^-|y| so that no exp overflows */
      const double e = exp(-fabs(y));
      return y >= 0.0 ? 1.0 / (1.0 + e) : e / (1.0 + e);
    }
    case ORC_LAPLACE:     /* 1/2 e^y below the centre, 1 - 1/2 e^-y above it */
      return y < 0.0 ? 0.5 * exp(y) : 1.0 - 0.5 * exp(-y);
    case ORC_CAUCHY:      /* 1/2 + atan(y) / pi */
      return 0.5 + atan(y) / M_PI;
    default:
      return orc_Phi(z);
  }
}

double orc_f(int32_t fam, double z) {
  const double c = family_scale(fam), y = z / c;
  switch (fam) {
    case ORC_LOGISTIC: {  /* e^-y / (1 + e^-y)^2, even in y */
      const double e = exp(-fabs(y));
      return e / ((1.0 + e) * (1.0 + e)) / c;
    }
    case ORC_LAPLACE: return 0.5 * exp(-fabs(y)) / c;
    case ORC_CAUCHY: return 1.0 / (M_PI * (1.0 + y * y)) / c;
    default: return orc_phi(z);
  }
}

/* Eq. round: P^d = F((d + 1/2 - mu)/sigma) - F((d - 1/2 - mu)/sigma), F = Phi for
 * the Gaussian (App. D for the other families), the lower limit of bin 0 at -inf
 * and the upper limit of bin D-1 at +inf (Sec. 3.2 footnote).  Also returns
 * dP/dmu and dP/dsigma when asked. */
static void bin_masses_and_derivs(int32_t D, int32_t fam, double mu, double sigma, double *P,
                                  double *dPdmu, double *dPdsig) {
  for (int32_t d = 0; d < D; ++d) {
    double z_lo = (d - 0.5 - mu) / sigma, z_hi = (d + 0.5 - mu) / sigma;
    double F_lo = (d == 0) ? 0.0 : orc_F(fam, z_lo);
    double F_hi = (d == D - 1) ? 1.0 : orc_F(fam, z_hi);
    /* dF((x - mu)/sigma)/dmu = -f(z)/sigma ; d/dsigma = -z f(z)/sigma */
    double f_lo = (d == 0) ? 0.0 : orc_f(fam, z_lo);
    double f_hi = (d == D - 1) ? 0.0 : orc_f(fam, z_hi);
    double zf_lo = (d == 0) ? 0.0 : z_lo * f_lo;
    double zf_hi = (d == D - 1) ? 0.0 : z_hi * f_hi;
    /* above the centre the mass is taken from the upper tails, F(-z_lo) - F(-z_hi)
     * (every family is symmetric), so that far-tail bins keep relative accuracy */
    if (d > 0 && z_lo >= 0.0)
      P[d] = orc_F(fam, -z_lo) - ((d == D - 1) ? 0.0 : orc_F(fam, -z_hi));
    else
      P[d] = F_hi - F_lo;
    if (dPdmu) dPdmu[d] = -(f_hi - f_lo) / sigma;
    if (dPdsig) dPdsig[d] = -(zf_hi - zf_lo) / sigma;
  }
}

void orc_bin_masses(int32_t D, int32_t fam, double mu, double sigma, double *P) {
  bin_masses_and_derivs(D, fam, mu, sigma, P, NULL, NULL);
}

static int32_t fold_len(const orc_problem *p) { return p->II > 0 ? p->II : p->D; }
static int32_t fold_of(const orc_problem *p, int32_t d) { return p->II > 0 ? d % p->II : d; }

/* Successor and predecessor lists of the edge list (counting sort); a plain
 * data structure so that per-node loops do not rescan every edge. */
typedef struct { int32_t *ptr, *idx; } adj_list;

static adj_list make_adj(int32_t V, int32_t E, const int32_t *key, const int32_t *val) {
  adj_list a;
  a.ptr = calloc((size_t)V + 1, sizeof(int32_t));
  a.idx = malloc(sizeof(int32_t) * ((size_t)E + 1));
  for (int32_t e = 0; e < E; ++e) a.ptr[key[e] + 1]++;
  for (int32_t v = 0; v < V; ++v) a.ptr[v + 1] += a.ptr[v];
  int32_t *fill = malloc(sizeof(int32_t) * ((size_t)V + 1));
  memcpy(fill, a.ptr, sizeof(int32_t) * ((size_t)V + 1));
  for (int32_t e = 0; e < E; ++e) a.idx[fill[key[e]]++] = val[e];
  free(fill);
  return a;
}
static void free_adj(adj_list a) { free(a.ptr); free(a.idx); }

int orc_asap_alap(int32_t V, int32_t E, const int32_t *src, const int32_t *dst,
                  const int32_t *lat, int32_t D, int32_t *order, int32_t *asap,
                  int32_t *alap, int32_t *cp) {
  adj_list succ = make_adj(V, E, src, dst);
  int32_t *indeg = calloc((size_t)V + 1, sizeof(int32_t));
  int32_t head = 0, tail = 0;
  for (int32_t e = 0; e < E; ++e) indeg[dst[e]]++;
  for (int32_t v = 0; v < V; ++v)
    if (indeg[v] == 0) order[tail++] = v;
  /* Kahn's algorithm */
  while (head < tail) {
    int32_t u = order[head++];
    for (int32_t q = succ.ptr[u]; q < succ.ptr[u + 1]; ++q)
      if (--indeg[succ.idx[q]] == 0) order[tail++] = succ.idx[q];
  }
  free(indeg);
  if (tail != V) { free_adj(succ); return 1; }
  /* ASAP_v = max over predecessors of ASAP_u + Lat(u); 0 for sources. */
  for (int32_t v = 0; v < V; ++v) asap[v] = 0;
  for (int32_t i = 0; i < V; ++i) {
    int32_t u = order[i];
    for (int32_t q = succ.ptr[u]; q < succ.ptr[u + 1]; ++q)
      if (asap[succ.idx[q]] < asap[u] + lat[u]) asap[succ.idx[q]] = asap[u] + lat[u];
  }
  int32_t crit = 0;
  for (int32_t v = 0; v < V; ++v)
    if (asap[v] + lat[v] > crit) crit = asap[v] + lat[v];
  *cp = crit;
  /* ALAP_v = min(D - Lat(v), min over successors of ALAP_w - Lat(v)). */
  for (int32_t i = V - 1; i >= 0; --i) {
    int32_t v = order[i];
    int32_t a = D - lat[v];
    for (int32_t q = succ.ptr[v]; q < succ.ptr[v + 1]; ++q)
      if (alap[succ.idx[q]] - lat[v] < a) a = alap[succ.idx[q]] - lat[v];
    alap[v] = a;
  }
  free_adj(succ);
  return crit > D ? 2 : 0;
}

/* tau * log sum_t exp(x_t / tau), evaluated with the max shifted out; writes the
 * softmax weights (its gradient) to w. */
static double lse_tau(const double *x, int32_t n, double tau, double *w) {
  double m = -INFINITY, s = 0.0;
  for (int32_t t = 0; t < n; ++t) if (x[t] > m) m = x[t];
  for (int32_t t = 0; t < n; ++t) s += exp((x[t] - m) / tau);
  for (int32_t t = 0; t < n; ++t) w[t] = exp((x[t] - m) / tau) / s;
  return m + tau * log(s);
}

/* Cumulative C_x(d) = sum_{d' <= d} P_x^{d'} (Eq. active, second line). */
static void cumulative(const double *P, int32_t D, double *Cum) {
  double acc = 0.0;
  for (int32_t d = 0; d < D; ++d) { acc += P[d]; Cum[d] = acc; }
}

/* Expected live storage Reg(d) (Eq. active), before folding. */
static void expected_reg(const orc_problem *p, const adj_list *succ, const double *Cum, double *Reg) {
  int32_t V = p->V, D = p->D;
  for (int32_t d = 0; d < D; ++d) Reg[d] = 0.0;
  for (int32_t i = 0; i < V; ++i) {
    int has_succ = succ->ptr[i + 1] > succ->ptr[i];
    for (int32_t d = 0; d < D; ++d) {
      double prod = 0.0; /* leaf: the sink at step D has C_sink(d) = 0 */
      if (has_succ) {
        prod = 1.0;
        for (int32_t q = succ->ptr[i]; q < succ->ptr[i + 1]; ++q) prod *= Cum[(size_t)succ->idx[q] * D + d];
      }
      Reg[d] += p->bits[i] * Cum[(size_t)i * D + d] * (1.0 - prod);
    }
  }
}

void orc_expected_hist(const orc_problem *p, int32_t fam, const double *mu, const double *sigma,
                       double *U, double *Reg) {
  int32_t V = p->V, D = p->D, Dh = fold_len(p);
  double *P = malloc(sizeof(double) * (size_t)V * D);
  double *Cum = malloc(sizeof(double) * (size_t)V * D);
  double *R = malloc(sizeof(double) * (size_t)D);
  for (int32_t v = 0; v < V; ++v) {
    bin_masses_and_derivs(D, fam, mu[v], sigma[v], P + (size_t)v * D, NULL, NULL);
    cumulative(P + (size_t)v * D, D, Cum + (size_t)v * D);
  }
  for (int32_t i = 0; i < p->C * Dh; ++i) U[i] = 0.0;
  for (int32_t v = 0; v < V; ++v)
    for (int32_t d = 0; d < D; ++d)
      U[p->cls[v] * Dh + fold_of(p, d)] += p->demand[v] * P[(size_t)v * D + d];
  adj_list succ = make_adj(V, p->E, p->src, p->dst);
  expected_reg(p, &succ, Cum, R);
  free_adj(succ);
  for (int32_t t = 0; t < Dh; ++t) Reg[t] = 0.0;
  for (int32_t d = 0; d < D; ++d) Reg[fold_of(p, d)] += R[d];
  free(P); free(Cum); free(R);
}

/* One restart: forward values, then the gradient of the total loss (Sec. 3.3)
 * w.r.t. every bin mass, then chained to (mu, sigma). */
static void loss_grad_one(const orc_problem *p, const orc_hparams *h, const double *mu,
                          const double *sigma, const double *lambda, double *loss,
                          double *terms, double *gmu, double *gsig) {
  const int32_t V = p->V, D = p->D, E = p->E, C = p->C, Dh = fold_len(p);
  const uint32_t on = h->terms;
  double *P = calloc((size_t)V * D, sizeof(double));
  double *dPm = calloc((size_t)V * D, sizeof(double));
  double *dPs = calloc((size_t)V * D, sizeof(double));
  double *gP = calloc((size_t)V * D, sizeof(double));   /* dL/dP_v^d   */
  double *Cum = calloc((size_t)V * D, sizeof(double));
  double *gCum = calloc((size_t)V * D, sizeof(double)); /* dL/dC_v(d)  */
  double *U = calloc((size_t)C * Dh, sizeof(double));
  double *gU = calloc((size_t)C * Dh, sizeof(double));
  double *sm = calloc((size_t)(Dh > D ? Dh : D) + 1, sizeof(double));
  double *Reg = calloc((size_t)D, sizeof(double));
  double *MReg = calloc((size_t)Dh, sizeof(double));
  double *gMReg = calloc((size_t)Dh, sizeof(double));

  for (int32_t v = 0; v < V; ++v) {
    bin_masses_and_derivs(D, h->family, mu[v], sigma[v], P + (size_t)v * D, dPm + (size_t)v * D,
                          dPs + (size_t)v * D);
    cumulative(P + (size_t)v * D, D, Cum + (size_t)v * D);
  }
#define PP(v, d) P[(size_t)(v) * D + (d)]

  for (int32_t t = 0; t < ORC_NT; ++t) terms[t] = 0.0;
  double L = 0.0;

  /* ---- forward: expected usage per class (App. B.2), folded by App. B.3 ---- */
  for (int32_t v = 0; v < V; ++v)
    for (int32_t d = 0; d < D; ++d) U[p->cls[v] * Dh + fold_of(p, d)] += p->demand[v] * PP(v, d);

  if (on & ORC_RES_OBJ) {
    for (int32_t c = 0; c < C; ++c) {
      double l = lse_tau(U + c * Dh, Dh, h->tau, sm);
      terms[ORC_T_RES] += l;
      for (int32_t t = 0; t < Dh; ++t) gU[c * Dh + t] += h->w_res * sm[t];
    }
    L += h->w_res * terms[ORC_T_RES];
  }
  if (on & ORC_RES_VIOL) {
    double vres = 0.0;
    for (int32_t c = 0; c < C; ++c) {
      if (isinf(p->limit[c])) continue;
      for (int32_t t = 0; t < Dh; ++t)
        if (U[c * Dh + t] > p->limit[c]) vres += U[c * Dh + t] - p->limit[c];
    }
    terms[ORC_T_VRES] = vres;
    double coef = lambda[ORC_K_RES] + h->rho * vres;
    L += lambda[ORC_K_RES] * vres + 0.5 * h->rho * vres * vres;
    for (int32_t c = 0; c < C; ++c) {
      if (isinf(p->limit[c])) continue;
      for (int32_t t = 0; t < Dh; ++t)
        if (U[c * Dh + t] > p->limit[c]) gU[c * Dh + t] += coef;
    }
  }
  /* usage histogram -> bin masses: dU_c(fold d)/dP_v^d = r_v */
  for (int32_t v = 0; v < V; ++v)
    for (int32_t d = 0; d < D; ++d) gP[(size_t)v * D + d] += p->demand[v] * gU[p->cls[v] * Dh + fold_of(p, d)];

  /* ---- dependency violations, Eq. dep with latency: sum_e sum_a sum_b P_u^a P_v^b [b < a + Lat(u)] ---- */
  if (on & ORC_DEP) {
    double vdep = 0.0;
    for (int32_t e = 0; e < E; ++e) {
      int32_t u = p->src[e], v = p->dst[e], Lu = p->lat[u];
      for (int32_t a = 0; a < D; ++a)
        for (int32_t b = 0; b < D; ++b)
          if (b < a + Lu) vdep += PP(u, a) * PP(v, b);
    }
    terms[ORC_T_VDEP] = vdep;
    L += lambda[ORC_K_DEP] * vdep + 0.5 * h->rho * vdep * vdep;
    double coef = lambda[ORC_K_DEP] + h->rho * vdep;
    for (int32_t e = 0; e < E; ++e) {
      int32_t u = p->src[e], v = p->dst[e], Lu = p->lat[u];
      for (int32_t a = 0; a < D; ++a)
        for (int32_t b = 0; b < D; ++b)
          if (b < a + Lu) {
            gP[(size_t)u * D + a] += coef * PP(v, b);
            gP[(size_t)v * D + b] += coef * PP(u, a);
          }
    }
  }

  /* ---- communication, App. B.1: sum_e sum_a sum_{b >= a} P_u^a P_v^b (b - a) ---- */
  if (on & ORC_COM) {
    double lcom = 0.0;
    for (int32_t e = 0; e < E; ++e) {
      int32_t u = p->src[e], v = p->dst[e];
      for (int32_t a = 0; a < D; ++a)
        for (int32_t b = a; b < D; ++b) {
          lcom += PP(u, a) * PP(v, b) * (double)(b - a);
          gP[(size_t)u * D + a] += h->alpha * PP(v, b) * (double)(b - a);
          gP[(size_t)v * D + b] += h->alpha * PP(u, a) * (double)(b - a);
        }
    }
    terms[ORC_T_COM] = lcom;
    L += h->alpha * lcom;
  }

  /* ---- recurrence violations, App. B.3 with latency:
   *      sum_{(j->i,k)} sum_a sum_b P_i^a P_j^b [b + Lat(j) > a + k*II] ---- */
  if ((on & ORC_REC) && p->II > 0) {
    double vrec = 0.0;
    for (int32_t q = 0; q < p->NB; ++q) {
      int32_t j = p->bsrc[q], i = p->bdst[q], k = p->bdist[q], Lj = p->lat[j];
      for (int32_t a = 0; a < D; ++a)
        for (int32_t b = 0; b < D; ++b)
          if (b + Lj > a + k * p->II) vrec += PP(i, a) * PP(j, b);
    }
    terms[ORC_T_VREC] = vrec;
    L += lambda[ORC_K_REC] * vrec + 0.5 * h->rho * vrec * vrec;
    double coef = lambda[ORC_K_REC] + h->rho * vrec;
    for (int32_t q = 0; q < p->NB; ++q) {
      int32_t j = p->bsrc[q], i = p->bdst[q], k = p->bdist[q], Lj = p->lat[j];
      for (int32_t a = 0; a < D; ++a)
        for (int32_t b = 0; b < D; ++b)
          if (b + Lj > a + k * p->II) {
            gP[(size_t)i * D + a] += coef * PP(j, b);
            gP[(size_t)j * D + b] += coef * PP(i, a);
          }
    }
  }

  /* ---- expected live storage, Eq. active, and its LogSumExp (Eq. max) ---- */
  if (on & ORC_REG_OBJ) {
    adj_list succ = make_adj(V, E, p->src, p->dst);
    expected_reg(p, &succ, Cum, Reg);
    for (int32_t d = 0; d < D; ++d) MReg[fold_of(p, d)] += Reg[d];
    double l = lse_tau(MReg, Dh, h->tau, sm);
    terms[ORC_T_REG] = l;
    L += h->w_mem * l;
    for (int32_t t = 0; t < Dh; ++t) gMReg[t] = h->w_mem * sm[t];
    for (int32_t i = 0; i < V; ++i) {
      int32_t q0 = succ.ptr[i], q1 = succ.ptr[i + 1];
      for (int32_t d = 0; d < D; ++d) {
        double g = gMReg[fold_of(p, d)] * p->bits[i];
        double prod = 0.0;
        if (q1 > q0) {
          prod = 1.0;
          for (int32_t q = q0; q < q1; ++q) prod *= Cum[(size_t)succ.idx[q] * D + d];
        }
        gCum[(size_t)i * D + d] += g * (1.0 - prod);
        /* d/dC_j of -C_i * prod_{j'} C_j' : the product over the other successors */
        for (int32_t q = q0; q < q1; ++q) {
          double others = 1.0;
          for (int32_t q2 = q0; q2 < q1; ++q2)
            if (q2 != q) others *= Cum[(size_t)succ.idx[q2] * D + d];
          gCum[(size_t)succ.idx[q] * D + d] -= g * Cum[(size_t)i * D + d] * others;
        }
      }
    }
    free_adj(succ);
    /* C_x(d) = sum_{d' <= d} P_x^{d'}  =>  dL/dP_x^{d'} += sum_{d >= d'} dL/dC_x(d) */
    for (int32_t x = 0; x < V; ++x)
      for (int32_t dp = 0; dp < D; ++dp)
        for (int32_t d = dp; d < D; ++d) gP[(size_t)x * D + dp] += gCum[(size_t)x * D + d];
  }

  /* ---- chain rule through Eq. round ---- */
  for (int32_t v = 0; v < V; ++v) {
    double gm = 0.0, gs = 0.0;
    for (int32_t d = 0; d < D; ++d) {
      gm += gP[(size_t)v * D + d] * dPm[(size_t)v * D + d];
      gs += gP[(size_t)v * D + d] * dPs[(size_t)v * D + d];
    }
    gmu[v] = gm;
    gsig[v] = gs;
  }
  /* ---- continuous dependency penalty (a variant, not the paper's binned Eq. dep):
   *      X_u + Lat(u) - X_v ~ N(mu_u + Lat(u) - mu_v, sigma_u^2 + sigma_v^2) for the
   *      independent unrounded normals, so P(X_u + Lat(u) > X_v) = Phi(m / s) ---- */
  if (on & ORC_DEP_CF) {
    double vdep = 0.0;
    for (int32_t e = 0; e < E; ++e) {
      int32_t u = p->src[e], v = p->dst[e];
      double m = mu[u] + p->lat[u] - mu[v], s = sqrt(sigma[u] * sigma[u] + sigma[v] * sigma[v]);
      vdep += orc_Phi(m / s);
    }
    terms[ORC_T_VDEP] = vdep;
    L += lambda[ORC_K_DEP] * vdep + 0.5 * h->rho * vdep * vdep;
    double coef = lambda[ORC_K_DEP] + h->rho * vdep;
    for (int32_t e = 0; e < E; ++e) {
      int32_t u = p->src[e], v = p->dst[e];
      double m = mu[u] + p->lat[u] - mu[v], s = sqrt(sigma[u] * sigma[u] + sigma[v] * sigma[v]);
      double f = orc_phi(m / s);
      /* d Phi(m/s) = f (dm / s - m ds / s^2), ds/dsigma_x = sigma_x / s */
      gmu[u] += coef * f / s;
      gmu[v] -= coef * f / s;
      gsig[u] -= coef * f * m * sigma[u] / (s * s * s);
      gsig[v] -= coef * f * m * sigma[v] / (s * s * s);
    }
  }
  *loss = L;
#undef PP
  free(P); free(dPm); free(dPs); free(gP); free(Cum); free(gCum); free(U); free(gU);
  free(sm); free(Reg); free(MReg); free(gMReg);
}

void orc_loss_grad(const orc_problem *p, const orc_hparams *h, int32_t B,
                   const double *mu, const double *sigma, const double *lambda,
                   double *loss, double *terms, double *gmu, double *gsigma) {
  const int32_t V = p->V;
#pragma omp parallel for schedule(dynamic, 1)
  for (int32_t b = 0; b < B; ++b)
    loss_grad_one(p, h, mu + (size_t)b * V, sigma + (size_t)b * V, lambda + (size_t)b * ORC_K,
                  loss + b, terms + (size_t)b * ORC_NT, gmu + (size_t)b * V,
                  gsigma + (size_t)b * V);
}

/* Adam as implemented by torch.optim.Adam (no weight decay, no amsgrad). */
void orc_adam(int64_t n, double *theta, const double *g, double *m, double *v,
              int32_t step, double lr, double beta1, double beta2, double eps) {
  double bc1 = 1.0 - pow(beta1, step), bc2 = 1.0 - pow(beta2, step);
  for (int64_t i = 0; i < n; ++i) {
    m[i] = beta1 * m[i] + (1.0 - beta1) * g[i];
    v[i] = beta2 * v[i] + (1.0 - beta2) * g[i] * g[i];
    double mhat = m[i] / bc1, vhat = v[i] / bc2;
    theta[i] -= lr * mhat / (sqrt(vhat) + eps);
  }
}

void orc_round(int64_t n, const double *mu, int32_t *s) {
  for (int64_t i = 0; i < n; ++i) s[i] = (int32_t)floor(mu[i] + 0.5);
}

void orc_legalize_regular(const orc_problem *p, const int32_t *order,
                          const int32_t *asap, const int32_t *alap, int32_t *s) {
  adj_list pred = make_adj(p->V, p->E, p->dst, p->src);
  for (int32_t v = 0; v < p->V; ++v) {
    if (s[v] < asap[v]) s[v] = asap[v];
    if (s[v] > alap[v]) s[v] = alap[v];
  }
  for (int32_t i = 0; i < p->V; ++i) {
    int32_t v = order[i];
    if (pred.ptr[v + 1] == pred.ptr[v]) continue;
    int32_t treq = INT32_MIN;
    for (int32_t q = pred.ptr[v]; q < pred.ptr[v + 1]; ++q) {
      int32_t u = pred.idx[q], t = s[u] + p->lat[u];
      if (t > treq) treq = t;
    }
    if (treq > s[v]) s[v] = treq;
  }
  free_adj(pred);
}

int orc_legalize_modulo(const orc_problem *p, const int32_t *order, int32_t *s) {
  adj_list pred = make_adj(p->V, p->E, p->dst, p->src);
  int32_t *ones = malloc(sizeof(int32_t) * ((size_t)p->NB + 1));
  for (int32_t q = 0; q < p->NB; ++q) ones[q] = q;
  adj_list back = make_adj(p->V, p->NB, p->bdst, ones); /* back edges by consumer i */
  free(ones);
  int rc = 1;
  for (int32_t it = 0; it < p->V; ++it) {
    int changed = 0;
    for (int32_t n = 0; n < p->V; ++n) {
      int32_t v = order[n], tmin = 0, tback = 0;
      for (int32_t q = pred.ptr[v]; q < pred.ptr[v + 1]; ++q) {
        int32_t u = pred.idx[q];
        if (s[u] + p->lat[u] > tmin) tmin = s[u] + p->lat[u];
      }
      for (int32_t q = back.ptr[v]; q < back.ptr[v + 1]; ++q) {
        int32_t b = back.idx[q], j = p->bsrc[b];
        int32_t t = s[j] + p->lat[j] - p->bdist[b] * p->II;
        if (t > tback) tback = t;
      }
      int32_t treq = tmin > tback ? tmin : tback;
      if (treq > s[v]) { s[v] = treq; changed = 1; }
    }
    if (!changed) { rc = 0; break; }
  }
  free_adj(pred);
  free_adj(back);
  return rc;
}

void orc_verify(const orc_problem *p, const int32_t *s, orc_report *r) {
  const int32_t V = p->V, D = p->D, E = p->E, C = p->C;
  const int32_t Dh = fold_len(p);
  memset(r, 0, sizeof(*r));
  for (int32_t e = 0; e < E; ++e) {
    int32_t u = p->src[e], v = p->dst[e];
    if (s[v] < s[u] + p->lat[u]) r->n_dep_viol++;
    r->L_com += (int64_t)s[v] - s[u];
  }
  for (int32_t v = 0; v < V; ++v)
    if (s[v] < 0 || s[v] + p->lat[v] > D) r->n_lat_viol++;
  if (p->II > 0)
    for (int32_t q = 0; q < p->NB; ++q) {
      int32_t j = p->bsrc[q], i = p->bdst[q];
      if ((int64_t)s[i] + (int64_t)p->bdist[q] * p->II < (int64_t)s[j] + p->lat[j]) r->n_rec_viol++;
    }
  /* Res(d) = sum_v r_v [s_v = d] for d in [0, D), folded when II > 0 */
  int64_t *cnt = calloc((size_t)C * Dh, sizeof(int64_t));
  for (int32_t v = 0; v < V; ++v)
    if (s[v] >= 0 && s[v] < D) cnt[p->cls[v] * Dh + fold_of(p, s[v])] += (int64_t)llround(p->demand[v]);
  for (int32_t c = 0; c < C; ++c) {
    int64_t pk = 0;
    for (int32_t t = 0; t < Dh; ++t) {
      int64_t x = cnt[c * Dh + t];
      if (x > pk) pk = x;
      if (!isinf(p->limit[c]) && (double)x > p->limit[c]) r->n_res_viol++;
    }
    if (c < 16) r->peak[c] = pk;
    r->L_res += pk;
  }
  free(cnt);
  /* Mem(d) = sum_i b_i [s_i <= d < max_{j in succ(i)} s_j], leaves' sink at D */
  int64_t *mem = calloc((size_t)D, sizeof(int64_t));
  adj_list succ = make_adj(V, E, p->src, p->dst);
  for (int32_t i = 0; i < V; ++i) {
    int32_t last = D; /* leaf: the sink at step D */
    if (succ.ptr[i + 1] > succ.ptr[i]) {
      last = INT32_MIN;
      for (int32_t q = succ.ptr[i]; q < succ.ptr[i + 1]; ++q)
        if (s[succ.idx[q]] > last) last = s[succ.idx[q]];
    }
    for (int32_t d = 0; d < D; ++d)
      if (s[i] <= d && d < last) mem[d] += (int64_t)llround(p->bits[i]);
  }
  free_adj(succ);
  for (int32_t d = 0; d < D; ++d) if (mem[d] > r->L_mem) r->L_mem = mem[d];
  int64_t *mm = calloc((size_t)Dh, sizeof(int64_t));
  for (int32_t d = 0; d < D; ++d) mm[fold_of(p, d)] += mem[d];
  for (int32_t t = 0; t < Dh; ++t) if (mm[t] > r->L_mmem) r->L_mmem = mm[t];
  free(mem); free(mm);
  r->feasible = (r->n_dep_viol == 0 && r->n_lat_viol == 0 && r->n_rec_viol == 0);
  r->res_ok = (r->n_res_viol == 0);
}

/* ---- Outer loop of Alg. GauS ---- */

/* Sec. 3.3 Initialization: "sigma = kappa (s_ALAP - s_ASAP)" and mu the midpoint
 * of [ASAP, ALAP] (or a given mu0).  sigma is floored at sigma_min because a node
 * without slack would otherwise start with sigma = 0. */
void orc_init_state(int32_t V, const int32_t *asap, const int32_t *alap, double kappa, float sigma_min,
                    const float *mu0, float *mu, float *sigma) {
  for (int32_t v = 0; v < V; ++v) {
    float sv = (float)(kappa * (double)(alap[v] - asap[v]));
    if (!(sv >= sigma_min)) sv = sigma_min;
    sigma[v] = sv;
    mu[v] = mu0 ? mu0[v] : (float)(0.5 * ((double)asap[v] + (double)alap[v]));
  }
}

/* Alg. GauS: "s = round(mu); mu, sigma <- legalize(s) if s is illegal"; App. A:
 * when the legalized schedule does not improve on the running best, the
 * optimizer is reset to the prior best.  A legalized schedule is a candidate when
 * legalization succeeded and it has no dependency, latency or recurrence
 * violation (and no resource overflow when the ReLU resource term is on); its
 * score is the discrete objective of the active terms. */
int32_t orc_outer_step(int32_t V, int32_t leg_ok, const int32_t *s_legal, const orc_report *r, uint32_t terms,
                       int32_t II, double w_res, double alpha, double w_mem, int32_t iter, const int32_t *asap,
                       const int32_t *alap, const float *sigma_init, int32_t *best_sched, double *best_score,
                       int32_t *best_iter, float *mu, float *sigma, float *m_mu, float *v_mu, float *m_sg,
                       float *v_sg, int32_t *step) {
  int32_t moved = 0;
  for (int32_t v = 0; v < V; ++v) {
    const double m = (double)mu[v];
    if (!isfinite(m) || floor(m + 0.5) != (double)s_legal[v]) ++moved;
  }
  const int cand = leg_ok && r->feasible && (!(terms & ORC_RES_VIOL) || r->res_ok);
  double score = 0.0;
  if (terms & ORC_RES_OBJ) score += w_res * (double)r->L_res;
  if (terms & ORC_COM) score += alpha * (double)r->L_com;
  if (terms & ORC_REG_OBJ) score += w_mem * (double)(II > 0 ? r->L_mmem : r->L_mem);
  const int had_best = *best_iter >= 0;
  const int improved = cand && score < *best_score;
  const int illegal = !leg_ok || moved > 0;
  if (improved) {
    for (int32_t v = 0; v < V; ++v) best_sched[v] = s_legal[v];
    *best_score = score;
    *best_iter = iter;
  }
  if (illegal) {
    /* "mu, sigma <- legalize(s)": the legalized schedule, unless it does not improve
     * on a prior best (then that best); the midpoint only when legalization failed
     * and there is no best */
    for (int32_t v = 0; v < V; ++v) {
      if (improved || (leg_ok && !had_best)) mu[v] = (float)s_legal[v];
      else if (had_best) mu[v] = (float)best_sched[v];
      else mu[v] = (float)(0.5 * ((double)asap[v] + (double)alap[v]));
      sigma[v] = sigma_init[v];
      m_mu[v] = v_mu[v] = m_sg[v] = v_sg[v] = 0.0f;
    }
    *step = 0;
  }
  return leg_ok ? moved : -1;
}
