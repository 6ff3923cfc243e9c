/*
 * gaus_oracle.h -- fp64 CPU oracle for GauS (arXiv 2602.20427).
 *
 * TEST INFRASTRUCTURE.  Only the tests, the smoke check and the CPU-baseline leg
 * of the benchmark call this code.  It shares nothing with the CUDA library: no
 * header, no helper, no table.  Everything is evaluated over the whole horizon
 * d = 0..D-1 (no window), with the paper's double sums written out as stated.
 *
 * Arrays of per-restart data are restart-major here: x[b * V + v].
 */
#ifndef GAUS_ORACLE_H
#define GAUS_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* term bits (which parts of the objective and which constraints are active) */
#define ORC_DEP      1u   /* expected dependency violations (Sec. 3.2, Eq. dep)    */
#define ORC_COM      2u   /* expected communication cost (App. B.1)                */
#define ORC_RES_OBJ  4u   /* LogSumExp of expected usage per class (App. B.2)      */
#define ORC_RES_VIOL 8u   /* ReLU resource violation (App. B.2, Eq. relu)          */
#define ORC_REG_OBJ 16u   /* LogSumExp of expected live storage (Eq. active, max)  */
#define ORC_REC     32u   /* expected recurrence violations (App. B.3)             */
/* NOT the paper's Eq. dep: the continuous dependency penalty
 * sum_e Phi((mu_u + Lat(u) - mu_v) / sqrt(sigma_u^2 + sigma_v^2)) = sum_e P(X_u + Lat(u) > X_v)
 * of the unrounded normals, a variant kept apart from ORC_DEP (same multiplier). */
#define ORC_DEP_CF  64u

/* constraint slots of the augmented Lagrangian (Sec. 3.3) */
#define ORC_K_DEP 0
#define ORC_K_RES 1
#define ORC_K_REC 2
#define ORC_K     3

/* per-restart term values written by orc_loss_grad */
#define ORC_T_RES  0   /* sum_c LSE_tau(usage_c)       */
#define ORC_T_COM  1   /* expected communication       */
#define ORC_T_REG  2   /* LSE_tau(expected storage)    */
#define ORC_T_VDEP 3
#define ORC_T_VRES 4
#define ORC_T_VREC 5
#define ORC_NT     6

typedef struct {
  int32_t V, E;
  const int32_t *src, *dst;     /* edge e: src[e] -> dst[e] (producer -> consumer) */
  const int32_t *lat;           /* Lat(v) >= 0                                      */
  const int32_t *cls;           /* resource class of v, 0..C-1                      */
  int32_t C;
  const double *limit;          /* R_c; INFINITY = unlimited                        */
  const double *demand;         /* r_v (resource demand)                            */
  const double *bits;           /* b_v (storage units of v's output)                */
  int32_t NB;                   /* back edges (j -> i, distance k)                  */
  const int32_t *bsrc, *bdst, *bdist;
  int32_t D, II;                /* horizon; initiation interval (0 = regular)       */
} orc_problem;

/* CDF family of the relaxation (Sec. 3.2 with Phi; App. D for the others) */
#define ORC_GAUSSIAN 0
#define ORC_LOGISTIC 1
#define ORC_LAPLACE  2
#define ORC_CAUCHY   3

typedef struct {
  double tau, rho, alpha, w_res, w_mem;
  uint32_t terms;
  int32_t family;               /* ORC_GAUSSIAN .. ORC_CAUCHY                        */
} orc_hparams;

typedef struct {
  int64_t n_dep_viol, n_lat_viol, n_rec_viol, n_res_viol;
  int64_t L_res, L_com, L_mem, L_mmem;
  int64_t peak[16];             /* peak (folded when II > 0) usage per class        */
  int32_t feasible, res_ok;
} orc_report;

/* Standard normal CDF and density. */
double orc_Phi(double z);
double orc_phi(double z);

/* CDF F and density f of a family in the standardized z = (x - mu) / sigma,
 * scale-matched to N(0, 1) (App. D); F = Phi, f = phi for ORC_GAUSSIAN. */
double orc_F(int32_t fam, double z);
double orc_f(int32_t fam, double z);

/* Bin masses of Eq. round over d = 0..D-1, with open first and last bins. */
void orc_bin_masses(int32_t D, int32_t fam, double mu, double sigma, double *P);

/* Topological order (Kahn), ASAP, ALAP, critical path.
 * returns 0 ok, 1 cycle, 2 critical path longer than D. */
int orc_asap_alap(int32_t V, int32_t E, const int32_t *src, const int32_t *dst,
                  const int32_t *lat, int32_t D, int32_t *order, int32_t *asap,
                  int32_t *alap, int32_t *cp);

/* Expected histograms for one restart: usage U[c*Dh + t] and storage Reg[t],
 * folded modulo II when II > 0 (Dh = II), else Dh = D. */
void orc_expected_hist(const orc_problem *p, int32_t fam, const double *mu, const double *sigma,
                       double *U, double *Reg);

/* Loss, term values and gradient for B restarts (OpenMP over restarts). */
void orc_loss_grad(const orc_problem *p, const orc_hparams *h, int32_t B,
                   const double *mu, const double *sigma, const double *lambda,
                   double *loss, double *terms, double *gmu, double *gsigma);

/* One Adam step (PyTorch semantics) on n parameters; step is 1-based. */
void orc_adam(int64_t n, double *theta, const double *g, double *m, double *v,
              int32_t step, double lr, double beta1, double beta2, double eps);

/* s = floor(mu + 1/2) (round half up). */
void orc_round(int64_t n, const double *mu, int32_t *s);

/* App. A, Alg. 1 (regular legalization) in the given topological order. */
void orc_legalize_regular(const orc_problem *p, const int32_t *order,
                          const int32_t *asap, const int32_t *alap, int32_t *s);

/* App. A, Alg. 2 (modulo legalization).  returns 0 converged, 1 not converged
 * within |V| sweeps. */
int orc_legalize_modulo(const orc_problem *p, const int32_t *order, int32_t *s);

/* Discrete objectives and constraint checks (Sec. 2.1) of one schedule. */
void orc_verify(const orc_problem *p, const int32_t *s, orc_report *r);

/* Sec. 3.3 Initialization for one restart: sigma_v = kappa (ALAP_v - ASAP_v),
 * floored at sigma_min, and mu_v = (ASAP_v + ALAP_v) / 2 (or mu0[v] when given);
 * computed in double, stored as the float32 state. */
void orc_init_state(int32_t V, const int32_t *asap, const int32_t *alap, double kappa, float sigma_min,
                    const float *mu0, float *mu, float *sigma);

/* One outer step of Alg. GauS for one restart (sampling, "legalize if illegal";
 * App. A: reset to the prior best).  s_legal = legalization of round(mu), leg_ok
 * its success, r its report.  Updates the best (sched, score, iter) and, when the
 * rounded schedule was illegal, resets mu, sigma, the Adam moments and step.
 * Returns the number of nodes legalization moved, or -1 when it failed. */
int32_t orc_outer_step(int32_t V, int32_t leg_ok, const int32_t *s_legal, const orc_report *r, uint32_t terms,
                       int32_t II, double w_res, double alpha, double w_mem, int32_t iter, const int32_t *asap,
                       const int32_t *alap, const float *sigma_init, int32_t *best_sched, double *best_score,
                       int32_t *best_iter, float *mu, float *sigma, float *m_mu, float *v_mu, float *m_sg,
                       float *v_sg, int32_t *step);

#ifdef __cplusplus
}
#endif
#endif
