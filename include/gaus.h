/*
 * gaus.h -- C ABI of the GB300 (sm_103a) GauS hot path.
 *
 * GauS (arXiv 2602.20427) relaxes each operator's start step to a Gaussian
 * X_v ~ N(mu_v, sigma_v^2) (Sec. 3.1; App. D: or a scale-matched logistic,
 * Laplace or Cauchy variable), turns objectives and constraint
 * violations into expectations over the rounded steps (Sec. 3.2, App. B) and
 * minimises them with an augmented Lagrangian and Adam (Sec. 3.3).  This
 * library evaluates that loss and its gradient, applies Adam and the
 * multiplier update, rounds and legalizes the means (App. A), and verifies
 * schedules (Sec. 2.1), for B independent restarts at once, on one GPU.
 *
 * Conventions (every entry point):
 *  - Per-restart node arrays are (V, B) row-major fp32/int32 device arrays:
 *    element [v * B + b] belongs to node v (the caller's id) and restart b.
 *    Per-restart vectors are (B, K) row-major.
 *  - The caller owns every device buffer it passes; the library owns only the
 *    context, its device copy of the graph and its scratch memory.
 *  - Every call is asynchronous on the context's stream.  Argument errors are
 *    returned at once and enqueue nothing.  Data-dependent conditions (a
 *    non-finite mu or sigma, Alg. 2 not settling) are written to per-restart
 *    device status words and never abort the call.
 *  - Entry points are not thread-safe on one context.
 */
#ifndef GAUS_H
#define GAUS_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct gaus_ctx gaus_ctx;

typedef enum {
  GAUS_OK = 0,
  GAUS_EINVAL = 1,      /* bad argument, graph arrays disagree, size out of range */
  GAUS_ECYCLE = 2,      /* the dependency graph has a cycle                        */
  GAUS_EHORIZON = 3,    /* critical path longer than the horizon D                 */
  GAUS_ENOMEM = 4,      /* device or host allocation failed                        */
  GAUS_ECUDA = 5,       /* a CUDA runtime call failed (see gaus_last_error)        */
  GAUS_ENONFINITE = 6,  /* per restart: a mu or sigma was NaN/Inf or sigma < 1e-30 */
  GAUS_ENOTCONV = 7,    /* per restart: Alg. 2 did not settle within |V| sweeps    */
  GAUS_ETIMEOUT = 8     /* per restart: a barrier of the persistent iteration kernel
                           waited longer than its limit (4 s); that call's outputs
                           for the restart are unspecified                            */
} gaus_status;

/* Terms of the loss (bit mask).  Objectives are weighted, constraints enter the
 * augmented Lagrangian of Sec. 3.3. */
#define GAUS_DEP      1u  /* constraint: expected dependency violations, Eq. dep with latency    */
#define GAUS_COM      2u  /* objective:  alpha * expected communication, App. B.1                */
#define GAUS_RES_OBJ  4u  /* objective:  w_res * sum_c LSE_tau(expected usage of class c), App. B.2 */
#define GAUS_RES_VIOL 8u  /* constraint: sum_c sum_t ReLU(usage - R_c), Eq. relu                 */
#define GAUS_REG_OBJ 16u  /* objective:  w_mem * LSE_tau(expected live storage), Eq. active/max  */
#define GAUS_REC     32u  /* constraint: expected recurrence violations, App. B.3 (II > 0)       */
/* constraint, a VARIANT that is not the paper's Eq. dep: the continuous dependency
 * penalty sum_e Phi((mu_u + Lat(u) - mu_v) / sqrt(sigma_u^2 + sigma_v^2)), i.e.
 * P(X_u + Lat(u) > X_v) of the unrounded normals, O(1) per edge; it takes the
 * dependency multiplier and term slot (GAUS_K_DEP, GAUS_T_VDEP).  Excludes GAUS_DEP;
 * needs family GAUS_GAUSSIAN. */
#define GAUS_DEP_CF  64u

/* Constraint slots (lambda, multiplier update) and per-restart term values. */
#define GAUS_K_DEP 0
#define GAUS_K_RES 1
#define GAUS_K_REC 2
#define GAUS_K     3
#define GAUS_T_RES  0   /* sum_c LSE_tau(U_c)             */
#define GAUS_T_COM  1   /* expected communication         */
#define GAUS_T_REG  2   /* LSE_tau(Reg)                   */
#define GAUS_T_VDEP 3   /* expected dependency violations */
#define GAUS_T_VRES 4   /* sum of ReLU resource excess    */
#define GAUS_T_VREC 5   /* expected recurrence violations */
#define GAUS_NT     6

/* CDF family that rounds X_v to a step (gaus_hparams.family).  The normal of
 * Sec. 3.2 or, in its place (App. D), a logistic, Laplace or Cauchy CDF whose
 * scale is matched to sigma: logistic s = sigma sqrt(3)/pi and Laplace
 * b = sigma/sqrt(2) have the variance sigma^2; Cauchy gamma = sigma sqrt(2 ln 2)
 * has the normal's full width at half maximum. */
#define GAUS_GAUSSIAN 0
#define GAUS_LOGISTIC 1
#define GAUS_LAPLACE  2
#define GAUS_CAUCHY   3

/* Scheduling problem (Sec. 2.1).  All pointers are HOST pointers, read during
 * gaus_create and not kept.  Node ids are 0..V-1. */
typedef struct {
  int32_t V, E;
  const int32_t *succ_ptr, *succ_idx;  /* CSR of edges u -> v: (V+1), (E)                    */
  const int32_t *pred_ptr, *pred_idx;  /* CSC of the same edges: (V+1), (E); must agree      */
  const int32_t *latency;              /* Lat(v) >= 0 (0 = chaining, Sec. 2.1), (V)          */
  const int32_t *res_class;            /* class of v in 0..C-1, (V)                          */
  int32_t C;                           /* number of resource classes, 1..16                  */
  const float *limit;                  /* R_c, (C); INFINITY = unlimited                     */
  const int32_t *demand;               /* r_v >= 0, (V); NULL = all 1                        */
  const int32_t *bits;                 /* b_v >= 0 storage units of v's output, (V); NULL = 1 */
  int32_t n_back;                      /* loop-carried edges j -> i with distance k (Sec. 2.1 Rec) */
  const int32_t *back_src;             /* j, (n_back)                                         */
  const int32_t *back_dst;             /* i, (n_back)                                         */
  const int32_t *back_dist;            /* k >= 1, (n_back)                                    */
  int32_t D;                           /* horizon: start steps 0..D-1 (Sec. 3.2)              */
  int32_t II;                          /* initiation interval; 0 = regular scheduling         */
  int32_t B;                           /* restarts per call, >= 1                             */
} gaus_problem;

typedef struct {
  float tau;        /* LogSumExp temperature (Eq. max); paper 1e-2                     */
  float rho;        /* ALM penalty (Sec. 3.3); paper 1e-4                               */
  float lambda0;    /* initial multiplier the caller should use; paper 1e-6             */
  float alpha;      /* weight of the communication objective (Formulation A)           */
  float w_res;      /* weight of the usage LSE objective                                */
  float w_mem;      /* weight of the storage LSE objective                              */
  float lr;         /* Adam learning rate; paper 1e-2                                   */
  float beta1, beta2, eps;   /* Adam; 0.9, 0.999, 1e-8                                  */
  float window_k;   /* bins further than window_k * sigma from mu carry no mass; 6.
                       Other families widen the window to the point whose tail mass
                       equals the normal's beyond window_k (logistic ~1.9x, Laplace
                       ~2.4x, Cauchy: the whole horizon for any practical D)       */
  float sigma_min;  /* sigma is clamped to >= sigma_min after each Adam step; 0.05     */
  uint32_t terms;   /* GAUS_* bit mask                                                  */
  int32_t family;   /* GAUS_GAUSSIAN (default) .. GAUS_CAUCHY                           */
} gaus_hparams;

/* Discrete verdict on one schedule (Sec. 2.1; App. B.1 for L_com). */
typedef struct {
  int64_t n_dep_viol;   /* edges u -> v with s_v < s_u + Lat(u)                       */
  int64_t n_lat_viol;   /* nodes with s_v < 0 or s_v + Lat(v) > D                     */
  int64_t n_rec_viol;   /* back edges with s_i + k II < s_j + Lat(j)                  */
  int64_t n_res_viol;   /* (class, step) cells whose usage exceeds R_c (folded if II)  */
  int64_t L_res;        /* sum over classes of peak usage (folded if II > 0)          */
  int64_t L_com;        /* sum over edges of s_v - s_u                                */
  int64_t L_mem;        /* max over d in [0, D) of Mem(d), leaves live until D         */
  int64_t L_mmem;       /* max over t in [0, II) of the folded Mem (= L_mem if II = 0) */
  int64_t peak[16];     /* per-class peak usage                                       */
  int32_t feasible;     /* no Dep, Lat or Rec violation                               */
  int32_t res_ok;       /* no resource cell over its limit                            */
} gaus_report;

/* State of gaus_iterate: DEVICE pointers owned by the caller. */
typedef struct {
  float *mu, *sigma;                   /* (V, B), updated in place                   */
  float *m_mu, *v_mu, *m_sigma, *v_sigma; /* Adam moments (V, B), zero-initialised by the caller */
  float *lambda;                       /* (B, GAUS_K) multipliers, updated in place   */
  int32_t *step;                       /* (B) Adam step count, incremented each iteration */
  float *loss;                         /* (B) out: loss of the last iteration        */
  float *terms;                        /* (B, GAUS_NT) out: term values of the last iteration */
  int32_t *status;                     /* (B) out: GAUS_OK or GAUS_ENONFINITE         */
} gaus_state;

/* Paper defaults (Sec. 3.3, App. C.1): tau 1e-2, rho 1e-4, lambda0 1e-6, lr 1e-2;
 * Adam betas (0.9, 0.999), eps 1e-8; alpha = w_res = w_mem = 1; window 6 sigma;
 * sigma_min 0.05; terms = DEP | COM | RES_OBJ; family GAUSSIAN.  Returns GAUS_EINVAL
 * on NULL. */
gaus_status gaus_default_hparams(gaus_hparams *hp);

/* Validate the problem, sort it topologically (Kahn), compute ASAP/ALAP and the
 * critical path (App. A, Alg. 1 input), build the class-sorted node order and
 * upload the graph to the device on `cuda_stream` (a cudaStream_t; NULL = the
 * legacy default stream).  Errors: EINVAL (arrays missing or inconsistent,
 * CSR/CSC disagree, duplicate edge, ids out of range, C outside 1..16, D < 1,
 * II < 0, B < 1, sizes beyond the library's limits; hparams out of range, unknown
 * term bits or family, GAUS_REC without II, GAUS_DEP with GAUS_DEP_CF, GAUS_DEP_CF
 * with a family other than the normal), ECYCLE, EHORIZON, ENOMEM, ECUDA.  On
 * success *out owns device memory until gaus_destroy. */
gaus_status gaus_create(const gaus_problem *prob, const gaus_hparams *hp, void *cuda_stream,
                        gaus_ctx **out);

/* Replace the hyperparameters (same validation as gaus_create). */
gaus_status gaus_set_hparams(gaus_ctx *ctx, const gaus_hparams *hp);

/* Copy ASAP, ALAP (host int32 arrays of V, caller ids; either may be NULL) and
 * the critical path length (may be NULL) computed at creation. */
gaus_status gaus_bounds(const gaus_ctx *ctx, int32_t *asap, int32_t *alap, int32_t *cp);

/* Loss of Sec. 3.3 and its gradient for B restarts:
 *   L_b = w_res sum_c LSE_tau(U_c) + alpha L_com + w_mem LSE_tau(Reg)
 *         + sum_{k active} (lambda[b,k] V_k + rho/2 V_k^2),
 * with U_c(t) = sum_{cls(v)=c} r_v P_v^t (folded mod II when II > 0) and the
 * bin masses P of Eq. round, truncated to +-window_k sigma.
 *   mu, sigma   (V, B) device, read only.
 *   lambda      (B, GAUS_K) device, read only.
 *   grad_mu, grad_sigma (V, B) device, written.
 *   loss (B), terms (B, GAUS_NT), status (B) device, written; status may be NULL.
 * Non-finite mu/sigma or sigma < 1e-30 in restart b sets status[b] = ENONFINITE;
 * that restart's outputs are then unspecified. */
gaus_status gaus_loss_grad(gaus_ctx *ctx, const float *mu, const float *sigma,
                           const float *lambda, float *grad_mu, float *grad_sigma,
                           float *loss, float *terms, int32_t *status);

/* One Adam step (torch.optim.Adam semantics, no weight decay) on mu and sigma,
 * then sigma <- max(sigma, sigma_min) and, for every active constraint k,
 * lambda[b,k] += rho * terms[b, V_k] (Sec. 3.3 multiplier update).
 *   step >= 1 is the 1-based Adam step shared by all restarts.
 * All pointers are device pointers of the shapes above. */
gaus_status gaus_adam_step(gaus_ctx *ctx, float *mu, float *sigma, const float *grad_mu,
                           const float *grad_sigma, float *m_mu, float *v_mu, float *m_sigma,
                           float *v_sigma, float *lambda, const float *terms, int32_t step);

/* n_iters fused iterations of Alg. GauS's inner loop (loss, gradient, Adam,
 * multiplier update), enqueued on the context stream as replays of captured CUDA
 * graphs (ten iterations per graph, one-iteration graphs for the remainder; the
 * graphs are captured on first use and again after gaus_set_hparams or a change of
 * state pointers).  Equivalent to gaus_loss_grad + gaus_adam_step with
 * step = st->step[b] + 1 per iteration.  Gradients are not materialised.  EINVAL
 * on NULL state pointers or n_iters < 0. */
gaus_status gaus_iterate(gaus_ctx *ctx, int32_t n_iters, const gaus_state *st);

/* Kernel-level timing of gaus_iterate: runs n_iters iterations exactly as
 * gaus_iterate does, but launched without a graph and with CUDA events between
 * the phases, and adds the mean duration in milliseconds of each phase of an
 * iteration to ms_out[0..3] (host array of 4): [0] node pass (windows, CDF table,
 * usage histograms), [1] edge pass (the usage reduction runs beside it on a second
 * stream), [2] storage pass + per-restart finalize, [3] gradient gather + Adam.
 * Synchronises the context's stream.  Library feature for measurement; not on the
 * hot path. */
gaus_status gaus_profile_iterate(gaus_ctx *ctx, int32_t n_iters, const gaus_state *st, double *ms_out);

/* Phase profile of the persistent iteration kernel (measurement helper, not on the
 * hot path): runs n_iters iterations exactly as gaus_iterate does, with every block
 * recording the device's global timer at the start and end of each of its three
 * phases, and writes to out[0..11] (host, milliseconds, means over the
 * iterations): [0..2] critical path of phase 1 (windows, CDF table, usage
 * histogram), phase 2 (usage terms, edge terms) and phase 3 (gradient, Adam) --
 * the last block's end minus the first block's start; [3..5] the mean block's time
 * in each phase; [6..7] latency of the two group barriers (last arrival to first
 * release); [8] the whole iteration; [9..11] the slowest block in each phase.
 * Synchronises the context's stream.  EINVAL when the context's terms or sizes run
 * the multi-kernel path (storage term, continuous dependency penalty, D > 32767). */
gaus_status gaus_profile_phases(gaus_ctx *ctx, int32_t n_iters, const gaus_state *st, double *out);

/* The execution plan the context chose for its sizes and current hyperparameters
 * (host only: no CUDA call).  out (host, n entries, at most 16 written):
 *   [0] 1 when the persistent fused kernel applies to the current terms and sizes,
 *       0 when only the multi-kernel path does (storage term, continuous dependency
 *       penalty, D > 32767, or a device that cannot hold one block per restart group);
 *   [1] fused: cooperative kernel launches per fused gaus_iterate call (1 unless B
 *       exceeds the restart groups the device holds at once), else 0;
 *   [2] multi-kernel path: kernel launches per iteration;
 *   [3] restart groups; [4] blocks per restart group; [5] restarts per group;
 *   [6] points per CDF table row; [7] dynamic shared memory per fused block (bytes);
 *   [8] streaming multiprocessors of the device; [9] node segments of the fused
 *   kernel; [10] edge chunks of the fused kernel; [11] threads per fused block;
 *   [12] the path mode (gaus_set_path); since the context was created: [13]
 *   gaus_iterate calls run by the fused kernel, [14] iterations run by the
 *   multi-kernel path, [15] path-choice reductions launched (one kernel each).
 * EINVAL for a NULL context or out, or n < 1. */
gaus_status gaus_plan_info(const gaus_ctx *ctx, int64_t *out, int32_t n);

/* Which path gaus_iterate runs (gaus_set_path).  AUTO, the default, chooses per call
 * from the state's windows (window points of every (node, restart) under the
 * family's window, summed and maximised by one small reduction whose 16 bytes are
 * read back, so an AUTO call synchronises the context's stream once; a call made
 * while the stream is being captured takes the fused path): the persistent fused
 * kernel when the mean window is under one point, or when the longest window is at
 * most 32 points and at most twice the mean; the multi-kernel path otherwise.  Without
 * the reduction: problems of fewer than 16,384 (node, restart) items always take the
 * fused kernel, and restart groups of fewer than 64 restarts (B < 64) the multi-kernel
 * path.  FUSED
 * and MULTI force a path (FUSED falls back to the multi-kernel path where the fused
 * kernel does not apply).  gaus_loss_grad uses the fused kernel unless MULTI is set
 * or AUTO's size rule picks the multi-kernel path. */
#define GAUS_PATH_AUTO 0
#define GAUS_PATH_FUSED 1
#define GAUS_PATH_MULTI 2
gaus_status gaus_set_path(gaus_ctx *ctx, int32_t mode);

/* Exercises the fused kernel's bounded barrier waits (a check of the failure path,
 * not part of the method): one iteration of gaus_iterate whose group barriers can
 * never complete, each wait ending after limit_ns.  Every restart's status becomes
 * GAUS_ETIMEOUT; mu, sigma, the Adam moments, lambda and step are left as they were
 * (the kernel writes the caller's state only at the end of a completed call), and
 * the context stays usable.  limit_ns in 1,000 .. 1,000,000,000.  EINVAL for NULL
 * pointers, a limit outside that range, or a context on the multi-kernel path.
 * Asynchronous on the context's stream. */
gaus_status gaus_check_barrier_timeout(gaus_ctx *ctx, const gaus_state *st, uint64_t limit_ns);

/* Round every mean to s = floor(mu + 1/2) (Sec. 3.3 Sampling; exact for every
 * fp32 value) and legalize it: Alg. 1 (clamp to [ASAP, ALAP], then a forward push
 * in topological order with +Lat(u)) when II = 0, Alg. 2 (fixed-point relaxation
 * of forward and back edges, at most |V| sweeps) when II > 0.
 *   mu (V, B) device; sched (V, B) int32 device, written; status (B) device,
 *   written with OK, ENONFINITE or ENOTCONV (sched then unspecified). */
gaus_status gaus_legalize(gaus_ctx *ctx, const float *mu, int32_t *sched, int32_t *status);

/* Round only (no legalization): sched = floor(mu + 1/2). */
gaus_status gaus_round(gaus_ctx *ctx, const float *mu, int32_t *sched);

/* Verify B schedules (Sec. 2.1): sched (V, B) int32 device; rep (B) device array
 * of gaus_report, written.  Integer arithmetic only. */
gaus_status gaus_verify(gaus_ctx *ctx, const int32_t *sched, gaus_report *rep);

/* ---- Outer loop of Alg. GauS: initialization, sampling, legalization, best ---- */

/* Best legal schedule found per restart; device arrays owned by the caller. */
typedef struct {
  int32_t *sched;   /* (V, B) best legal schedule (caller node ids)               */
  double *score;    /* (B) its score; +inf while none was found                   */
  int32_t *iter;    /* (B) iteration count when it was found; -1 while none       */
} gaus_best;

/* Initialization of Alg. GauS (Sec. 3.3 Initialization): per node
 * sigma = max(kappa (ALAP - ASAP), sigma_min) (computed in double, rounded to
 * float) and mu = mu0 (device (V, B)) or, when mu0 is NULL, the midpoint
 * (ASAP + ALAP) / 2; Adam moments and step zeroed, lambda = lambda0, status OK.
 * sigma_init (V, B) device, written with that sigma (the value a reset returns
 * to), or NULL.  best (optional): score = +inf, iter = -1.  EINVAL on NULL state
 * pointers or kappa not finite and > 0. */
gaus_status gaus_init_state(gaus_ctx *ctx, const float *mu0, float kappa, const gaus_state *st, float *sigma_init,
                            const gaus_best *best);

/* One outer step of Alg. GauS on all B restarts (sampling and "legalize if
 * illegal"; App. A: the optimizer is reset to the prior best when the legalized
 * schedule does not improve on it).  Inputs (device): sched (V, B) = the
 * legalization of round(st->mu) and leg_status (B) from gaus_legalize, rep (B)
 * from gaus_verify of sched, sigma_init (V, B) from gaus_init_state; iter is
 * recorded with a new best.  Per restart:
 *   candidate: leg_status OK, rep.feasible, and rep.res_ok if GAUS_RES_VIOL is on;
 *     score = w_res L_res [RES_OBJ] + alpha L_com [COM] + w_mem (II > 0 ? L_mmem
 *     : L_mem) [REG_OBJ] (double);
 *   improved: a candidate with score < best score: best sched, score, iter set;
 *   illegal: some node of sched differs from round(mu), or legalization failed:
 *     reset mu to sched (Alg. GauS: mu <- legalize(s)) unless sched does not
 *     improve on an existing best (then that best), or legalization failed (then
 *     the best if any, else (ASAP + ALAP) / 2); sigma to sigma_init; Adam moments
 *     and step to 0; lambda kept.
 * moved (B) device, written: nodes legalization moved (-1 if it failed).
 * Asynchronous on the context's stream. */
gaus_status gaus_outer_step(gaus_ctx *ctx, const int32_t *sched, const int32_t *leg_status, const gaus_report *rep,
                            int32_t iter, const float *sigma_init, const gaus_state *st, const gaus_best *best,
                            int32_t *moved);

/* n_periods periods of Alg. GauS on the device, with no host synchronisation:
 * each runs `period` fused iterations (gaus_iterate), then gaus_legalize,
 * gaus_verify and gaus_outer_step (iteration count iter0 + (p + 1) period).
 * Work buffers (device, caller-owned, overwritten): sched (V, B) int32,
 * leg_status (B), rep (B), moved (B).  EINVAL on NULL pointers or counts < 1. */
gaus_status gaus_solve(gaus_ctx *ctx, int32_t n_periods, int32_t period, int32_t iter0, const gaus_state *st,
                       const float *sigma_init, const gaus_best *best, int32_t *sched, int32_t *leg_status,
                       gaus_report *rep, int32_t *moved);

/* Expected usage per resource class without allocating device memory.
 *
 * For callers that cannot call cudaMalloc -- code that runs inside a memory pool
 * or arena owned by another framework, allocation-free real-time loops, or hosts
 * whose device memory is budgeted before this library is used.  It needs no
 * context: the caller passes device arrays it already owns, and the only working
 * memory is a fixed 16 MiB array that the library keeps in device globals on every
 * GPU that loads it, until the process exits.  The paper has no counterpart; this
 * is the usage reduction of gaus_loss_grad offered on its own.
 *
 *   usage[b, c, t] = sum over nodes v of class c of demand[v] * P_v^d, summed over the
 *   bins d with d mod II = t (t < II) when II > 0, else d = t (t < D),
 * with P_v^d the mass the normal N(mu_v, sigma_v^2) rounds to step d, over the bins
 * within window_k * sigma of mu (the mass beyond them lumped into the end bins), in
 * exact fixed-point sums (deterministic), with the same bin-mass arithmetic as
 * gaus_loss_grad.
 *   mu, sigma (V, B) fp32, res_class (V) int32 in 0..C-1, demand (V) int32 or NULL
 *   (= 1): DEVICE pointers, read only.  A demand outside 0..64 is not added: the
 *   usage row (b, c) of every restart b that met it in class c is written as NaN.
 *   usage (B, C, II or D) fp64 DEVICE pointer, written.
 *   cuda_stream: cudaStream_t of the work (NULL = legacy default stream).
 * Limits: (II or D) * min(B, 32) <= 25,600; at most 1,024 (restart group, class)
 * pairs with groups of 32 restarts; the partial histograms of all blocks must fit
 * in the 16 MiB array (EINVAL with a message otherwise, nothing enqueued).  A
 * restart whose mean or sigma is non-finite (or sigma < 1e-30) contributes nothing.
 * The first call on a device looks up the array's device address and sets the
 * kernel's shared-memory limit; make that first call before any stream capture.  A
 * cudaDeviceReset of that device in the same process invalidates what it looked up:
 * do not call this entry point on the device again after such a reset.
 * Every call shares the array: calls whose work overlaps on the GPU race and give
 * undefined results.  No cudaMalloc, cudaFree or allocating library routine is
 * called.  Errors: EINVAL, ECUDA (message in gaus_last_error(NULL)). */
gaus_status gaus_expected_usage_noalloc(const float *mu, const float *sigma, const int32_t *res_class,
                                        const int32_t *demand, int32_t V, int32_t B, int32_t C, int32_t D,
                                        int32_t II, float window_k, double *usage, void *cuda_stream);

/* Measurement helper, not on the scheduling path: the throughput of this device's
 * FP32 FMA pipe (what = GAUS_PEAK_FP32; FLOP/s, an FMA counted as 2) or of its
 * special-function unit's exp2 (what = GAUS_PEAK_EX2; results/s), the two
 * arithmetic bounds of the node and edge passes.  A microbenchmark of independent
 * dependency chains on every SM (one wave of 256-thread blocks), best of three timed
 * runs after a warm-up, with CUDA events on `cuda_stream` (a cudaStream_t; NULL =
 * the legacy default stream), which it synchronises.  Allocates and frees 1 KiB of
 * device memory.  Errors: EINVAL (NULL per_second or unknown what), ECUDA. */
#define GAUS_PEAK_FP32 0
#define GAUS_PEAK_EX2  1
gaus_status gaus_measure_peak(int32_t what, double *per_second, void *cuda_stream);

/* Message of the last error on this context ("" if none), or with ctx = NULL the
 * message of this thread's last failed gaus_create or gaus_expected_usage_noalloc.
 * Valid until the next call. */
const char *gaus_last_error(const gaus_ctx *ctx);

/* Release the context and its device memory (synchronises its stream). */
void gaus_destroy(gaus_ctx *ctx);

#ifdef __cplusplus
}
#endif
#endif
