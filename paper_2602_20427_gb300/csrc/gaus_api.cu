// gaus_api.cu -- C ABI of the GauS hot path (include/gaus.h): context setup,
// launches, the captured iteration graph, and the integer entry points.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "gaus.h"
#include "gaus_int.cuh"
#include "gaus_internal.h"
#include "gaus_kernel_set.cuh"

using namespace gaus;

namespace {

thread_local std::string g_create_error;
constexpr size_t kMaxSmem = 227 * 1024;

gaus_status cuda_fail(gaus_ctx *ctx, cudaError_t e, const char *what) {
  if (ctx) ctx->err = std::string(what) + ": " + cudaGetErrorString(e);
  return e == cudaErrorMemoryAllocation ? GAUS_ENOMEM : GAUS_ECUDA;
}

#define CK(call, what)                                   \
  do {                                                   \
    cudaError_t e_ = (call);                             \
    if (e_ != cudaSuccess) return cuda_fail(ctx, e_, what); \
  } while (0)

template <typename T>
gaus_status upload(gaus_ctx *ctx, T **dst, const std::vector<T> &src) {
  size_t bytes = std::max<size_t>(sizeof(T), src.size() * sizeof(T));
  CK(cudaMalloc((void **)dst, bytes), "cudaMalloc");
  ctx->allocs.push_back(*dst);
  if (!src.empty()) CK(cudaMemcpy(*dst, src.data(), src.size() * sizeof(T), cudaMemcpyHostToDevice), "cudaMemcpy");
  return GAUS_OK;
}

template <typename T>
gaus_status scratch(gaus_ctx *ctx, T **dst, size_t count) {
  CK(cudaMalloc((void **)dst, std::max<size_t>(1, count) * sizeof(T)), "cudaMalloc scratch");
  ctx->allocs.push_back(*dst);
  CK(cudaMemset(*dst, 0, std::max<size_t>(1, count) * sizeof(T)), "cudaMemset");
  return GAUS_OK;
}

#define TRY(x)                           \
  do {                                   \
    gaus_status s_ = (x);                \
    if (s_ != GAUS_OK) return s_;        \
  } while (0)

IterArgs iter_args(gaus_ctx *ctx, const float *mu, const float *sg) {
  const Plan &P = ctx->plan;
  IterArgs A;
  A.mu = mu; A.sg = sg;
  A.V = P.V; A.B = P.B; A.D = P.D; A.II = P.II; A.Dh = P.Dh; A.C = P.C; A.RB = ctx->RB; A.G = ctx->G;
  A.W = ctx->W;
  A.k_win = ctx->k_win; A.alpha = ctx->hp.alpha;
  A.perm = ctx->d_perm; A.w = ctx->d_w; A.lat = ctx->d_lat;
  A.in_ptr = ctx->d_in_ptr; A.in_src = ctx->d_in_src; A.in_lat = ctx->d_in_lat;
  A.out_ptr = ctx->d_out_ptr; A.out_dst = ctx->d_out_dst;
  A.bin_ptr = ctx->d_bin_ptr; A.bin_src = ctx->d_bin_src; A.bin_shift = ctx->d_bin_shift;
  A.bout_ptr = ctx->d_bout_ptr; A.bout_dst = ctx->d_bout_dst; A.bout_shift = ctx->d_bout_shift;
  A.seg = ctx->d_seg; A.hpart = ctx->d_hpart; A.hspan = ctx->d_hspan; A.fwdtot = ctx->d_fwdtot;
  A.nonfinite = ctx->d_nonfinite; A.win = ctx->d_win; A.tab = ctx->d_tab;
  A.wstat = ctx->d_wstat;
  A.ed = ctx->d_ed; A.nEt = P.E + P.NB; A.ce = ctx->ce; A.E = P.E; A.eslot4 = ctx->d_eslot4;
  return A;
}

// The family-dependent kernels of a context's CDF family (the normal's are
// instantiated here, the others in their own translation units).
const KernelSet &kernels(int family) {
  static const KernelSet sets[4] = {make_kernel_set<GAUS_GAUSSIAN>(), kernel_set_logistic(), kernel_set_laplace(),
                                    kernel_set_cauchy()};
  return sets[(family >= GAUS_GAUSSIAN && family <= GAUS_CAUCHY) ? family : GAUS_GAUSSIAN];
}

// Enqueue loss + gradient (adam == false: gradient written to grad_*), or the
// fused iteration (adam == true: Adam on the state, lambda and step updated).
gaus_status enqueue_iteration(gaus_ctx *ctx, cudaStream_t st, const float *mu, const float *sg,
                              float *lambda, bool adam, float *grad_mu, float *grad_sg, float *loss,
                              float *terms, int32_t *status, const gaus_state *S,
                              cudaEvent_t *ev = nullptr) {
  if (ev) CK(cudaEventRecord(ev[0], st), "event");
  const Plan &P = ctx->plan;
  const unsigned on = ctx->hp.terms;
  IterArgs A = iter_args(ctx, mu, sg);
  const KernelSet &ks = kernels(ctx->hp.family);
  ks.nodes<<<ctx->nblk, kFwdThreads, ctx->smem_nodes, st>>>(A);
  CK(cudaGetLastError(), "k_nodes launch");
  if (ev) CK(cudaEventRecord(ev[1], st), "event");
  // usage reduction (needs only the node pass) on the side stream, beside the edge pass
  CK(cudaEventRecord(ctx->ev_fork, st), "fork");
  CK(cudaStreamWaitEvent(ctx->side, ctx->ev_fork, 0), "fork wait");
  {
    RedArgs R;
    R.B = P.B; R.C = P.C; R.Dh = P.Dh; R.RB = ctx->RB; R.G = ctx->G;
    R.cls_seg_ptr = ctx->d_cls_seg_ptr; R.hpart = ctx->d_hpart; R.hspan = ctx->d_hspan; R.U = ctx->d_U;
    k_reduce<<<ctx->red_blocks, 256, 0, ctx->side>>>(R);
    CK(cudaGetLastError(), "k_reduce launch");
  }
  CK(cudaEventRecord(ctx->ev_join, ctx->side), "join record");
  EdgeKernel ke = ks.edges[edge_variant(on, P.II, P.unit_lat != 0)];
  {
    // the edge pass at the device's greatest priority, so that its blocks start
    // ahead of the usage reduction's (which has until the finalize to finish)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)ctx->nblk_e);
    cfg.blockDim = dim3(kFwdThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributePriority;
    at[0].val.priority = ctx->prio_hi;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    CK(cudaLaunchKernelEx(&cfg, ke, A), "k_edges launch");
  }
  if (on & GAUS_DEP_CF) {
    k_dep_cf<<<ctx->nchunk * ctx->G, kFwdThreads, 0, st>>>(A);
    CK(cudaGetLastError(), "k_dep_cf launch");
  }
  if (ev) CK(cudaEventRecord(ev[2], st), "event");
  const bool reg = on & GAUS_REG_OBJ;
  RegArgs RA;
  if (reg) {
    RA.mu = mu; RA.sg = sg;
    RA.V = P.V; RA.B = P.B; RA.D = P.D; RA.II = P.II; RA.Dh = P.Dh; RA.RB = ctx->RBr; RA.G = ctx->Gr;
    RA.k_win = ctx->k_win; RA.perm = ctx->d_perm; RA.bits = ctx->d_bits;
    RA.out_ptr = ctx->d_out_ptr; RA.out_dst = ctx->d_out_dst; RA.seg = ctx->d_seg; RA.win = ctx->d_win;
    RA.qtab = ctx->d_qtab + (size_t)2 * kTailRows * ctx->hp.family;
    RA.tab = ctx->d_tab; RA.W = ctx->W; RA.ptab = ctx->d_ptab; RA.WP = ctx->WP;
    RA.rpart = ctx->d_rpart; RA.Hreg = ctx->d_Hreg; RA.gown = ctx->d_gown; RA.eslot = ctx->d_eslot;
    ks.reg_fwd<<<ctx->nblk_r, kFwdThreads, ctx->smem_rfwd, st>>>(RA);
    CK(cudaGetLastError(), "k_reg_fwd launch");
    k_reduce_reg<<<ctx->Gr * P.Dh, 256, 0, st>>>(ctx->d_rpart, ctx->d_Ureg, P.B, P.Dh, ctx->RBr, ctx->Gr,
                                                 P.nseg);
    CK(cudaGetLastError(), "k_reduce_reg launch");
  }
  // (k_reduce runs on the side stream, forked after k_nodes; joined here)
  CK(cudaStreamWaitEvent(st, ctx->ev_join, 0), "join");

  FinArgs F;
  F.B = P.B; F.C = P.C; F.Dh = P.Dh; F.RB = ctx->RB; F.G = ctx->G; F.Ug = ctx->d_U;
  F.Ureg = reg ? ctx->d_Ureg : nullptr; F.Hreg = ctx->d_Hreg;
  F.terms = on; F.tau = ctx->hp.tau; F.rho = ctx->hp.rho; F.alpha = ctx->hp.alpha;
  F.w_res = ctx->hp.w_res; F.w_mem = ctx->hp.w_mem;
  F.cls_seg_ptr = ctx->d_cls_seg_ptr; F.limit = ctx->d_limit;
  F.hpart = ctx->d_hpart; F.hspan = ctx->d_hspan; F.fwdtot = ctx->d_fwdtot;
  F.lambda = lambda; F.update_lambda = adam ? 1 : 0; F.step = adam ? S->step : nullptr;
  F.beta1 = ctx->hp.beta1; F.beta2 = ctx->hp.beta2;
  F.H = ctx->d_H; F.coef = ctx->d_coef; F.loss = loss; F.terms_out = terms;
  F.wstat = ctx->d_wstat; F.thr = ctx->d_thr; F.W = ctx->W;
  F.status = status; F.nonfinite = ctx->d_nonfinite;
  if (ctx->smem_fin > 0) k_finalize<true><<<P.B, 256, ctx->smem_fin, st>>>(F);
  else k_finalize<false><<<P.B, 256, 0, st>>>(F);
  CK(cudaGetLastError(), "k_finalize launch");
  if (reg) {
    ks.reg_bwd<<<ctx->nblk_r, kFwdThreads, ctx->smem_rbwd, st>>>(RA);
    CK(cudaGetLastError(), "k_reg_bwd launch");
  }
  if (ev) CK(cudaEventRecord(ev[3], st), "event");

  UpdArgs U;
  U.in_ptr = ctx->d_in_ptr; U.in_eslot = ctx->d_in_eslot; U.out_ptr = ctx->d_out_ptr;
  U.bin_ptr = ctx->d_bin_ptr; U.bout_ptr = ctx->d_bout_ptr;
  U.E = P.E; U.nEt = P.E + P.NB; U.has_back = (on & GAUS_REC) && P.II > 0 && P.NB > 0; U.eslot4 = ctx->d_eslot4;
  U.eslot = reg ? ctx->d_eslot : nullptr; U.gown = reg ? ctx->d_gown : nullptr;
  U.mu = const_cast<float *>(mu); U.sg = const_cast<float *>(sg);
  U.V = P.V; U.B = P.B; U.D = P.D; U.II = P.II; U.Dh = P.Dh; U.C = P.C; U.RB = ctx->RB; U.G = ctx->G;
  U.k_win = ctx->k_win; U.W = ctx->W; U.perm = ctx->d_perm; U.cls = ctx->d_cls; U.w = ctx->d_w;
  U.H = ctx->d_H; U.coef = ctx->d_coef; U.thr = ctx->d_thr;
  U.grad_mu = grad_mu; U.grad_sg = grad_sg;
  U.m_mu = adam ? S->m_mu : nullptr; U.v_mu = adam ? S->v_mu : nullptr;
  U.m_sg = adam ? S->m_sigma : nullptr; U.v_sg = adam ? S->v_sigma : nullptr;
  U.step_dev = adam ? S->step : nullptr;
  U.lr = ctx->hp.lr; U.beta1 = ctx->hp.beta1; U.beta2 = ctx->hp.beta2; U.eps = ctx->hp.eps;
  U.sigma_min = ctx->hp.sigma_min;
  const bool hist = on & (GAUS_RES_OBJ | GAUS_RES_VIOL);
  ks.update[2 * (adam ? 1 : 0) + (hist ? 1 : 0)]<<<ctx->nblk_u, kUpdThreads, 0, st>>>(U);
  CK(cudaGetLastError(), "k_update launch");
  if (ev) CK(cudaEventRecord(ev[4], st), "event");
  return GAUS_OK;
}

// The persistent kernel covers every term but the storage term and the continuous
// dependency penalty (those run on the multi-kernel path).
bool fused_ok(const gaus_ctx *ctx) {
  return ctx->fK > 0 && !(ctx->hp.terms & (GAUS_REG_OBJ | GAUS_DEP_CF));
}

// Window points of every (node, restart) of the state: their sum and maximum, for
// the per-call choice between the fused kernel and the multi-kernel path.
__global__ void __launch_bounds__(256) k_window_stats(const float *mu, const float *sg, size_t n, float k, int D,
                                                      unsigned long long *out) {
  unsigned long long sum = 0;
  unsigned mx = 0;
  for (size_t i = (size_t)blockIdx.x * 256 + threadIdx.x; i < n; i += (size_t)gridDim.x * 256) {
    const float m = mu[i], s = sg[i];
    int a = 0, b = -1;
    if (usable(m, s)) window(m, s, k, D, a, b);
    const unsigned w = (unsigned)max(b - a + 1, 0);
    sum += w;
    mx = max(mx, w);
  }
  for (int o = 16; o > 0; o >>= 1) {
    sum += __shfl_down_sync(0xffffffffu, sum, o);
    mx = max(mx, __shfl_down_sync(0xffffffffu, mx, o));
  }
  if ((threadIdx.x & 31) == 0) {
    atomicAdd(out, sum);
    atomicMax(out + 1, (unsigned long long)mx);
  }
}

// Enqueue n_iters fused iterations (adam) or one loss + gradient evaluation
// (!adam) as cooperative launches of the persistent kernel, one per batch of
// restart groups the device holds at once (a single launch unless B is huge).
gaus_status enqueue_fused(gaus_ctx *ctx, cudaStream_t st, int n_iters, bool adam, const float *mu, const float *sg,
                          float *m_mu, float *v_mu, float *m_sg, float *v_sg, float *lambda, int32_t *step,
                          float *grad_mu, float *grad_sg, float *loss, float *terms, int32_t *status,
                          unsigned long long *prof, unsigned bar_extra = 0,
                          unsigned long long bar_limit_ns = kBarrierTimeoutNs) {
  const Plan &P = ctx->plan;
  FusedArgs A;
  A.bar_extra = bar_extra;
  A.bar_limit_ns = bar_limit_ns;
  A.V = P.V; A.B = P.B; A.D = P.D; A.II = P.II; A.Dh = P.Dh; A.C = P.C; A.K = ctx->fK;
  A.RG = ctx->fRG; A.RBp = ctx->fRBp; A.RB1 = ctx->fRB1;
  A.W = ctx->fW; A.n_iters = n_iters; A.nseg = P.nfseg;
  A.k_win = ctx->k_win; A.alpha = ctx->hp.alpha; A.tau = ctx->hp.tau; A.rho = ctx->hp.rho; A.w_res = ctx->hp.w_res;
  A.lr = ctx->hp.lr; A.beta1 = ctx->hp.beta1; A.beta2 = ctx->hp.beta2; A.eps = ctx->hp.eps;
  A.sigma_min = ctx->hp.sigma_min; A.terms = ctx->hp.terms; A.adam = adam ? 1 : 0;
  A.perm = ctx->d_perm; A.w = ctx->d_w; A.lat = ctx->d_lat; A.cls = ctx->d_cls; A.seg = ctx->d_fseg;
  A.finc = ctx->d_finc; A.chunk = ctx->d_chunk; A.cptr = ctx->d_cptr;
  A.nchunk = P.nchunk;
  A.in_ptr = ctx->d_in_ptr; A.fin = ctx->d_fin; A.out_ptr = ctx->d_out_ptr; A.fout = ctx->d_fout;
  A.bin_ptr = ctx->d_bin_ptr; A.fbin = ctx->d_fbin; A.bout_ptr = ctx->d_bout_ptr; A.fbout = ctx->d_fbout;
  A.limit = ctx->d_limit;
  A.mu = const_cast<float *>(mu); A.sg = const_cast<float *>(sg);
  A.m_mu = m_mu; A.v_mu = v_mu; A.m_sg = m_sg; A.v_sg = v_sg;
  A.lambda = lambda; A.step = step; A.grad_mu = grad_mu; A.grad_sg = grad_sg;
  A.loss = loss; A.terms_out = terms; A.status = status;
  A.xs = ctx->d_xs; A.adm = ctx->d_adm; A.win = ctx->d_win; A.tab = ctx->d_tab; A.part = ctx->d_part;
  A.partr = ctx->d_partr; A.H = ctx->d_H;
  A.bar = reinterpret_cast<unsigned *>(ctx->d_facc);
  A.abort_flag = reinterpret_cast<int32_t *>(ctx->d_facc + ctx->off_abort);
  A.ctr = reinterpret_cast<unsigned *>(ctx->d_facc + ctx->off_ctr);
  A.U = reinterpret_cast<long long *>(ctx->d_facc + ctx->off_U);
  A.fwd = reinterpret_cast<unsigned long long *>(ctx->d_facc + ctx->off_fwd);
  A.wst = reinterpret_cast<unsigned long long *>(ctx->d_facc + ctx->off_wst);
  A.nonf = reinterpret_cast<int32_t *>(ctx->d_facc + ctx->off_nonf);
  A.rstat = ctx->d_rstat; A.prof = prof;
  const void *fn = (const void *)kernels(ctx->hp.family).fused[(ctx->hp.terms & GAUS_COM) ? 1 : 0];
  for (int g0 = 0; g0 < ctx->fG; g0 += ctx->fGl) {
    A.g0 = g0;
    A.G = std::min(ctx->fGl, ctx->fG - g0);
    A.ord = ctx->d_ord + (size_t)g0 * P.V * 64;
    CK(cudaMemsetAsync(ctx->d_facc, 0, ctx->facc_bytes, st), "fused memset");
    void *args[] = {(void *)&A};
    CK(cudaLaunchCooperativeKernel(fn, dim3((unsigned)(A.G * A.K)), dim3(kFusedThreads), args, ctx->smem_fused, st),
       "k_fused launch");
    if (prof) break;  // phase stamps: the first batch of groups
  }
  return GAUS_OK;
}

// Blocks per restart group and segments of the fused kernel: one wave of blocks of
// every family's and variant's kernel (so a family switch needs no re-plan), at
// most one segment per block; 0 when the sizes need the multi-kernel path.
gaus_status plan_fused(gaus_ctx *ctx, int nsm) {
  Plan &P = ctx->plan;
  ctx->fK = 0;
  if (P.D > 32767) return GAUS_OK;
  // groups of up to 64 restarts; phases 2-3 rows of RBp lanes; phase 1 rows of RB1
  // restarts, as many as keep its histogram within the staging buffer's size
  ctx->fRG = std::min(P.B, kMaxRG);
  ctx->fG = (P.B + ctx->fRG - 1) / ctx->fRG;
  ctx->fRBp = 32;  // one node per warp in phases 2 and 3
  const size_t stage = (size_t)kFusedWarps * kStage * 32 * sizeof(float2);
  // phase 1: the whole group's histogram when it fits the staging buffer, else rows
  // of a power of two <= 32 restarts
  if (2 * (size_t)ctx->fRG * P.Dh * sizeof(unsigned) <= stage) {
    ctx->fRB1 = ctx->fRG;
  } else {
    ctx->fRB1 = 32;
    while (ctx->fRB1 > 1 && 2 * (size_t)ctx->fRB1 * P.Dh * sizeof(unsigned) > stage) ctx->fRB1 >>= 1;
  }
  const size_t hist = 2 * (size_t)ctx->fRB1 * P.Dh * sizeof(unsigned);
  ctx->smem_fused = std::max(hist, stage);
  int dev = 0, optin = 0;
  CK(cudaGetDevice(&dev), "cudaGetDevice");
  CK(cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev), "smem opt-in");
  int occ = INT32_MAX;
  for (int fam = GAUS_GAUSSIAN; fam <= GAUS_CAUCHY; ++fam)
    for (int c = 0; c < 2; ++c) {
      const void *fn = (const void *)kernels(fam).fused[c];
      cudaFuncAttributes fa;
      CK(cudaFuncGetAttributes(&fa, fn), "cudaFuncGetAttributes");
      if (fa.sharedSizeBytes + ctx->smem_fused > (size_t)optin) return GAUS_OK;
      CK(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - (int)fa.sharedSizeBytes),
         "smem attr");
      int o = 0;
      CK(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, fn, kFusedThreads, ctx->smem_fused), "occupancy");
      occ = std::min(occ, o);
    }
  if (occ < 1) return GAUS_OK;
  const int resident = occ * nsm;
  if (ctx->fG <= resident) {
    const int per_group = resident / ctx->fG;
    // the fewest rows per segment that keep the segment count within one block each
    plan_fused_segments(P, per_group, ctx->fRB1);
    ctx->fK = std::min(per_group, P.nfseg);
    ctx->fGl = ctx->fG;
  } else {
    plan_fused_segments(P, 1, ctx->fRB1);
    ctx->fK = 1;
    ctx->fGl = resident;
  }
  return GAUS_OK;
}

// The dynamic shared-memory limit is a per-kernel attribute of the process, not of
// a context: set it to the device maximum once per kernel, so that contexts of
// different sizes can be used side by side (each launch still requests its own size).
gaus_status set_smem_attrs(gaus_ctx *ctx) {
  const KernelSet &ks = kernels(ctx->hp.family);
  const void *fns[] = {(const void *)ks.nodes, (const void *)k_finalize<true>, (const void *)ks.reg_fwd,
                       (const void *)ks.reg_bwd, (const void *)k_verify_fin, (const void *)k_legalize_regular_smem};
  int dev = 0, optin = 0;
  CK(cudaGetDevice(&dev), "cudaGetDevice");
  CK(cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev), "smem opt-in");
  std::vector<const void *> all(fns, fns + sizeof(fns) / sizeof(fns[0]));
  for (int c = 0; c < 2; ++c) all.push_back((const void *)ks.fused[c]);
  for (const void *f : all) {
    cudaFuncAttributes fa;
    CK(cudaFuncGetAttributes(&fa, f), "cudaFuncGetAttributes");
    CK(cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - (int)fa.sharedSizeBytes),
       "smem attr");
  }
  return GAUS_OK;
}

gaus_status alloc_storage_scratch(gaus_ctx *ctx);

gaus_status build_ctx(gaus_ctx *ctx, const gaus_problem *prob) {
  // Validate and plan on the host first: argument and graph errors never touch CUDA.
  int dev = 0, nsm = 152;
  const bool have_dev = cudaGetDevice(&dev) == cudaSuccess &&
                        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess;
  std::string err;
  ctx->nsm = nsm;
  gaus_status st = plan_problem(prob, 8 * nsm, &ctx->plan, &err);
  if (st != GAUS_OK) { ctx->err = err; return st; }
  Plan &P = ctx->plan;
  if ((ctx->hp.terms & GAUS_REC) && P.II <= 0) { ctx->err = "GAUS_REC needs II > 0"; return GAUS_EINVAL; }
  if (!have_dev) {
    cudaGetLastError();
    ctx->err = "no CUDA device";
    return GAUS_ECUDA;
  }
  // restarts per warp row: up to kMaxRB (8 with the storage term, whose workloads
  // measured faster with shorter rows), fewer for long horizons so that the node
  // pass's usage histogram (two u32 halves per bin and restart) fits shared memory
  const int max_rb = (ctx->hp.terms & GAUS_REG_OBJ) ? kMaxRB / 2 : kMaxRB;
  ctx->RB = 1;
  while (ctx->RB < P.B && ctx->RB < max_rb) ctx->RB <<= 1;
  while (ctx->RB > 1 && 2 * (size_t)ctx->RB * P.Dh * sizeof(unsigned) > kMaxSmem - 1024) ctx->RB >>= 1;
  ctx->G = (P.B + ctx->RB - 1) / ctx->RB;
  ctx->smem_nodes = 2 * (size_t)ctx->RB * P.Dh * sizeof(unsigned);
  if (ctx->smem_nodes > kMaxSmem - 1024) {
    ctx->err = "usage histogram of this horizon/II does not fit in shared memory";
    return GAUS_EINVAL;
  }
  TRY(set_smem_attrs(ctx));
  // Grids of the node, edge and update passes sized to one wave: the blocks the
  // device holds at once (occupancy calculator x SMs), so that no pass ends with a
  // partly filled second wave.
  const KernelSet &ks = kernels(ctx->hp.family);
  auto resident = [&](const void *fn, int threads, size_t smem) {
    int occ = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fn, threads, smem) != cudaSuccess) {
      cudaGetLastError();
      occ = 0;
    }
    return std::max(1, occ) * nsm;
  };
  plan_segments(P, resident((const void *)ks.nodes, kFwdThreads, ctx->smem_nodes), ctx->RB);
  ctx->nblk = P.nseg * ctx->G;
  // edge pass: one wave of blocks, the same number per restart group (rows of
  // edges grid-stride); k_dep_cf: one block per chunk of a warp pass per group
  {
    const int nEt = P.E + P.NB, per_pass = (kFwdThreads / 32) * (32 / ctx->RB);
    const void *ke = (const void *)ks.edges[edge_variant(ctx->hp.terms, P.II, P.unit_lat != 0)];
    ctx->ce = per_pass;
    ctx->nchunk = std::max(1, (nEt + per_pass - 1) / per_pass);
    const int per_group = std::max(1, std::min(ctx->nchunk, resident(ke, kFwdThreads, 0) / ctx->G));
    ctx->nblk_e = per_group * ctx->G;
  }
  // k_update: one warp-item (32 / RB nodes x one restart group) per warp
  {
    const long nwi = ((long)P.V + (32 / ctx->RB) - 1) / (32 / ctx->RB) * ctx->G;
    ctx->nblk_u = (int)std::max(1L, (nwi + kUpdThreads / 32 - 1) / (kUpdThreads / 32));
    ctx->nblk_u = std::min(ctx->nblk_u, resident((const void *)ks.update[3], kUpdThreads, 0));
  }
  ctx->red_blocks = ctx->G * P.C * P.Dh;
  // CDF table rows: up to kTableMax points per (node, restart), a multiple of 4,
  // with the table kept under kTableBytes (longer windows are evaluated directly)
  {
    const size_t per_pt = (size_t)P.V * P.B * sizeof(float);
    size_t w = std::min<size_t>(kTableMax, kTableBytes / per_pt);
    w = std::max<size_t>(4, w & ~(size_t)3);
    ctx->W = (int)w;
    // fused path: rows of up to kTableMaxFused entries, never longer than a window
    // can use (D - 1 points and the two sentinels)
    const size_t wf = std::min<size_t>(std::min<size_t>(kTableMaxFused, (size_t)P.D + 2), kTableBytesFused / per_pt);
    ctx->fW = (int)std::max<size_t>(4, wf);
  }
  // storage-term kernels: their own restarts-per-row, at most 4 (a row's loops over
  // successors and points run to the longest among its restarts; measured on the
  // loop-body and wide workloads), fewer where the storage histogram (two u32
  // halves), its difference array and constants would not fit in shared memory
  ctx->RBr = std::min(ctx->RB, 4);
  auto rfwd_bytes = [&](int rb) {
    return (2 * (size_t)P.Dh * rb + (size_t)(P.Dh + 1) * rb + rb) * sizeof(unsigned);
  };
  while (ctx->RBr > 1 && rfwd_bytes(ctx->RBr) > kMaxSmem - 1024) ctx->RBr >>= 1;
  if (rfwd_bytes(ctx->RBr) > kMaxSmem - 1024) {
    ctx->err = "storage histogram of this horizon/II does not fit in shared memory";
    return GAUS_EINVAL;
  }
  ctx->Gr = (P.B + ctx->RBr - 1) / ctx->RBr;
  ctx->nblk_r = P.nseg * ctx->Gr;
  ctx->smem_rfwd = rfwd_bytes(ctx->RBr);
  ctx->smem_rbwd = (size_t)P.Dh * ctx->RBr * sizeof(float);
  // finalize and verifier pass 2 stage a restart's rows in shared memory when they
  // fit (else the kernels read them in place)
  ctx->smem_fin = (size_t)(P.C + 1) * P.Dh * sizeof(double);
  ctx->smem_ver = ((size_t)P.C * P.Dh + (P.D + 1) + P.Dh) * sizeof(long long);
  if (ctx->smem_fin > kMaxSmem - 4096) ctx->smem_fin = 0;
  if (ctx->smem_ver > kMaxSmem - 1024) ctx->smem_ver = 0;
  ctx->smem_leg = (size_t)P.V * sizeof(int) <= kMaxSmem - 1024 ? (size_t)P.V * sizeof(int) : 0;
  CK(cudaStreamCreateWithFlags(&ctx->side, cudaStreamNonBlocking), "side stream");
  {
    int least = 0, greatest = 0;
    CK(cudaDeviceGetStreamPriorityRange(&least, &greatest), "priority range");
    ctx->prio_hi = greatest;
  }
  CK(cudaEventCreateWithFlags(&ctx->ev_fork, cudaEventDisableTiming), "event");
  CK(cudaEventCreateWithFlags(&ctx->ev_join, cudaEventDisableTiming), "event");

  TRY(upload(ctx, &ctx->d_perm, P.perm));
  TRY(upload(ctx, &ctx->d_w, P.w));
  TRY(upload(ctx, &ctx->d_bits, P.bits));
  TRY(upload(ctx, &ctx->d_limit, P.limit));
  TRY(upload(ctx, &ctx->d_lat, P.lat));
  TRY(upload(ctx, &ctx->d_cls, P.cls));
  TRY(upload(ctx, &ctx->d_in_ptr, P.in_ptr));
  TRY(upload(ctx, &ctx->d_in_src, P.in_src));
  TRY(upload(ctx, &ctx->d_in_lat, P.in_lat));
  TRY(upload(ctx, &ctx->d_out_ptr, P.out_ptr));
  TRY(upload(ctx, &ctx->d_out_dst, P.out_dst));
  TRY(upload(ctx, &ctx->d_in_eslot, P.in_eslot));
  {
    int32_t *ed = nullptr;
    TRY(upload(ctx, &ed, P.ed));
    ctx->d_ed = reinterpret_cast<int4 *>(ed);
  }
  TRY(upload(ctx, &ctx->d_bin_ptr, P.bin_ptr));
  TRY(upload(ctx, &ctx->d_bin_src, P.bin_src));
  TRY(upload(ctx, &ctx->d_bin_shift, P.bin_shift));
  TRY(upload(ctx, &ctx->d_bout_ptr, P.bout_ptr));
  TRY(upload(ctx, &ctx->d_bout_dst, P.bout_dst));
  TRY(upload(ctx, &ctx->d_bout_shift, P.bout_shift));
  TRY(upload(ctx, &ctx->d_seg, P.seg));
  TRY(upload(ctx, &ctx->d_cls_seg_ptr, P.cls_seg_ptr));
  TRY(upload(ctx, &ctx->d_lvl_ptr, P.lvl_ptr));
  TRY(upload(ctx, &ctx->d_lvl_nodes, P.lvl_nodes));
  TRY(upload(ctx, &ctx->d_lq_ptr, P.lq_ptr));
  TRY(upload(ctx, &ctx->d_lq_src, P.lq_src));
  TRY(upload(ctx, &ctx->d_lq_lat, P.lq_lat));
  TRY(upload(ctx, &ctx->d_cpred_ptr, P.cpred_ptr));
  TRY(upload(ctx, &ctx->d_cpred_src, P.cpred_src));
  TRY(upload(ctx, &ctx->d_csucc_ptr, P.csucc_ptr));
  TRY(upload(ctx, &ctx->d_csucc_dst, P.csucc_dst));
  TRY(upload(ctx, &ctx->d_cback_ptr, P.cback_ptr));
  TRY(upload(ctx, &ctx->d_cback_src, P.cback_src));
  TRY(upload(ctx, &ctx->d_cback_shift, P.cback_shift));
  TRY(upload(ctx, &ctx->d_c_lat, P.c_lat));
  TRY(upload(ctx, &ctx->d_c_cls, P.c_cls));
  TRY(upload(ctx, &ctx->d_c_dem, P.c_dem));
  TRY(upload(ctx, &ctx->d_c_bits, P.c_bits));
  TRY(upload(ctx, &ctx->d_e_src, P.e_src));
  TRY(upload(ctx, &ctx->d_e_dst, P.e_dst));
  TRY(upload(ctx, &ctx->d_b_src, P.b_src));
  TRY(upload(ctx, &ctx->d_b_dst, P.b_dst));
  TRY(upload(ctx, &ctx->d_b_dist, P.b_dist));
  TRY(upload(ctx, &ctx->d_asap, P.asap));
  TRY(upload(ctx, &ctx->d_alap, P.alap));

  const size_t VB = (size_t)P.V * P.B;
  TRY(scratch(ctx, &ctx->d_hpart, (size_t)ctx->nblk * ctx->RB * P.Dh));
  TRY(scratch(ctx, &ctx->d_U, (size_t)P.B * P.C * P.Dh));
  if (ctx->hp.terms & GAUS_REG_OBJ) TRY(alloc_storage_scratch(ctx));
  TRY(scratch(ctx, &ctx->d_hspan, (size_t)ctx->nblk));
  TRY(scratch(ctx, &ctx->d_fwdtot, (size_t)P.B * 3));
  // verifier: per-restart counts, usage counts and storage difference arrays
  ctx->vacc_words = (size_t)P.B * (4 + (size_t)P.C * P.Dh + (size_t)P.D + 1 + (size_t)P.Dh);
  TRY(scratch(ctx, &ctx->d_vacc, ctx->vacc_words));
  ctx->RBv = 1;
  while (ctx->RBv < P.B && ctx->RBv < 32) ctx->RBv <<= 1;
  ctx->Gv = (P.B + ctx->RBv - 1) / ctx->RBv;
  ctx->nblk_v = std::max(1, resident((const void *)k_verify_scan, 256, 0) / ctx->Gv) * ctx->Gv;
  TRY(scratch(ctx, &ctx->d_eslot4, 2 * ((size_t)P.E + P.NB) * P.B));
  TRY(scratch(ctx, &ctx->d_win, VB));
  TRY(scratch(ctx, &ctx->d_tab, VB * std::max(ctx->W, ctx->fW)));
  TRY(scratch(ctx, &ctx->d_H, (size_t)P.B * P.C * P.Dh));
  TRY(scratch(ctx, &ctx->d_coef, (size_t)P.B * 4));
  TRY(scratch(ctx, &ctx->d_wstat, (size_t)P.B * 2));
  TRY(scratch(ctx, &ctx->d_thr, (size_t)P.B));
  TRY(scratch(ctx, &ctx->d_decision, (size_t)P.B));
  TRY(scratch(ctx, &ctx->d_nonfinite, (size_t)P.B));
  TRY(scratch(ctx, &ctx->d_status_tmp, (size_t)P.B));
  TRY(scratch(ctx, &ctx->d_loss_tmp, (size_t)P.B));
  TRY(scratch(ctx, &ctx->d_terms_tmp, (size_t)P.B * GAUS_NT));
  TRY(scratch(ctx, &ctx->d_wsel, 2));
  CK(cudaMallocHost((void **)&ctx->h_wsel, 2 * sizeof(unsigned long long)), "cudaMallocHost");
  // fused persistent kernel
  TRY(plan_fused(ctx, nsm));
  if (ctx->fK > 0) {
    TRY(upload(ctx, &ctx->d_fseg, P.fseg));
    TRY(upload(ctx, &ctx->d_cptr, P.cptr));
    {
      int32_t *t4 = nullptr;
      TRY(upload(ctx, &t4, P.finc));
      ctx->d_finc = reinterpret_cast<int4 *>(t4);
      TRY(upload(ctx, &t4, P.chunk));
      ctx->d_chunk = reinterpret_cast<int4 *>(t4);
    }
    int32_t *tmp = nullptr;
    TRY(upload(ctx, &tmp, P.fout));
    ctx->d_fout = reinterpret_cast<int2 *>(tmp);
    TRY(upload(ctx, &tmp, P.fin));
    ctx->d_fin = reinterpret_cast<int2 *>(tmp);
    TRY(upload(ctx, &tmp, P.fbin));
    ctx->d_fbin = reinterpret_cast<int2 *>(tmp);
    TRY(upload(ctx, &tmp, P.fbout));
    ctx->d_fbout = reinterpret_cast<int2 *>(tmp);
    TRY(scratch(ctx, &ctx->d_xs, VB));
    TRY(scratch(ctx, &ctx->d_adm, VB));
    TRY(scratch(ctx, &ctx->d_part, (size_t)std::max(1, P.nchunk) * P.B));
    TRY(scratch(ctx, &ctx->d_partr, (size_t)std::max(1, P.nchunk) * P.B));
    TRY(scratch(ctx, &ctx->d_rstat, (size_t)P.B * 2));
    {
      // every node's restart order starts as the identity (restart l + 32 q in pass q)
      std::vector<signed char> ord((size_t)ctx->fG * P.V * 64);
      for (size_t i = 0; i < ord.size(); ++i) {
        const int r = (int)(i % 64);
        ord[i] = (signed char)(r < ctx->fRG ? r : -1);
      }
      TRY(upload(ctx, &ctx->d_ord, ord));
    }
    auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
    size_t off = al((size_t)ctx->fG * sizeof(unsigned));
    ctx->off_ctr = off; off = al(off + 2 * (size_t)ctx->fG * sizeof(unsigned));
    ctx->off_abort = off; off = al(off + sizeof(int32_t));
    ctx->off_U = off; off = al(off + 2 * (size_t)P.B * P.C * P.Dh * sizeof(long long));
    ctx->off_fwd = off; off = al(off + 2 * (size_t)P.B * 3 * sizeof(unsigned long long));
    ctx->off_wst = off; off = al(off + 2 * (size_t)P.B * 2 * sizeof(unsigned long long));
    ctx->off_nonf = off; off = al(off + 2 * (size_t)P.B * sizeof(int32_t));
    ctx->facc_bytes = off;
    TRY(scratch(ctx, &ctx->d_facc, ctx->facc_bytes));
  }
  CK(cudaDeviceSynchronize(), "setup sync");
  return GAUS_OK;
}

// Scratch of the storage term (also allocated when the term is switched on later).
gaus_status alloc_storage_scratch(gaus_ctx *ctx) {
  if (ctx->d_rpart) return GAUS_OK;
  const Plan &P = ctx->plan;
  TRY(scratch(ctx, &ctx->d_rpart, (size_t)ctx->nblk_r * P.Dh * ctx->RBr));
  TRY(scratch(ctx, &ctx->d_Ureg, (size_t)P.B * P.Dh));
  TRY(scratch(ctx, &ctx->d_Hreg, (size_t)P.B * P.Dh));
  TRY(scratch(ctx, &ctx->d_gown, (size_t)P.V * P.B));
  TRY(scratch(ctx, &ctx->d_eslot, (size_t)std::max(1, P.E) * P.B));
  TRY(scratch(ctx, &ctx->d_qtab, (size_t)2 * 4 * kTailRows));
  // rows of the successors' product for the backward: up to 32 points, 128 MB at most
  ctx->WP = (int)std::max<size_t>(4, std::min<size_t>(32, ((size_t)128 << 20) / ((size_t)P.V * P.B * sizeof(float))));
  TRY(scratch(ctx, &ctx->d_ptab, (size_t)P.V * P.B * ctx->WP));
  k_tail_tables<<<(4 * kTailRows + 255) / 256, 256, 0, ctx->stream>>>(ctx->d_qtab);
  CK(cudaGetLastError(), "k_tail_tables launch");
  CK(cudaStreamSynchronize(ctx->stream), "k_tail_tables sync");
  return GAUS_OK;
}

uint64_t state_hash(const gaus_state *s) {
  const void *p[] = {s->mu, s->sigma, s->m_mu, s->v_mu, s->m_sigma, s->v_sigma,
                     s->lambda, s->step, s->loss, s->terms, s->status};
  uint64_t h = 1469598103934665603ull;
  for (const void *x : p) {
    h ^= (uint64_t)(uintptr_t)x;
    h *= 1099511628211ull;
  }
  return h;
}

void drop_graph(gaus_ctx *ctx) {
  for (cudaGraphExec_t *g : {&ctx->gexec, &ctx->gexec_n}) {
    if (*g) cudaGraphExecDestroy(*g);
    *g = nullptr;
  }
  ctx->ghash = 0;
}

// Capture `iters` fused iterations into one executable graph.
gaus_status capture_iterations(gaus_ctx *ctx, const gaus_state *S, int iters, cudaGraphExec_t *out) {
  cudaStream_t cap;
  CK(cudaStreamCreateWithFlags(&cap, cudaStreamNonBlocking), "capture stream");
  cudaError_t e = cudaStreamBeginCapture(cap, cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) {
    cudaStreamDestroy(cap);
    return cuda_fail(ctx, e, "begin capture");
  }
  gaus_status st = GAUS_OK;
  for (int i = 0; i < iters && st == GAUS_OK; ++i)
    st = enqueue_iteration(ctx, cap, S->mu, S->sigma, S->lambda, true, nullptr, nullptr, S->loss, S->terms,
                           S->status, S);
  cudaGraph_t graph = nullptr;
  e = cudaStreamEndCapture(cap, &graph);
  cudaStreamDestroy(cap);
  if (st != GAUS_OK) {
    if (graph) cudaGraphDestroy(graph);
    return st;
  }
  if (e != cudaSuccess) return cuda_fail(ctx, e, "end capture");
  e = cudaGraphInstantiate(out, graph, cudaGraphInstantiateFlagUseNodePriority);
  cudaGraphDestroy(graph);
  if (e != cudaSuccess) {
    *out = nullptr;
    return cuda_fail(ctx, e, "graph instantiate");
  }
  return GAUS_OK;
}

// Per-block phase stamps of n_iters fused iterations, summarised (ms, means over
// the iterations): [0..2] critical path of phases 1-3 (last block done - first
// block started), [3..5] mean block time per phase, [6..7] barrier latency (last
// arrival to first release), [8] iteration time, [9..11] slowest block per phase.
gaus_status fused_phases(gaus_ctx *ctx, int n_iters, const gaus_state *S, double *out) {
  for (int k = 0; k < 12; ++k) out[k] = 0.0;
  if (n_iters <= 0) return GAUS_OK;
  const int nb = std::min(ctx->fGl, ctx->fG) * ctx->fK;
  const size_t need = (size_t)n_iters * nb * 6;
  if ((size_t)ctx->prof_cap < need) {
    if (ctx->d_prof) cudaFree(ctx->d_prof);
    ctx->d_prof = nullptr;
    ctx->prof_cap = 0;
    CK(cudaMalloc((void **)&ctx->d_prof, need * sizeof(unsigned long long)), "cudaMalloc prof");
    ctx->prof_cap = (int)need;
  }
  TRY(enqueue_fused(ctx, ctx->stream, n_iters, true, S->mu, S->sigma, S->m_mu, S->v_mu, S->m_sigma, S->v_sigma,
                    S->lambda, S->step, nullptr, nullptr, S->loss, S->terms, S->status, ctx->d_prof));
  std::vector<unsigned long long> ts(need);
  CK(cudaMemcpyAsync(ts.data(), ctx->d_prof, need * sizeof(unsigned long long), cudaMemcpyDeviceToHost, ctx->stream),
     "prof copy");
  CK(cudaStreamSynchronize(ctx->stream), "profile sync");
  auto at = [&](int it, int b, int q) { return (double)ts[((size_t)it * nb + b) * 6 + q]; };
  for (int it = 0; it < n_iters; ++it) {
    double mn[6], mx[6], sum[3] = {0, 0, 0}, wmx[3] = {0, 0, 0};
    for (int q = 0; q < 6; ++q) { mn[q] = 1e300; mx[q] = -1e300; }
    for (int b = 0; b < nb; ++b) {
      for (int q = 0; q < 6; ++q) { mn[q] = std::min(mn[q], at(it, b, q)); mx[q] = std::max(mx[q], at(it, b, q)); }
      for (int q = 0; q < 3; ++q) {
        const double w = at(it, b, 2 * q + 1) - at(it, b, 2 * q);
        sum[q] += w;
        wmx[q] = std::max(wmx[q], w);
      }
    }
    out[0] += mx[1] - mn[0];
    out[1] += mx[3] - mn[2];
    out[2] += mx[5] - mn[4];
    for (int q = 0; q < 3; ++q) { out[3 + q] += sum[q] / nb; out[9 + q] += wmx[q]; }
    out[6] += mn[2] - mx[1];
    out[7] += mn[4] - mx[3];
    double next = 0;
    if (it + 1 < n_iters) {
      next = 1e300;
      for (int b = 0; b < nb; ++b) next = std::min(next, at(it + 1, b, 0));
    } else {
      next = mx[5];
    }
    out[8] += next - mn[0];
  }
  for (int k = 0; k < 12; ++k) out[k] *= 1e-6 / n_iters;
  return GAUS_OK;
}

}  // namespace

namespace gaus {
// Message for gaus_last_error(NULL) from entry points that have no context.
void set_thread_error(const std::string &msg) { g_create_error = msg; }
}  // namespace gaus

extern "C" {

gaus_status gaus_default_hparams(gaus_hparams *hp) {
  if (!hp) return GAUS_EINVAL;
  hp->tau = 1e-2f;
  hp->rho = 1e-4f;
  hp->lambda0 = 1e-6f;
  hp->alpha = 1.0f;
  hp->w_res = 1.0f;
  hp->w_mem = 1.0f;
  hp->lr = 1e-2f;
  hp->beta1 = 0.9f;
  hp->beta2 = 0.999f;
  hp->eps = 1e-8f;
  hp->window_k = 6.0f;
  hp->sigma_min = 0.05f;
  hp->terms = GAUS_DEP | GAUS_COM | GAUS_RES_OBJ;
  hp->family = GAUS_GAUSSIAN;
  return GAUS_OK;
}

gaus_status gaus_create(const gaus_problem *prob, const gaus_hparams *hp, void *cuda_stream, gaus_ctx **out) {
  if (!out) return GAUS_EINVAL;
  *out = nullptr;
  std::string err;
  gaus_status st = check_hparams(hp, &err);
  if (st != GAUS_OK) {
    g_create_error = err;
    return st;
  }
  gaus_ctx *ctx = new (std::nothrow) gaus_ctx();
  if (!ctx) return GAUS_ENOMEM;
  ctx->hp = *hp;
  ctx->k_win = family_window_k(hp->window_k, hp->family);
  ctx->stream = (cudaStream_t)cuda_stream;
  st = build_ctx(ctx, prob);
  if (st != GAUS_OK) {
    g_create_error = ctx->err;
    gaus_destroy(ctx);
    return st;
  }
  *out = ctx;
  return GAUS_OK;
}

gaus_status gaus_set_hparams(gaus_ctx *ctx, const gaus_hparams *hp) {
  if (!ctx) return GAUS_EINVAL;
  gaus_status st = check_hparams(hp, &ctx->err);
  if (st != GAUS_OK) return st;
  if ((hp->terms & GAUS_REC) && ctx->plan.II <= 0) { ctx->err = "GAUS_REC needs II > 0"; return GAUS_EINVAL; }
  if (hp->terms & GAUS_REG_OBJ) {
    gaus_status st2 = alloc_storage_scratch(ctx);
    if (st2 != GAUS_OK) return st2;
  }
  const int old_family = ctx->hp.family;
  ctx->hp = *hp;
  ctx->k_win = family_window_k(hp->window_k, hp->family);
  drop_graph(ctx);
  if (hp->family != old_family) return set_smem_attrs(ctx);
  return GAUS_OK;
}

gaus_status gaus_check_barrier_timeout(gaus_ctx *ctx, const gaus_state *S, uint64_t limit_ns) {
  if (!ctx) return GAUS_EINVAL;
  if (!S || !S->mu || !S->sigma || !S->m_mu || !S->v_mu || !S->m_sigma || !S->v_sigma || !S->lambda ||
      !S->step || !S->loss || !S->terms || !S->status || limit_ns < 1000 || limit_ns > 1000000000ull) {
    ctx->err = "gaus_check_barrier_timeout: NULL state pointer or limit outside 1 us .. 1 s";
    return GAUS_EINVAL;
  }
  if (!fused_ok(ctx)) {
    ctx->err = "gaus_check_barrier_timeout: the context runs the multi-kernel path";
    return GAUS_EINVAL;
  }
  return enqueue_fused(ctx, ctx->stream, 1, true, S->mu, S->sigma, S->m_mu, S->v_mu, S->m_sigma, S->v_sigma,
                       S->lambda, S->step, nullptr, nullptr, S->loss, S->terms, S->status, nullptr, 1u,
                       (unsigned long long)limit_ns);
}

gaus_status gaus_plan_info(const gaus_ctx *ctx, int64_t *out, int32_t n) {
  if (!ctx || !out || n < 1) return GAUS_EINVAL;
  const Plan &P = ctx->plan;
  const bool fused = fused_ok(ctx);
  const unsigned on = ctx->hp.terms;
  const int64_t per_iter = 5 + ((on & GAUS_DEP_CF) ? 1 : 0) + ((on & GAUS_REG_OBJ) ? 3 : 0);
  const int64_t v[16] = {fused ? 1 : 0,
                         fused ? (ctx->fG + ctx->fGl - 1) / std::max(1, ctx->fGl) : 0,
                         per_iter,
                         ctx->fG, ctx->fK, ctx->fRG, ctx->fW, (int64_t)ctx->smem_fused, ctx->nsm,
                         P.nfseg, P.nchunk, kFusedThreads, ctx->path_mode, ctx->n_fused_calls,
                         ctx->n_multi_iters, ctx->n_path_stats};
  for (int i = 0; i < std::min(n, 16); ++i) out[i] = v[i];
  return GAUS_OK;
}

gaus_status gaus_set_path(gaus_ctx *ctx, int32_t mode) {
  if (!ctx) return GAUS_EINVAL;
  if (mode < GAUS_PATH_AUTO || mode > GAUS_PATH_MULTI) {
    ctx->err = "gaus_set_path: mode must be GAUS_PATH_AUTO, GAUS_PATH_FUSED or GAUS_PATH_MULTI";
    return GAUS_EINVAL;
  }
  ctx->path_mode = mode;
  return GAUS_OK;
}

gaus_status gaus_bounds(const gaus_ctx *ctx, int32_t *asap, int32_t *alap, int32_t *cp) {
  if (!ctx) return GAUS_EINVAL;
  const Plan &P = ctx->plan;
  if (asap) std::memcpy(asap, P.asap.data(), sizeof(int32_t) * P.V);
  if (alap) std::memcpy(alap, P.alap.data(), sizeof(int32_t) * P.V);
  if (cp) *cp = P.cp;
  return GAUS_OK;
}

gaus_status gaus_loss_grad(gaus_ctx *ctx, const float *mu, const float *sigma, const float *lambda,
                           float *grad_mu, float *grad_sigma, float *loss, float *terms, int32_t *status) {
  if (!ctx) return GAUS_EINVAL;
  if (!mu || !sigma || !lambda || !grad_mu || !grad_sigma || !loss || !terms) {
    ctx->err = "gaus_loss_grad: NULL pointer";
    return GAUS_EINVAL;
  }
  // the fused kernel unless MULTI is set, or AUTO's size rule picks the multi-kernel
  // path (restart groups of fewer than 64 on a problem of 16,384 items or more)
  const bool small_groups = ctx->path_mode == GAUS_PATH_AUTO && ctx->fRG < 64 &&
                            (size_t)ctx->plan.V * ctx->plan.B >= 16384;
  if (fused_ok(ctx) && ctx->path_mode != GAUS_PATH_MULTI && !small_groups)
    return enqueue_fused(ctx, ctx->stream, 1, false, mu, sigma, nullptr, nullptr, nullptr, nullptr,
                         const_cast<float *>(lambda), nullptr, grad_mu, grad_sigma, loss, terms,
                         status ? status : ctx->d_status_tmp, nullptr);
  return enqueue_iteration(ctx, ctx->stream, mu, sigma, const_cast<float *>(lambda), false, grad_mu, grad_sigma,
                           loss, terms, status ? status : ctx->d_status_tmp, nullptr);
}

gaus_status gaus_adam_step(gaus_ctx *ctx, float *mu, float *sigma, const float *grad_mu, const float *grad_sigma,
                           float *m_mu, float *v_mu, float *m_sigma, float *v_sigma, float *lambda,
                           const float *terms, int32_t step) {
  if (!ctx) return GAUS_EINVAL;
  if (!mu || !sigma || !grad_mu || !grad_sigma || !m_mu || !v_mu || !m_sigma || !v_sigma || !lambda || !terms ||
      step < 1) {
    ctx->err = "gaus_adam_step: NULL pointer or step < 1";
    return GAUS_EINVAL;
  }
  const size_t n = (size_t)ctx->plan.V * ctx->plan.B;
  const gaus_hparams &h = ctx->hp;
  int blocks = (int)std::min<size_t>((n + 255) / 256, 4096);
  k_adam<<<blocks, 256, 0, ctx->stream>>>(mu, sigma, grad_mu, grad_sigma, m_mu, v_mu, m_sigma, v_sigma, n, step,
                                          h.lr, h.beta1, h.beta2, h.eps, h.sigma_min);
  CK(cudaGetLastError(), "k_adam launch");
  k_lambda<<<(ctx->plan.B + 127) / 128, 128, 0, ctx->stream>>>(lambda, terms, ctx->plan.B, h.terms, h.rho);
  CK(cudaGetLastError(), "k_lambda launch");
  return GAUS_OK;
}

// The path of one gaus_iterate call (gaus_set_path).  The fused kernel wins where the
// windows are short (under a point on average: its one launch per call and node-side
// edges beat the five kernels per iteration) or uniform and within its 32-point
// staging (as at a uniform initial sigma); the multi-kernel path wins where windows
// vary across restarts or exceed the staging (the fused kernel's long items go one
// warp at a time): measured on the logic-network workload along a 2,000-iteration
// normal-family run and the logistic and kappa-initialized regimes.  Two cases are
// decided by the sizes alone, with no reduction: problems of fewer than 16,384
// (node, restart) items run the fused kernel (they are bound by launch latency, and
// it is one launch per call), and restart groups of fewer than 64 restarts the
// multi-kernel path (the fused kernel's phases 2 and 3 take one node per warp, so a
// smaller group leaves lanes idle, where the multi-kernel path packs two nodes per
// warp): measured with the logic-network DAG at B = 16 and 32 and the tiny DAG at B = 1.
static gaus_status choose_path(gaus_ctx *ctx, const float *mu, const float *sg, bool *fused) {
  *fused = false;
  if (!fused_ok(ctx) || ctx->path_mode == GAUS_PATH_MULTI) return GAUS_OK;
  *fused = true;
  if (ctx->path_mode == GAUS_PATH_FUSED) return GAUS_OK;
  const Plan &P = ctx->plan;
  const size_t n = (size_t)P.V * P.B;
  if (n < 16384) return GAUS_OK;
  if (ctx->fRG < 64) {
    *fused = false;
    return GAUS_OK;
  }
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  CK(cudaStreamIsCapturing(ctx->stream, &cs), "cudaStreamIsCapturing");
  if (cs != cudaStreamCaptureStatusNone) return GAUS_OK;
  CK(cudaMemsetAsync(ctx->d_wsel, 0, 2 * sizeof(unsigned long long), ctx->stream), "path memset");
  const int blocks = (int)std::min<size_t>((n + 255) / 256, (size_t)2 * std::max(1, ctx->nsm));
  k_window_stats<<<blocks, 256, 0, ctx->stream>>>(mu, sg, n, ctx->k_win, P.D, ctx->d_wsel);
  CK(cudaGetLastError(), "k_window_stats launch");
  CK(cudaMemcpyAsync(ctx->h_wsel, ctx->d_wsel, 2 * sizeof(unsigned long long), cudaMemcpyDeviceToHost, ctx->stream),
     "path copy");
  CK(cudaStreamSynchronize(ctx->stream), "path sync");
  ++ctx->n_path_stats;
  const double mean = (double)ctx->h_wsel[0] / (double)n;
  const double mx = (double)ctx->h_wsel[1];
  *fused = mean < 1.0 || (mx <= (double)kStage && mx <= 2.0 * mean);
  return GAUS_OK;
}

gaus_status gaus_iterate(gaus_ctx *ctx, int32_t n_iters, const gaus_state *S) {
  if (!ctx) return GAUS_EINVAL;
  if (!S || n_iters < 0 || !S->mu || !S->sigma || !S->m_mu || !S->v_mu || !S->m_sigma || !S->v_sigma ||
      !S->lambda || !S->step || !S->loss || !S->terms || !S->status) {
    ctx->err = "gaus_iterate: NULL state pointer or n_iters < 0";
    return GAUS_EINVAL;
  }
  if (n_iters == 0) return GAUS_OK;
  bool fused = false;
  TRY(choose_path(ctx, S->mu, S->sigma, &fused));
  if (fused) {
    ++ctx->n_fused_calls;
    return enqueue_fused(ctx, ctx->stream, n_iters, true, S->mu, S->sigma, S->m_mu, S->v_mu, S->m_sigma, S->v_sigma,
                         S->lambda, S->step, nullptr, nullptr, S->loss, S->terms, S->status, nullptr);
  }
  ctx->n_multi_iters += n_iters;
  // two captured graphs of the same iteration: kGraphUnroll iterations, and one
  const uint64_t h = state_hash(S);
  if (!ctx->gexec || ctx->ghash != h) {
    drop_graph(ctx);
    TRY(capture_iterations(ctx, S, 1, &ctx->gexec));
    TRY(capture_iterations(ctx, S, kGraphUnroll, &ctx->gexec_n));
    ctx->ghash = h;
  }
  int left = n_iters;
  for (; left >= kGraphUnroll; left -= kGraphUnroll) CK(cudaGraphLaunch(ctx->gexec_n, ctx->stream), "graph launch");
  for (; left > 0; --left) CK(cudaGraphLaunch(ctx->gexec, ctx->stream), "graph launch");
  return GAUS_OK;
}

gaus_status gaus_profile_iterate(gaus_ctx *ctx, int32_t n_iters, const gaus_state *S, double *ms_out) {
  if (!ctx) return GAUS_EINVAL;
  if (!S || !ms_out || n_iters < 0 || !S->mu || !S->sigma || !S->m_mu || !S->v_mu || !S->m_sigma ||
      !S->v_sigma || !S->lambda || !S->step || !S->loss || !S->terms || !S->status) {
    ctx->err = "gaus_profile_iterate: NULL pointer or n_iters < 0";
    return GAUS_EINVAL;
  }
  bool fused = false;
  TRY(choose_path(ctx, S->mu, S->sigma, &fused));
  if (fused) {
    double ph[12];
    TRY(fused_phases(ctx, n_iters, S, ph));
    // iteration start to the first barrier's release, to the second's, to the next start
    ms_out[0] += ph[0] + ph[6];
    ms_out[1] += ph[1] + ph[7];
    ms_out[3] += ph[8] - (ph[0] + ph[6]) - (ph[1] + ph[7]);
    return GAUS_OK;
  }
  constexpr int kEv = 5;  // before k_nodes, before / after k_edges, after finalize, after update
  std::vector<cudaEvent_t> ev(kEv * (size_t)n_iters);
  for (auto &e : ev) CK(cudaEventCreate(&e), "event create");
  gaus_status st = GAUS_OK;
  for (int i = 0; i < n_iters && st == GAUS_OK; ++i)
    st = enqueue_iteration(ctx, ctx->stream, S->mu, S->sigma, S->lambda, true, nullptr, nullptr, S->loss,
                           S->terms, S->status, S, &ev[kEv * (size_t)i]);
  cudaError_t e = cudaStreamSynchronize(ctx->stream);
  double acc[kEv - 1] = {0, 0, 0, 0};
  for (int i = 0; i < n_iters && st == GAUS_OK && e == cudaSuccess; ++i)
    for (int k = 0; k < kEv - 1; ++k) {
      float ms = 0.f;
      cudaEventElapsedTime(&ms, ev[kEv * (size_t)i + k], ev[kEv * (size_t)i + k + 1]);
      acc[k] += ms;
    }
  for (auto &x : ev) cudaEventDestroy(x);
  if (st != GAUS_OK) return st;
  if (e != cudaSuccess) return cuda_fail(ctx, e, "profile sync");
  for (int k = 0; k < kEv - 1; ++k) ms_out[k] += n_iters ? acc[k] / n_iters : 0.0;
  return GAUS_OK;
}

gaus_status gaus_profile_phases(gaus_ctx *ctx, int32_t n_iters, const gaus_state *S, double *out) {
  if (!ctx) return GAUS_EINVAL;
  if (!S || !out || n_iters < 0 || !S->mu || !S->sigma || !S->m_mu || !S->v_mu || !S->m_sigma || !S->v_sigma ||
      !S->lambda || !S->step || !S->loss || !S->terms || !S->status) {
    ctx->err = "gaus_profile_phases: NULL pointer or n_iters < 0";
    return GAUS_EINVAL;
  }
  if (!fused_ok(ctx)) {
    ctx->err = "gaus_profile_phases: these terms or sizes run the multi-kernel path";
    return GAUS_EINVAL;
  }
  return fused_phases(ctx, n_iters, S, out);
}

gaus_status gaus_round(gaus_ctx *ctx, const float *mu, int32_t *sched) {
  if (!ctx) return GAUS_EINVAL;
  if (!mu || !sched) { ctx->err = "gaus_round: NULL pointer"; return GAUS_EINVAL; }
  const size_t n = (size_t)ctx->plan.V * ctx->plan.B;
  k_round<<<(int)std::min<size_t>((n + 255) / 256, 4096), 256, 0, ctx->stream>>>(mu, sched, n);
  CK(cudaGetLastError(), "k_round launch");
  return GAUS_OK;
}

gaus_status gaus_legalize(gaus_ctx *ctx, const float *mu, int32_t *sched, int32_t *status) {
  if (!ctx) return GAUS_EINVAL;
  if (!mu || !sched || !status) { ctx->err = "gaus_legalize: NULL pointer"; return GAUS_EINVAL; }
  const Plan &P = ctx->plan;
  LegArgs A;
  A.mu = mu; A.s = sched; A.status = status;
  A.V = P.V; A.B = P.B; A.D = P.D; A.II = P.II; A.nlvl = P.nlvl;
  A.lvl_ptr = ctx->d_lvl_ptr; A.lvl_nodes = ctx->d_lvl_nodes;
  A.pred_ptr = ctx->d_cpred_ptr; A.pred_src = ctx->d_cpred_src; A.lat = ctx->d_c_lat;
  A.back_ptr = ctx->d_cback_ptr; A.back_src = ctx->d_cback_src; A.back_shift = ctx->d_cback_shift;
  A.asap = ctx->d_asap; A.alap = ctx->d_alap;
  A.lq_ptr = ctx->d_lq_ptr; A.lq_src = ctx->d_lq_src; A.lq_lat = ctx->d_lq_lat;
  const int grid = (P.B + 31) / 32;
  if (P.II > 0) k_legalize_modulo<<<grid, 256, 0, ctx->stream>>>(A);
  else if (ctx->smem_leg) k_legalize_regular_smem<<<P.B, 512, ctx->smem_leg, ctx->stream>>>(A);
  else k_legalize_regular<<<grid, 256, 0, ctx->stream>>>(A);
  CK(cudaGetLastError(), "legalize launch");
  return GAUS_OK;
}

gaus_status gaus_verify(gaus_ctx *ctx, const int32_t *sched, gaus_report *rep) {
  if (!ctx) return GAUS_EINVAL;
  if (!sched || !rep) { ctx->err = "gaus_verify: NULL pointer"; return GAUS_EINVAL; }
  const Plan &P = ctx->plan;
  VerArgs A;
  A.s = sched; A.rep = rep;
  A.V = P.V; A.E = P.E; A.NB = P.NB; A.B = P.B; A.C = P.C; A.D = P.D; A.II = P.II; A.Dh = P.Dh;
  A.e_src = ctx->d_e_src; A.e_dst = ctx->d_e_dst; A.lat = ctx->d_c_lat; A.cls = ctx->d_c_cls;
  A.dem = ctx->d_c_dem; A.bits = ctx->d_c_bits;
  A.b_src = ctx->d_b_src; A.b_dst = ctx->d_b_dst; A.b_dist = ctx->d_b_dist;
  A.succ_ptr = ctx->d_csucc_ptr; A.succ_dst = ctx->d_csucc_dst; A.limit = ctx->d_limit;
  A.RB = ctx->RBv; A.G = ctx->Gv;
  A.vacc = ctx->d_vacc;
  A.vcnt = A.vacc + (size_t)P.B * 4;
  A.vdiff = A.vcnt + (size_t)P.B * P.C * P.Dh;
  A.vmm = reinterpret_cast<long long *>(A.vdiff + (size_t)P.B * (P.D + 1));
  A.vsmem = ctx->smem_ver > 0;
  CK(cudaMemsetAsync(ctx->d_vacc, 0, ctx->vacc_words * sizeof(unsigned long long), ctx->stream), "verify memset");
  k_verify_scan<<<ctx->nblk_v, 256, 0, ctx->stream>>>(A);
  CK(cudaGetLastError(), "k_verify_scan launch");
  k_verify_fin<<<P.B, 256, ctx->smem_ver, ctx->stream>>>(A);
  CK(cudaGetLastError(), "k_verify_fin launch");
  return GAUS_OK;
}

gaus_status gaus_init_state(gaus_ctx *ctx, const float *mu0, float kappa, const gaus_state *S, float *sigma_init,
                            const gaus_best *best) {
  if (!ctx) return GAUS_EINVAL;
  if (!S || !S->mu || !S->sigma || !S->m_mu || !S->v_mu || !S->m_sigma || !S->v_sigma || !S->lambda || !S->step ||
      !S->status || !std::isfinite(kappa) || !(kappa > 0.0f)) {
    ctx->err = "gaus_init_state: NULL state pointer or kappa not finite and > 0";
    return GAUS_EINVAL;
  }
  const Plan &P = ctx->plan;
  const size_t n = (size_t)P.V * P.B;
  k_init_state<<<(int)std::min<size_t>((n + 255) / 256, 4096), 256, 0, ctx->stream>>>(
      mu0, S->mu, S->sigma, sigma_init, S->m_mu, S->v_mu, S->m_sigma, S->v_sigma, ctx->d_asap, ctx->d_alap, P.V, P.B,
      (double)kappa, ctx->hp.sigma_min);
  CK(cudaGetLastError(), "k_init_state launch");
  k_init_restart<<<(P.B + 127) / 128, 128, 0, ctx->stream>>>(S->lambda, S->step, S->status,
                                                                best ? best->score : nullptr,
                                                                best ? best->iter : nullptr, P.B, ctx->hp.lambda0);
  CK(cudaGetLastError(), "k_init_restart launch");
  return GAUS_OK;
}

gaus_status gaus_outer_step(gaus_ctx *ctx, const int32_t *sched, const int32_t *leg_status, const gaus_report *rep,
                            int32_t iter, const float *sigma_init, const gaus_state *S, const gaus_best *best,
                            int32_t *moved) {
  if (!ctx) return GAUS_EINVAL;
  if (!sched || !leg_status || !rep || !sigma_init || !S || !S->mu || !S->sigma || !S->m_mu || !S->v_mu ||
      !S->m_sigma || !S->v_sigma || !S->step || !best || !best->sched || !best->score || !best->iter || !moved) {
    ctx->err = "gaus_outer_step: NULL pointer";
    return GAUS_EINVAL;
  }
  const Plan &P = ctx->plan;
  OuterArgs O;
  O.sched = sched; O.leg_status = leg_status; O.rep = rep; O.mu = S->mu;
  O.V = P.V; O.B = P.B; O.II = P.II; O.iter = iter; O.terms = ctx->hp.terms;
  O.w_res = ctx->hp.w_res; O.alpha = ctx->hp.alpha; O.w_mem = ctx->hp.w_mem;
  O.best_score = best->score; O.best_iter = best->iter; O.step = S->step; O.moved = moved;
  O.decision = ctx->d_decision;
  k_outer_decide<<<P.B, 256, 0, ctx->stream>>>(O);
  CK(cudaGetLastError(), "k_outer_decide launch");
  const size_t n = (size_t)P.V * P.B;
  k_outer_apply<<<(int)std::min<size_t>((n + 255) / 256, 4096), 256, 0, ctx->stream>>>(
      ctx->d_decision, sched, best->sched, S->mu, S->sigma, sigma_init, S->m_mu, S->v_mu, S->m_sigma, S->v_sigma,
      ctx->d_asap, ctx->d_alap, P.V, P.B);
  CK(cudaGetLastError(), "k_outer_apply launch");
  return GAUS_OK;
}

gaus_status gaus_solve(gaus_ctx *ctx, int32_t n_periods, int32_t period, int32_t iter0, const gaus_state *S,
                       const float *sigma_init, const gaus_best *best, int32_t *sched, int32_t *leg_status,
                       gaus_report *rep, int32_t *moved) {
  if (!ctx) return GAUS_EINVAL;
  if (n_periods < 1 || period < 1 || !S || !sigma_init || !best || !sched || !leg_status || !rep || !moved) {
    ctx->err = "gaus_solve: NULL pointer or n_periods, period < 1";
    return GAUS_EINVAL;
  }
  for (int32_t p = 0; p < n_periods; ++p) {
    gaus_status st = gaus_iterate(ctx, period, S);
    if (st == GAUS_OK) st = gaus_legalize(ctx, S->mu, sched, leg_status);
    if (st == GAUS_OK) st = gaus_verify(ctx, sched, rep);
    if (st == GAUS_OK)
      st = gaus_outer_step(ctx, sched, leg_status, rep, iter0 + (p + 1) * period, sigma_init, S, best, moved);
    if (st != GAUS_OK) return st;
  }
  return GAUS_OK;
}

const char *gaus_last_error(const gaus_ctx *ctx) { return ctx ? ctx->err.c_str() : g_create_error.c_str(); }

void gaus_destroy(gaus_ctx *ctx) {
  if (!ctx) return;
  if (!ctx->allocs.empty() || ctx->gexec || ctx->gexec_n) {
    if (ctx->stream) cudaStreamSynchronize(ctx->stream);
    else cudaDeviceSynchronize();
  }
  drop_graph(ctx);
  if (ctx->side) cudaStreamSynchronize(ctx->side);
  for (void *p : ctx->allocs) cudaFree(p);
  if (ctx->d_prof) cudaFree(ctx->d_prof);
  if (ctx->h_wsel) cudaFreeHost(ctx->h_wsel);
  if (ctx->ev_fork) cudaEventDestroy(ctx->ev_fork);
  if (ctx->ev_join) cudaEventDestroy(ctx->ev_join);
  if (ctx->side) cudaStreamDestroy(ctx->side);
  delete ctx;
}

}  // extern "C"
