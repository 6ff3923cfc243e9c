// gaus_internal.h -- context layout shared by the host planner and the CUDA code.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "gaus.h"

namespace gaus {

// Threads per block of the node and edge passes and of the update kernel.
constexpr int kFwdThreads = 256;
constexpr int kUpdThreads = 256;
constexpr int kGraphUnroll = 10;               // iterations per captured graph
constexpr int kReduceSpans = 1024;             // segment spans staged per k_reduce pass
// Restarts per warp row of the node, edge and update passes (a power of two <= 32):
// lanes = (item, restart), 32 / kMaxRB items per warp.  Fewer restarts per row
// means each warp's loops run to the longest window of fewer restarts.
constexpr int kMaxRB = 16;
constexpr int kTableMax = 32;                    // points per CDF table row, at most
constexpr size_t kTableBytes = (size_t)64 << 20;  // CDF table size bound
// The fused kernel's table ([node][point][restart]: a row's entries are B floats
// apart, so a longer row costs address space, not cache lines): up to 64 points
// per row and 256 MB.
constexpr int kTableMaxFused = 64;
constexpr size_t kTableBytesFused = (size_t)256 << 20;
// Fixed-point scale of the usage histograms and forward sums: values * 2^32 in int64.
constexpr double kInvFix = 1.0 / 4294967296.0;
// Limits checked by gaus_create.
constexpr int kMaxClasses = 16;
// Incident edges per work item of the fused kernel's edge phase (longer lists are
// cut into several items, so that no item is much longer than the others).
constexpr int kChunkEdges = 4;

// Host-side plan produced by plan_problem() (pure C++, no CUDA).
struct Plan {
  int V = 0, E = 0, NB = 0, C = 0, D = 0, II = 0, Dh = 0, B = 0, cp = 0;
  std::vector<int32_t> asap, alap;        // caller order
  std::vector<int32_t> perm;              // internal -> caller
  std::vector<int32_t> inv;               // caller -> internal
  std::vector<int32_t> level;             // caller order, topological level
  // internal-order node attributes
  std::vector<float> w, bits;
  std::vector<int32_t> lat, cls;
  // CSC of internal consumers: producer caller id, producer latency
  std::vector<int32_t> in_ptr, in_src, in_lat;
  // CSR of internal producers: consumer caller id
  std::vector<int32_t> out_ptr, out_dst;
  // CSR position of each internal in-edge (CSC order)
  std::vector<int32_t> in_eslot;
  // back edges grouped by internal consumer i: producer caller id j, shift Lat(j) - k II
  std::vector<int32_t> bin_ptr, bin_src, bin_shift;
  // back edges grouped by internal producer j: consumer caller id i, same shift
  std::vector<int32_t> bout_ptr, bout_dst, bout_shift;
  // bout position of each back edge in bin order
  std::vector<int32_t> bin_eslot;
  // edge list of the edge pass, 4 per edge: producer, consumer (caller ids),
  // latency or shift, kind (0 forward, 1 back); E forward edges then NB back edges
  std::vector<int32_t> ed;
  // segments of internal nodes, each inside one class: start, end, class
  std::vector<int32_t> seg;               // 3 * nseg
  std::vector<int32_t> cls_seg_ptr;       // C + 1, segments of class c
  int nseg = 0;
  // caller-order data for the integer kernels
  // fused kernel: incident edges by internal id -- in-edges (producer, Lat(producer)),
  // out-edges (consumer, Lat(producer)), back edges into i (j, shift) and out of j
  // (i, shift); int2 pairs
  std::vector<int32_t> fin, fout, fbin, fbout;
  // fused kernel segments (same layout as seg): start, end, class
  std::vector<int32_t> fseg;
  // fused kernel's edge phase: every node's incident edges in one list of int4
  // (neighbour, latency or shift, kind 0 in / 1 out / 2 back in / 3 back out, 0),
  // cut into chunks of at most kChunkEdges: int4 (node, first entry, entries, 0),
  // in claim order (the most entries first; .w = the chunk's index in node-major
  // order, cptr (V + 1) the node-major chunk indices of each node); p2ord: that order
  std::vector<int32_t> finc, chunk, cptr, p2ord;
  int nchunk = 0;
  int nfseg = 0;
  std::vector<int32_t> lvl_ptr, lvl_nodes;           // nodes (caller ids) by level
  std::vector<int32_t> lq_ptr, lq_src, lq_lat;       // predecessors by level-order position
  std::vector<int32_t> cpred_ptr, cpred_src;         // CSC by caller consumer id
  std::vector<int32_t> csucc_ptr, csucc_dst;         // CSR by caller producer id
  std::vector<int32_t> cback_ptr, cback_src, cback_shift;  // back edges by caller consumer
  std::vector<int32_t> c_lat, c_cls, c_dem, c_bits;  // caller order
  std::vector<int32_t> e_src, e_dst;                 // edge list (caller ids)
  std::vector<int32_t> b_src, b_dst, b_dist;
  std::vector<float> limit;
  int nlvl = 0;
  int has_reg_succ_any = 0;
  int unit_lat = 0;  // every producer of an edge has latency 1
};

// Returns GAUS_OK or an error with a message.
gaus_status plan_problem(const gaus_problem *p, int target_blocks, Plan *out, std::string *err);
void plan_segments(Plan &P, int target_blocks, int RB);
// Segments of the fused kernel: about target_per_group segments of whole rows of
// RB-restart warp rows, each inside one class (written to P.fseg / P.nfseg).
void plan_fused_segments(Plan &P, int target_per_group, int RB);
gaus_status check_hparams(const gaus_hparams *hp, std::string *err);
float family_window_k(float window_k, int family);

}  // namespace gaus

struct gaus_ctx {
  gaus::Plan plan;
  gaus_hparams hp;
  float k_win = 6.0f;            // window half-width in sigma for the CDF family (family_window_k)
  cudaStream_t stream = nullptr;
  cudaStream_t side = nullptr;                     // usage reduction beside the edge pass
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  int prio_hi = 0;                                 // greatest stream priority (the edge pass)
  std::string err;
  int RB = 32, G = 1, nblk = 0;  // restarts per block row, restart groups, blocks per node pass
  int ce = 0, nchunk = 0;        // k_dep_cf: edges per block, chunks per restart group
  int nblk_e = 0;                // edge pass blocks (one wave, a multiple of G)
  int nblk_u = 0;                // k_update blocks
  int W = 0;                     // points per CDF table row
  int red_blocks = 0;
  int RBr = 32, Gr = 1, nblk_r = 0;  // storage-term kernels: restarts per row, groups, blocks
  size_t smem_rfwd = 0, smem_rbwd = 0;
  size_t smem_nodes = 0, smem_fin = 0, smem_ver = 0;
  // device graph
  int32_t *d_perm = nullptr;
  float *d_w = nullptr, *d_bits = nullptr, *d_limit = nullptr;
  int32_t *d_lat = nullptr, *d_cls = nullptr;
  int32_t *d_in_ptr = nullptr, *d_in_src = nullptr, *d_in_lat = nullptr;
  int32_t *d_out_ptr = nullptr, *d_out_dst = nullptr;
  int32_t *d_bin_ptr = nullptr, *d_bin_src = nullptr, *d_bin_shift = nullptr;
  int32_t *d_bout_ptr = nullptr, *d_bout_dst = nullptr, *d_bout_shift = nullptr;
  int32_t *d_seg = nullptr, *d_cls_seg_ptr = nullptr;
  int32_t *d_lvl_ptr = nullptr, *d_lvl_nodes = nullptr;
  int32_t *d_lq_ptr = nullptr, *d_lq_src = nullptr, *d_lq_lat = nullptr;
  size_t smem_leg = 0;           // k_legalize_regular_smem (0: schedule does not fit)
  int32_t *d_cpred_ptr = nullptr, *d_cpred_src = nullptr;
  int32_t *d_csucc_ptr = nullptr, *d_csucc_dst = nullptr;
  int32_t *d_cback_ptr = nullptr, *d_cback_src = nullptr, *d_cback_shift = nullptr;
  int32_t *d_c_lat = nullptr, *d_c_cls = nullptr, *d_c_dem = nullptr, *d_c_bits = nullptr;
  int32_t *d_e_src = nullptr, *d_e_dst = nullptr;
  int32_t *d_b_src = nullptr, *d_b_dst = nullptr, *d_b_dist = nullptr;
  int32_t *d_asap = nullptr, *d_alap = nullptr;
  // scratch
  long long *d_hpart = nullptr;  // nblk * Dh * RB fixed-point usage partials
  int2 *d_hspan = nullptr;       // nblk folded bin span written by each block
  unsigned long long *d_fwdtot = nullptr;  // B * 3 forward sums (dep, com, rec), 2^32 fixed point
  long long *d_U = nullptr;      // B * C * Dh usage (k_reduce), 2^32 fixed point
  long long *d_rpart = nullptr;  // nblk_r * Dh * RBr storage partials
  long long *d_Ureg = nullptr;   // B * Dh expected (folded) storage, 2^32 fixed point
  float4 *d_qtab = nullptr;      // tail tables of the storage forward (k_tail_tables), all families
  float *d_ptab = nullptr;       // (V, B, WP) successors' products, forward -> backward
  int WP = 0;
  float *d_Hreg = nullptr;       // B * Dh storage adjoint
  float2 *d_eslot = nullptr;     // E * B successor shares of the storage gradient
  int32_t *d_in_eslot = nullptr; // E
  int4 *d_ed = nullptr;          // E + NB edge list of the edge pass
  float4 *d_eslot4 = nullptr;    // 2 (E + NB) * B per-edge partials [edge][side][restart]
  float2 *d_gown = nullptr;      // V * B own-window storage adjoint (internal index)
  unsigned *d_win = nullptr;     // V * B packed windows (caller order)
  float *d_tab = nullptr;        // V * B * W CDF values at the window points (caller order)
  float *d_H = nullptr;          // B * C * Dh usage adjoint dL/dU
  float *d_coef = nullptr;       // B * 4 (c_dep, c_rec, Adam bias corrections)
  unsigned long long *d_wstat = nullptr;  // B * 2 window statistics of the iteration
  int32_t *d_thr = nullptr;      // B long-window thresholds
  int32_t *d_decision = nullptr; // B outer-step decisions
  unsigned long long *d_vacc = nullptr;  // verifier counts, usage counts, storage differences
  size_t vacc_words = 0;
  int RBv = 32, Gv = 1, nblk_v = 1;      // verifier pass 1: restarts per row, groups, blocks
  int32_t *d_nonfinite = nullptr;  // B flags
  int32_t *d_status_tmp = nullptr; // B
  float *d_loss_tmp = nullptr, *d_terms_tmp = nullptr;
  // fused persistent iteration (gaus_fused.cuh): blocks per restart group, groups
  // per cooperative launch, dynamic shared memory; 0 = the terms or sizes need the
  // multi-kernel path (storage term, continuous dependency penalty, D > 32767)
  int fK = 0, fGl = 0;
  int path_mode = 0;             // GAUS_PATH_AUTO, GAUS_PATH_FUSED or GAUS_PATH_MULTI (gaus_set_path)
  long long n_fused_calls = 0, n_multi_iters = 0, n_path_stats = 0;  // what gaus_iterate ran so far
  unsigned long long *d_wsel = nullptr;  // window points sum and maximum of the path choice
  unsigned long long *h_wsel = nullptr;  // its pinned host copy
  int nsm = 0;                   // streaming multiprocessors of the device
  int fRG = 1, fRBp = 1, fRB1 = 1, fG = 1;
  int fW = 0;  // table row length of the fused path ([node][point][restart] layout)  // restarts per group, lanes per row (phases 2-3, phase 1), groups
  size_t smem_fused = 0;
  int32_t *d_fseg = nullptr, *d_cptr = nullptr;
  int4 *d_finc = nullptr, *d_chunk = nullptr;
  signed char *d_ord = nullptr;  // fG * V * 64 restart orders (identity at creation)
  int2 *d_fin = nullptr, *d_fout = nullptr, *d_fbin = nullptr, *d_fbout = nullptr;
  float2 *d_xs = nullptr, *d_partr = nullptr;
  float4 *d_adm = nullptr, *d_part = nullptr;
  double *d_rstat = nullptr;
  unsigned char *d_facc = nullptr;  // group barriers, abort flag and the parity-buffered accumulators
  size_t facc_bytes = 0, off_ctr = 0, off_abort = 0, off_U = 0, off_fwd = 0, off_wst = 0, off_nonf = 0;
  unsigned long long *d_prof = nullptr;
  int prof_cap = 0;
  // captured iteration
  cudaGraphExec_t gexec = nullptr, gexec_n = nullptr;  // one iteration, kGraphUnroll iterations
  gaus_state gstate{};
  uint64_t ghash = 0;
  std::vector<void *> allocs;
};
