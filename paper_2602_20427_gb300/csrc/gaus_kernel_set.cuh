// gaus_kernel_set.cuh -- the iteration kernels that depend on the CDF family, as
// one table of launchable pointers per family.  The normal's set is instantiated
// in gaus_api.cu; each other family's (App. D) in its own translation unit
// (gaus_family.cu compiled once per family), so that the builds run side by side.
#pragma once

#include "gaus_fused.cuh"
#include "gaus_kernels.cuh"

namespace gaus {

using NodeKernel = void (*)(const IterArgs);
using EdgeKernel = void (*)(const IterArgs);
using UpdKernel = void (*)(const UpdArgs);
using RegKernel = void (*)(const RegArgs);
using FusedKernel = void (*)(const FusedArgs);

constexpr int kEdgeVariants = 12;

struct KernelSet {
  NodeKernel nodes = nullptr;
  EdgeKernel edges[kEdgeVariants] = {};  // by edge_variant()
  UpdKernel update[4] = {};              // [2 * adam + hist]
  RegKernel reg_fwd = nullptr, reg_bwd = nullptr;
  FusedKernel fused[2] = {};             // [com]
};

// Edge-pass variant of a term mask: which of the dependency, communication and
// recurrence sums it computes, and whether every edge has latency 1 (no back edges).
inline int edge_variant(unsigned terms, int II, bool unit) {
  const bool dep = terms & GAUS_DEP, com = terms & GAUS_COM, rec = (terms & GAUS_REC) && II > 0;
  if (rec) return (dep ? 1 : 0) + (com ? 2 : 0);  // 0..3
  return 4 + (unit ? 4 : 0) + (dep ? 1 : 0) + (com ? 2 : 0);  // 4..11
}

template <int kFam>
KernelSet make_kernel_set() {
  KernelSet s;
  s.nodes = k_nodes<kFam>;
  s.edges[0] = k_edges<kFam, false, false, true, false>;
  s.edges[1] = k_edges<kFam, true, false, true, false>;
  s.edges[2] = k_edges<kFam, false, true, true, false>;
  s.edges[3] = k_edges<kFam, true, true, true, false>;
  s.edges[4] = k_edges<kFam, false, false, false, false>;
  s.edges[5] = k_edges<kFam, true, false, false, false>;
  s.edges[6] = k_edges<kFam, false, true, false, false>;
  s.edges[7] = k_edges<kFam, true, true, false, false>;
  s.edges[8] = k_edges<kFam, false, false, false, true>;
  s.edges[9] = k_edges<kFam, true, false, false, true>;
  s.edges[10] = k_edges<kFam, false, true, false, true>;
  s.edges[11] = k_edges<kFam, true, true, false, true>;
  s.update[0] = k_update<kFam, false, false>;
  s.update[1] = k_update<kFam, false, true>;
  s.update[2] = k_update<kFam, true, false>;
  s.update[3] = k_update<kFam, true, true>;
  s.reg_fwd = k_reg_fwd<kFam>;
  s.reg_bwd = k_reg_bwd<kFam>;
  s.fused[0] = k_fused<kFam, false>;
  s.fused[1] = k_fused<kFam, true>;
  return s;
}

// Defined in the per-family translation units.
KernelSet kernel_set_logistic();
KernelSet kernel_set_laplace();
KernelSet kernel_set_cauchy();

}  // namespace gaus
