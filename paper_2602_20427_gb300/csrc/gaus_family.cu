// gaus_family.cu -- the iteration kernels of one non-normal CDF family (App. D):
// compiled once per family with GAUS_FAMILY_ID = GAUS_LOGISTIC, GAUS_LAPLACE or
// GAUS_CAUCHY (and GAUS_FAMILY_KERNELS_ONLY, which leaves out the kernels that do
// not depend on the family; gaus_api.cu holds those).
#include "gaus_kernel_set.cuh"

#ifndef GAUS_FAMILY_ID
#error "GAUS_FAMILY_ID must name the CDF family of this translation unit"
#endif

namespace gaus {

#if GAUS_FAMILY_ID == GAUS_LOGISTIC
KernelSet kernel_set_logistic() { return make_kernel_set<GAUS_LOGISTIC>(); }
#elif GAUS_FAMILY_ID == GAUS_LAPLACE
KernelSet kernel_set_laplace() { return make_kernel_set<GAUS_LAPLACE>(); }
#elif GAUS_FAMILY_ID == GAUS_CAUCHY
KernelSet kernel_set_cauchy() { return make_kernel_set<GAUS_CAUCHY>(); }
#else
#error "GAUS_FAMILY_ID must be GAUS_LOGISTIC, GAUS_LAPLACE or GAUS_CAUCHY"
#endif

}  // namespace gaus
