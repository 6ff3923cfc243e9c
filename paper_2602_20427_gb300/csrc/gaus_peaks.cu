// gaus_peaks.cu -- measurement helpers, not on the scheduling path: the throughput
// of this device's FP32 FMA pipe and of its special-function unit's exp2, which
// bound the node and edge passes' arithmetic, from microbenchmarks of independent
// dependency chains on every SM timed with CUDA events.
#include <cuda_runtime.h>

#include <algorithm>

#include "gaus.h"

namespace gaus {
namespace {

constexpr int kPeakThreads = 256;
constexpr int kChains = 8;    // independent chains per thread
constexpr int kUnroll = 16;   // chain steps per loop trip

// Each thread runs kChains independent FMA chains (x <- x a + b with |a| < 1, so the
// values stay bounded); the sum is stored only under a condition the data never
// meets, which keeps the chains from being optimised away.
__global__ void __launch_bounds__(kPeakThreads) k_peak_fma(float *out, int iters, float a, float b) {
  float x[kChains];
#pragma unroll
  for (int k = 0; k < kChains; ++k) x[k] = 1e-3f * (float)threadIdx.x + (float)k;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
#pragma unroll
      for (int k = 0; k < kChains; ++k) x[k] = fmaf(x[k], a, b);
  }
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < kChains; ++k) s += x[k];
  if (s == -1.0f) out[threadIdx.x] = s;
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// kChains independent chains x <- 2^(-x): every value stays in (0, 1].
__global__ void __launch_bounds__(kPeakThreads) k_peak_ex2(float *out, int iters) {
  float x[kChains];
#pragma unroll
  for (int k = 0; k < kChains; ++k) x[k] = 1e-3f * (float)threadIdx.x + 0.1f * (float)k;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
#pragma unroll
      for (int k = 0; k < kChains; ++k) x[k] = ex2_approx(-x[k]);
  }
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < kChains; ++k) s += x[k];
  if (s == -1.0f) out[threadIdx.x] = s;
}

}  // namespace
}  // namespace gaus

extern "C" gaus_status gaus_measure_peak(int32_t what, double *per_second, void *cuda_stream) {
  using namespace gaus;
  if (!per_second || (what != GAUS_PEAK_FP32 && what != GAUS_PEAK_EX2)) return GAUS_EINVAL;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(cuda_stream);
  int dev = 0, nsm = 0, occ = 0;
  float *out = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  gaus_status rc = GAUS_OK;
  auto ck = [&](cudaError_t e) {
    if (e != cudaSuccess && rc == GAUS_OK) {
      cudaGetLastError();
      rc = GAUS_ECUDA;
    }
    return e == cudaSuccess;
  };
  const void *fn = what == GAUS_PEAK_FP32 ? (const void *)k_peak_fma : (const void *)k_peak_ex2;
  if (ck(cudaGetDevice(&dev)) && ck(cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) &&
      ck(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fn, kPeakThreads, 0)) &&
      ck(cudaMalloc(&out, kPeakThreads * sizeof(float))) && ck(cudaEventCreate(&e0)) && ck(cudaEventCreate(&e1))) {
    const int blocks = std::max(1, occ) * nsm;
    const int iters = what == GAUS_PEAK_FP32 ? 4096 : 1024;
    double best = 0.0;
    for (int rep = 0; rep < 4 && rc == GAUS_OK; ++rep) {  // the first run warms up
      ck(cudaEventRecord(e0, st));
      if (what == GAUS_PEAK_FP32) k_peak_fma<<<blocks, kPeakThreads, 0, st>>>(out, iters, 0.999f, 1e-4f);
      else k_peak_ex2<<<blocks, kPeakThreads, 0, st>>>(out, iters);
      ck(cudaGetLastError());
      ck(cudaEventRecord(e1, st));
      ck(cudaEventSynchronize(e1));
      float ms = 0.f;
      if (rc == GAUS_OK && ck(cudaEventElapsedTime(&ms, e0, e1)) && rep > 0 && ms > 0.f) {
        const double ops = (double)blocks * kPeakThreads * iters * kUnroll * kChains *
                           (what == GAUS_PEAK_FP32 ? 2.0 : 1.0);
        best = std::max(best, ops / (ms * 1e-3));
      }
    }
    *per_second = best;
  }
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (out) cudaFree(out);
  return rc;
}
