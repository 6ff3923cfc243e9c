// gaus_noalloc.cu -- expected usage histograms for callers that cannot allocate
// device memory.
//
// Some callers cannot call cudaMalloc at all: code running inside a memory pool
// or arena owned by another framework, allocation-free real-time loops, or hosts
// whose device memory is budgeted up front.  gaus_expected_usage_noalloc serves
// them: it computes the expected per-class usage histograms (the segmented usage
// reduction of the iteration) from device arrays the caller already owns, and its
// only working memory is a fixed array in this file's device globals.
//
// The array below is allocated by the CUDA runtime when the library is loaded on
// a device and stays there until the process exits.  All calls share it: the
// completion counters are cleared at the start of every call, and the partial
// histograms are fully rewritten before they are read.  Two calls whose work
// overlaps on the GPU (different streams, or different host threads on one
// device) race on this array and give undefined results; serialise them.
#include <cuda_runtime.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <mutex>
#include <string>

#include "gaus.h"
#include "gaus_device.cuh"
#include "gaus_internal.h"

namespace gaus {
void set_thread_error(const std::string &msg);  // gaus_api.cu
}

namespace {

using namespace gaus;

constexpr size_t kNoAllocScratchBytes = 16u << 20;  // 16 MiB per device
// one u32 completion counter per (restart group, class), then one u32 per (restart
// group, class) of flags: bit r set when restart r of the group met a demand
// outside 0..kMaxDemand in that class
constexpr size_t kCounterBytes = 8192;
constexpr int kMaxPairs = 1024;
constexpr int kMaxDevices = 64;
constexpr int kMaxDemand = 64;

static __device__ __align__(256) unsigned char g_usage_scratch[kNoAllocScratchBytes];

std::mutex g_setup_mu;
void *g_scratch_addr[kMaxDevices] = {};

struct UsageArgs {
  const float *mu, *sg;
  const int32_t *cls, *dem;
  int V, B, C, D, II, Dh, RB, G, NC, CL;
  float k_win;
  unsigned *counters, *bad;
  long long *part;
  double *usage;
};

// Block = (restart group g, class c, node chunk ch).  Lanes are restarts; each
// warp claims the chunk's nodes in groups of 32 / RB, skips other classes, and adds
// its bin masses to a shared-memory histogram (exact fixed point; the bin masses
// from the same upper-tail evaluation as the context path's node pass).  The
// block's histogram goes to the scratch array; the last block of (g, c) to finish
// sums the chunks in a fixed order and writes the usage.  A demand outside
// 0..kMaxDemand (the bound that keeps the histogram's 16-bit halves from
// overflowing) is not added: it marks the restart's row of that class, which is
// then written as NaN.
__global__ void __launch_bounds__(256) k_usage_noalloc(const UsageArgs A) {
  extern __shared__ __align__(16) unsigned char smem[];
  constexpr unsigned FULL = 0xffffffffu;
  const int tid = threadIdx.x, RB = A.RB, Dh = A.Dh;
  unsigned *hlo = reinterpret_cast<unsigned *>(smem);
  unsigned *hhi = hlo + (size_t)Dh * RB;
  __shared__ int s_next, s_last;
  __shared__ unsigned s_bad;
  const int blk = blockIdx.x, ch = blk % A.NC, gc = blk / A.NC, c = gc % A.C, g = gc / A.C;
  const int v0 = ch * A.CL, v1 = min(A.V, v0 + A.CL);
  for (int i = tid; i < 2 * Dh * RB; i += 256) hlo[i] = 0u;
  if (tid == 0) { s_next = 0; s_bad = 0u; }
  __syncthreads();

  const int lane = tid & 31, r = tid % RB, b = g * RB + r, npw = 32 / RB;
  for (;;) {
    int base = 0;
    if (lane == 0) base = atomicAdd(&s_next, npw);
    base = __shfl_sync(FULL, base, 0);
    if (base >= v1 - v0) break;
    const int v = v0 + base + lane / RB;
    bool valid = b < A.B && v < v1 && A.cls[v] == c;
    const float mu = valid ? A.mu[(size_t)v * A.B + b] : 0.f, sg = valid ? A.sg[(size_t)v * A.B + b] : 1.f;
    valid = valid && usable(mu, sg);
    const int dm = valid ? (A.dem ? A.dem[v] : 1) : 0;
    if (valid && (dm < 0 || dm > kMaxDemand)) {
      atomicOr(&s_bad, 1u << r);
      valid = false;
    }
    const float inv_s = valid ? 1.0f / sg : 1.0f;
    const float wv = valid ? (float)dm : 0.f;
    int a = 0, bw = -2;
    if (valid) window(mu, sg, A.k_win, A.D, a, bw);
    const int n = bw - a + 1;
    const int nmax = __reduce_max_sync(FULL, n);
    float zp = 0.f, qp = 0.f;
    for (int j = 0; j <= nmax; ++j) {
      const bool pt = j < n;
      const float zc = ((float)(a + j) + 0.5f - mu) * inv_s;
      const float qc = pt ? tail_fast(zc) : 0.f;
      if (j <= n) hist_add(hlo, hhi, fold_bin(a + j, A.II) * RB + r, wv * bin_mass(pt, j == 0, zc, qc, zp, qp));
      zp = zc;
      qp = qc;
    }
    __syncwarp();
  }
  __syncthreads();
  long long *mine = A.part + (size_t)blk * Dh * RB;
  for (int i = tid; i < Dh * RB; i += 256)
    mine[i] = (long long)(((unsigned long long)hhi[i] << 16) + (unsigned long long)hlo[i]);
  if (tid == 0 && s_bad) atomicOr(&A.bad[gc], s_bad);
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(&A.counters[gc], 1u) == (unsigned)(A.NC - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const long long *first = A.part + (size_t)gc * A.NC * Dh * RB;
  const unsigned bad = __ldcg(&A.bad[gc]);
  for (int i = tid; i < Dh * RB; i += 256) {
    const int d = i / RB, rr = i % RB, bb = g * RB + rr;
    if (bb >= A.B) continue;
    long long acc = 0;
    for (int k = 0; k < A.NC; ++k) acc += __ldcg(first + (size_t)k * Dh * RB + i);
    A.usage[((size_t)bb * A.C + c) * Dh + d] = ((bad >> rr) & 1u) ? __longlong_as_double(0x7ff8000000000000ll)
                                                                   : (double)acc * kInvFix;
  }
  if (tid == 0) A.counters[gc] = 0u;
}

gaus_status fail(gaus_status st, const std::string &msg) {
  set_thread_error(msg);
  return st;
}

}  // namespace

extern "C" gaus_status gaus_expected_usage_noalloc(const float *mu, const float *sigma, const int32_t *res_class,
                                                   const int32_t *demand, int32_t V, int32_t B, int32_t C,
                                                   int32_t D, int32_t II, float window_k, double *usage,
                                                   void *cuda_stream) {
  if (!mu || !sigma || !res_class || !usage) return fail(GAUS_EINVAL, "gaus_expected_usage_noalloc: NULL pointer");
  if (V < 1 || B < 1 || C < 1 || C > kMaxClasses || D < 1 || D > 65536 || II < 0 ||
      !(window_k > 0.0f) || !std::isfinite(window_k))
    return fail(GAUS_EINVAL, "gaus_expected_usage_noalloc: V, B >= 1, C in 1..16, D in 1..65536, II >= 0, "
                             "window_k > 0 required");
  if ((int64_t)V * B >= ((int64_t)1 << 31)) return fail(GAUS_EINVAL, "gaus_expected_usage_noalloc: V * B >= 2^31");
  const int Dh = II > 0 ? II : D;
  int RB = 1;
  while (RB < B && RB < 32) RB <<= 1;
  const int G = (B + RB - 1) / RB;
  const size_t smem = 2 * (size_t)Dh * RB * sizeof(unsigned);
  if (smem > 200 * 1024)
    return fail(GAUS_EINVAL, "gaus_expected_usage_noalloc: histogram length (II or D) times min(B, 32) "
                             "exceeds 25,600");
  if (G * C > kMaxPairs)
    return fail(GAUS_EINVAL, "gaus_expected_usage_noalloc: more than 1,024 (restart group, class) pairs");
  const size_t per_block = (size_t)Dh * RB * sizeof(long long);
  const size_t cap_blocks = (kNoAllocScratchBytes - kCounterBytes) / per_block;
  // chunk length bounded so that the 16-bit halves of the histogram cannot overflow
  const int folds = (D + Dh - 1) / Dh;
  const int max_chunk = std::max(1, 32768 / (kMaxDemand * folds));
  long nc = std::max<long>((V + 63) / 64, (V + max_chunk - 1) / max_chunk);
  nc = std::min<long>(nc, (long)(cap_blocks / ((size_t)G * C)));
  if (nc < 1 || (V + nc - 1) / nc > max_chunk)
    return fail(GAUS_EINVAL, "gaus_expected_usage_noalloc: problem exceeds the 16 MiB fixed scratch array");
  const int NC = (int)nc, CL = (V + NC - 1) / NC;

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(GAUS_ECUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(GAUS_EINVAL, "gaus_expected_usage_noalloc: device index >= 64");
  void *base = nullptr;
  {
    // once per device, with that device current: the device address of the array
    // (a cudaDeviceReset in this process invalidates it; see include/gaus.h)
    std::lock_guard<std::mutex> lock(g_setup_mu);
    if (!g_scratch_addr[dev]) {
      void *p = nullptr;
      e = cudaGetSymbolAddress(&p, g_usage_scratch);
      if (e != cudaSuccess) return fail(GAUS_ECUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
      e = cudaFuncSetAttribute((const void *)k_usage_noalloc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               200 * 1024);
      if (e != cudaSuccess) return fail(GAUS_ECUDA, std::string("cudaFuncSetAttribute: ") + cudaGetErrorString(e));
      g_scratch_addr[dev] = p;
    }
    base = g_scratch_addr[dev];
  }
  cudaStream_t st = (cudaStream_t)cuda_stream;
  UsageArgs A;
  A.mu = mu; A.sg = sigma; A.cls = res_class; A.dem = demand;
  A.V = V; A.B = B; A.C = C; A.D = D; A.II = II; A.Dh = Dh; A.RB = RB; A.G = G; A.NC = NC; A.CL = CL;
  A.k_win = window_k;
  A.counters = reinterpret_cast<unsigned *>(base);
  A.bad = A.counters + kMaxPairs;
  A.part = reinterpret_cast<long long *>(reinterpret_cast<unsigned char *>(base) + kCounterBytes);
  A.usage = usage;
  e = cudaMemsetAsync(A.counters, 0, kCounterBytes, st);
  if (e != cudaSuccess) return fail(GAUS_ECUDA, std::string("cudaMemsetAsync: ") + cudaGetErrorString(e));
  k_usage_noalloc<<<G * C * NC, 256, smem, st>>>(A);
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(GAUS_ECUDA, std::string("k_usage_noalloc launch: ") + cudaGetErrorString(e));
  return GAUS_OK;
}
