// palquant_act_steps_noalloc: the per-group activation step initialisation
// without any memory allocation.
//
// palquant_act_steps needs device scratch for its per-block partial sums and
// asks the caller for it.  Some callers have no way to provide it: code that
// must not call cudaMalloc (for example a plug-in running inside a host
// framework that owns every device allocation, or a latency-critical path whose
// memory budget is fixed up front) and code that cannot hold on to a buffer
// between calls.  This entry point keeps its scratch in a fixed-size array in
// the library's own device memory instead, so it allocates nothing.
//
// The array is a file-scope static __device__ variable: every GPU that loads
// the library holds it (kNoAllocScratchBytes) until the process exits.  Host
// code cannot pass the array's name to a kernel (on the host the name is only a
// stand-in for the symbol, not a device address), so the first call on each
// device looks up the device address with cudaGetSymbolAddress while that device
// is current and caches it.  Make that first call before any stream capture.  The
// cache lives as long as the process: after cudaDeviceReset the module may load the
// array at another address, so the entry point must not be used on a reset device.
//
// All calls share the array.  Each call overwrites every partial sum it reads
// (pass 1 writes all of them before pass 2 adds them), so nothing has to start
// at zero and the array simply keeps the last call's contents.  Calls that run
// on the GPU at the same time (different streams, or different host threads)
// race on the array and must be serialised by the caller.
#include <cuda_runtime.h>

#include <cmath>
#include <mutex>

#include "palquant.h"
#include "pq_internal.h"

namespace {

// Fixed layout of the scratch: kBlocks x G partial sums, then G totals (doubles).
constexpr int kNoAllocBlocks = 256;  // the same fixed partition as palquant_act_steps
constexpr int kNoAllocMaxG = 64;
constexpr size_t kNoAllocScratchBytes = sizeof(double) * (static_cast<size_t>(kNoAllocBlocks) * kNoAllocMaxG + kNoAllocMaxG);

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of g_noalloc_scratch for the current device (looked up once per device).
double* noalloc_scratch_for_current_device() {
  static std::mutex mu;
  static void* cached[64] = {nullptr};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (cached[dev] == nullptr) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || ptr == nullptr) return nullptr;
    cached[dev] = ptr;
  }
  return static_cast<double*>(cached[dev]);
}

}  // namespace

extern "C" pq_status palquant_act_steps_noalloc(const float* x_dev, int64_t N, int32_t H, int32_t W, int32_t G,
                                                int32_t Cg, int32_t bits, float* s_out_host, pq_stream_t stream) {
  if (x_dev == nullptr || s_out_host == nullptr) return PQ_EINVAL;
  if (N < 1 || H < 1 || W < 1 || G < 1 || Cg < 1 || bits < 1 || bits > 8) return PQ_EINVAL;
  // The fixed scratch holds at most kNoAllocMaxG groups.
  if (G > kNoAllocMaxG) return PQ_EUNSUPPORTED;
  double* partial = noalloc_scratch_for_current_device();
  if (partial == nullptr) return PQ_ECUDA;
  double* sums = partial + static_cast<size_t>(kNoAllocBlocks) * G;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int64_t P = N * H * W;
  if (pq::launch_act_sum(x_dev, P, G, Cg, partial, kNoAllocBlocks, s) != 0) return PQ_ECUDA;
  if (pq::launch_act_sum_finish(partial, kNoAllocBlocks, G, sums, s) != 0) return PQ_ECUDA;
  double h[kNoAllocMaxG];
  if (cudaMemcpyAsync(h, sums, sizeof(double) * G, cudaMemcpyDeviceToHost, s) != cudaSuccess) return PQ_ECUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return PQ_ECUDA;
  const double qp = static_cast<double>((1 << bits) - 1);
  for (int g = 0; g < G; ++g) {
    const double mean = h[g] / static_cast<double>(P * Cg);
    s_out_host[g] = static_cast<float>(2.0 * mean / std::sqrt(qp));
  }
  return PQ_OK;
}
