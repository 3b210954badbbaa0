// Device error word and the watchdog self-test.
//
// Every kernel of the library receives the address of a per-device error word.
// A bounded wait that runs out ORs PQ_ERR_TIMEOUT (and the role's bit) into it;
// palquant_sync_check() reads and clears it after synchronising.  The self-test
// kernel waits on a barrier nobody arrives on, so its wait runs out by design and
// exercises exactly that path without faulting the GPU.
#include <cuda_runtime.h>

#include <mutex>

#include "pq_device.cuh"
#include "pq_internal.h"

namespace pq {

__device__ unsigned int g_pq_error_word;

unsigned int* device_error_word() {
  static std::mutex mu;
  static unsigned int* cached[64] = {nullptr};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (cached[dev] == nullptr) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_pq_error_word) != cudaSuccess) return nullptr;
    cached[dev] = static_cast<unsigned int*>(ptr);
  }
  return cached[dev];
}

__global__ void pq_watchdog_selftest_kernel(unsigned int* err, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  // Nobody arrives on `bar`: the first phase never completes.
  WaitCtx ctx{&abort_flag, err, limit_ns, PQ_ERR_SELFTEST};
  mbar_wait(smem_u32(&bar), 0, ctx);
  __syncthreads();
}

int launch_watchdog_selftest(unsigned int* err, uint64_t limit_ns, cudaStream_t stream) {
  pq_watchdog_selftest_kernel<<<1, 32, 0, stream>>>(err, limit_ns);
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // namespace pq
