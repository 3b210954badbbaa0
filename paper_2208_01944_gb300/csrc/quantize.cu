// Group-wise activation quantisation (Sec. 3.2 Eq. 2 with l = 0, u = s (2^b - 1),
// Sec. 4.1 "quantize the activations ... to B-bit in each group") and the
// deterministic per-group sums behind the step initialisation.
//
// Quantisation is HBM-bound (4 bytes in, 1 byte out per element).  The fast path
// gives each thread 16 consecutive elements of one pixel (so they share a group
// when C_g is a multiple of 16): four 16-byte streaming loads, one fp32 multiply,
// a round-to-nearest-even conversion and an integer clamp per element, and one
// 16-byte streaming store, in a grid-stride loop over a grid sized to the SM count.
#include <cuda_runtime.h>

#include <cstdint>

#include "pq_internal.h"
#include "pq_device.cuh"

namespace pq {

struct QuantArgs {
  float inv_s[kMaxG];
};

__device__ __forceinline__ uint32_t quant4(float4 v, float inv, int qmax) {
  // __float2int_rn = round half to even; NaN -> 0, +-inf saturate and clamp below.
  int a = __float2int_rn(__fmul_rn(v.x, inv));
  int b = __float2int_rn(__fmul_rn(v.y, inv));
  int c = __float2int_rn(__fmul_rn(v.z, inv));
  int d = __float2int_rn(__fmul_rn(v.w, inv));
  a = min(max(a, 0), qmax);
  b = min(max(b, 0), qmax);
  c = min(max(c, 0), qmax);
  d = min(max(d, 0), qmax);
  return static_cast<uint32_t>(a) | (static_cast<uint32_t>(b) << 8) | (static_cast<uint32_t>(c) << 16) |
         (static_cast<uint32_t>(d) << 24);
}

// 16 elements per thread-iteration; requires C_g % 16 == 0 and 16-byte aligned x, q.
__global__ void __launch_bounds__(256) pq_quantize_vec16(const float4* __restrict__ x, uint4* __restrict__ q,
                                                         int64_t nvec, int vec_per_pix, int vec_per_group, int qmax,
                                                         const __grid_constant__ QuantArgs args) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t v = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    const int cv = static_cast<int>(v % vec_per_pix);
    const float inv = args.inv_s[cv / vec_per_group];
    const float4* src = x + 4 * v;
    const float4 a = __ldcs(src), b = __ldcs(src + 1), c = __ldcs(src + 2), d = __ldcs(src + 3);
    uint4 out;
    out.x = quant4(a, inv, qmax);
    out.y = quant4(b, inv, qmax);
    out.z = quant4(c, inv, qmax);
    out.w = quant4(d, inv, qmax);
    __stcs(q + v, out);
  }
}

// Any shape: one element per thread-iteration.
__global__ void __launch_bounds__(256) pq_quantize_scalar(const float* __restrict__ x, uint8_t* __restrict__ q,
                                                          int64_t n, int C, int Cg, int qmax,
                                                          const __grid_constant__ QuantArgs args) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n; e += stride) {
    const int c = static_cast<int>(e % C);
    int v = __float2int_rn(__fmul_rn(x[e], args.inv_s[c / Cg]));
    v = min(max(v, 0), qmax);
    q[e] = static_cast<uint8_t>(v);
  }
}

// Channel-blocked output [N][C/16][HW][16].  A warp takes 8 consecutive pixels
// x 4 consecutive 16-channel blocks of one image: lane (p, j) reads the 64 bytes
// of its pixel's block (the warp reads 8 runs of 256 contiguous bytes) and writes
// the block's 16 codes (the warp writes 4 runs of 128 contiguous bytes, one per
// block).  Consecutive warps take the next 4 blocks of the same pixels, so whole
// pixel rows are read by neighbouring warps at about the same time.  A grid of a
// few blocks per SM, striding over the (image, pixel group, block group) units,
// keeps enough loads in flight for the HBM bandwidth.
// PACK = 1: the block's codes packed four to a 32-bit word; PACK = 2: two to a
// byte (8 bytes, half of the 16-byte row of its 32-channel block).
template <int PACK>
__global__ void __launch_bounds__(256) pq_quantize_c16(const float4* __restrict__ x, void* __restrict__ q, int64_t N,
                                                       int64_t HW, int C16, int blocks_per_group, int qmax,
                                                       const __grid_constant__ QuantArgs args) {
  const int lane = threadIdx.x & 31;
  const int jj = lane & 3, pp = lane >> 2;
  const int64_t pix_groups = (HW + 7) / 8;
  const int jgroups = (C16 + 3) / 4;
  const int64_t units = N * pix_groups * jgroups;
  const int64_t wstride = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  for (int64_t u = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5); u < units; u += wstride) {
    const int jg = static_cast<int>(u % jgroups);
    const int64_t r = u / jgroups;
    const int64_t n = r / pix_groups;
    const int64_t hw = (r - n * pix_groups) * 8 + pp;
    const int j = jg * 4 + jj;
    if (hw < HW && j < C16) {
      const float inv = args.inv_s[j / blocks_per_group];
      const float4* s4 = x + ((n * HW + hw) * C16 + j) * 4;
      const float4 a = __ldcs(s4), b = __ldcs(s4 + 1), c = __ldcs(s4 + 2), d = __ldcs(s4 + 3);
      uint4 out;
      out.x = quant4(a, inv, qmax);
      out.y = quant4(b, inv, qmax);
      out.z = quant4(c, inv, qmax);
      out.w = quant4(d, inv, qmax);
      if (PACK == 1)
        __stcs(static_cast<uint32_t*>(q) + (n * C16 + j) * HW + hw, pack2_word(out));
      else if (PACK == 2)
        __stcs(static_cast<uint2*>(q) + ((n * (C16 >> 1) + (j >> 1)) * HW + hw) * 2 + (j & 1), pack4_word(out));
      else
        __stcs(static_cast<uint4*>(q) + (n * C16 + j) * HW + hw, out);
    }
  }
}

int launch_quantize_c16(const float* x, uint8_t* q, int64_t N, int64_t HW, int G, int Cg, int bits, const float* inv_s,
                        int pack, cudaStream_t stream) {
  QuantArgs args;
  for (int g = 0; g < G; ++g) args.inv_s[g] = inv_s[g];
  const int C16 = G * Cg / 16;
  if (N == 0 || HW == 0) return 0;
  const int64_t warps = N * ((HW + 7) / 8) * ((C16 + 3) / 4);
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (warps + 7) / 8;  // 8 warps per block
  const int64_t cap = static_cast<int64_t>(sms) * 4;
  const unsigned grid = static_cast<unsigned>(want < cap ? want : cap);
  const float4* xv = reinterpret_cast<const float4*>(x);
  const int qmax = (1 << bits) - 1;
  if (pack == 1)
    pq_quantize_c16<1><<<grid, 256, 0, stream>>>(xv, q, N, HW, C16, Cg / 16, qmax, args);
  else if (pack == 2)
    pq_quantize_c16<2><<<grid, 256, 0, stream>>>(xv, q, N, HW, C16, Cg / 16, qmax, args);
  else
    pq_quantize_c16<0><<<grid, 256, 0, stream>>>(xv, q, N, HW, C16, Cg / 16, qmax, args);
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

static int quant_grid(int64_t work) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (work + 255) / 256;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  return static_cast<int>(want < cap ? (want > 0 ? want : 1) : cap);
}

int launch_quantize(const float* x, uint8_t* q, int64_t P, int G, int Cg, int bits, const float* inv_s,
                    cudaStream_t stream) {
  QuantArgs args;
  for (int g = 0; g < G; ++g) args.inv_s[g] = inv_s[g];
  const int C = G * Cg;
  const int64_t n = P * C;
  const int qmax = (1 << bits) - 1;
  if (n == 0) return 0;
  const bool aligned = (reinterpret_cast<uintptr_t>(x) % 16 == 0) && (reinterpret_cast<uintptr_t>(q) % 16 == 0);
  if (Cg % 16 == 0 && aligned) {
    const int64_t nvec = n / 16;
    pq_quantize_vec16<<<quant_grid(nvec), 256, 0, stream>>>(reinterpret_cast<const float4*>(x),
                                                           reinterpret_cast<uint4*>(q), nvec, C / 16, Cg / 16, qmax,
                                                           args);
  } else {
    pq_quantize_scalar<<<quant_grid(n), 256, 0, stream>>>(x, q, n, C, Cg, qmax, args);
  }
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

// --------------------------------------------------------------------------
// Deterministic per-group sums for the step initialisation.  Pass 1: block b
// sums, in double and in a fixed order, group g's elements of the pixel range
// [b P / B, (b+1) P / B) and writes partial[b * G + g].  Pass 2: partial sums
// are added in block order.  B is fixed, so the result does not depend on the
// device or on timing.
// --------------------------------------------------------------------------
__global__ void __launch_bounds__(256) pq_act_sum_pass1(const float* __restrict__ x, int64_t P, int G, int Cg,
                                                        double* __restrict__ partial) {
  __shared__ double red[256];
  const int64_t p0 = static_cast<int64_t>(blockIdx.x) * P / gridDim.x;
  const int64_t p1 = static_cast<int64_t>(blockIdx.x + 1) * P / gridDim.x;
  const int64_t C = static_cast<int64_t>(G) * Cg;
  const int64_t cnt = (p1 - p0) * Cg;
  for (int g = 0; g < G; ++g) {
    double s = 0.0;
    for (int64_t e = threadIdx.x; e < cnt; e += blockDim.x) {
      const int64_t pix = p0 + e / Cg;
      const int j = static_cast<int>(e % Cg);
      s += static_cast<double>(x[pix * C + static_cast<int64_t>(g) * Cg + j]);
    }
    red[threadIdx.x] = s;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
      if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
      __syncthreads();
    }
    if (threadIdx.x == 0) partial[static_cast<int64_t>(blockIdx.x) * G + g] = red[0];
    __syncthreads();
  }
}

__global__ void pq_act_sum_pass2(const double* __restrict__ partial, int nblocks, int G, double* __restrict__ sums) {
  const int g = blockIdx.x * blockDim.x + threadIdx.x;
  if (g >= G) return;
  double s = 0.0;
  for (int b = 0; b < nblocks; ++b) s += partial[static_cast<int64_t>(b) * G + g];
  sums[g] = s;
}

int launch_act_sum(const float* x, int64_t P, int G, int Cg, double* partial, int nblocks, cudaStream_t stream) {
  pq_act_sum_pass1<<<nblocks, 256, 0, stream>>>(x, P, G, Cg, partial);
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

int launch_act_sum_finish(const double* partial, int nblocks, int G, double* sums, cudaStream_t stream) {
  pq_act_sum_pass2<<<(G + 63) / 64, 64, 0, stream>>>(partial, nblocks, G, sums);
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // namespace pq
