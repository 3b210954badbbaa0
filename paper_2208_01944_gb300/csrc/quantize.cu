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

// Per-group quantiser constants.  lu = 0: code = clamp(rint(x * inv_s), 0, Qp)
// (Eq. 2 with l = 0).  lu = 1, learned bounds l < u (Eq. 2 as trained):
// code = rint(sat((x - l) * inv_r) * Qp), inv_r = fl(1 / fl(u - l)), sat = clamp to
// [0, 1] with NaN -> 0; one rounding per operation.
struct QuantArgs {
  float inv_s[kMaxG];
  float l[kMaxG];
  float inv_r[kMaxG];
  float qp;
  int lu;
};

struct QuantGroup {
  float a, b;  // lu = 0: inv_s, unused; lu = 1: l, inv_r
};

// LU is a compile-time choice (one kernel instance per quantiser form), so the
// l = 0 form keeps its short per-element path.
template <bool LU>
__device__ __forceinline__ QuantGroup quant_group(const QuantArgs& args, int g) {
  return LU ? QuantGroup{args.l[g], args.inv_r[g]} : QuantGroup{args.inv_s[g], 0.0f};
}

template <bool LU>
__device__ __forceinline__ int quant1(float x, QuantGroup k, const QuantArgs& args, int qmax) {
  // __float2int_rn = round half to even; NaN -> 0, +-inf saturate and clamp below.
  if (LU) return __float2int_rn(__fmul_rn(__saturatef(__fmul_rn(__fsub_rn(x, k.a), k.b)), args.qp));
  return min(max(__float2int_rn(__fmul_rn(x, k.a)), 0), qmax);
}

template <bool LU>
__device__ __forceinline__ uint32_t quant4(float4 v, QuantGroup k, const QuantArgs& args, int qmax) {
  const int a = quant1<LU>(v.x, k, args, qmax), b = quant1<LU>(v.y, k, args, qmax);
  const int c = quant1<LU>(v.z, k, args, qmax), d = quant1<LU>(v.w, k, args, qmax);
  return static_cast<uint32_t>(a) | (static_cast<uint32_t>(b) << 8) | (static_cast<uint32_t>(c) << 16) |
         (static_cast<uint32_t>(d) << 24);
}

// 16 elements per thread-iteration; requires C_g % 16 == 0 and 16-byte aligned x, q.
template <bool LU>
__global__ void __launch_bounds__(256) pq_quantize_vec16(const float4* __restrict__ x, uint4* __restrict__ q,
                                                         int64_t nvec, int vec_per_pix, int vec_per_group, int qmax,
                                                         const __grid_constant__ QuantArgs args) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t v = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    const int cv = static_cast<int>(v % vec_per_pix);
    const QuantGroup k = quant_group<LU>(args, cv / vec_per_group);
    const float4* src = x + 4 * v;
    const float4 a = __ldcs(src), b = __ldcs(src + 1), c = __ldcs(src + 2), d = __ldcs(src + 3);
    uint4 out;
    out.x = quant4<LU>(a, k, args, qmax);
    out.y = quant4<LU>(b, k, args, qmax);
    out.z = quant4<LU>(c, k, args, qmax);
    out.w = quant4<LU>(d, k, args, qmax);
    __stcs(q + v, out);
  }
}

// Any shape: one element per thread-iteration.
template <bool LU>
__global__ void __launch_bounds__(256) pq_quantize_scalar(const float* __restrict__ x, uint8_t* __restrict__ q,
                                                          int64_t n, int C, int Cg, int qmax,
                                                          const __grid_constant__ QuantArgs args) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n; e += stride) {
    const int c = static_cast<int>(e % C);
    q[e] = static_cast<uint8_t>(quant1<LU>(x[e], quant_group<LU>(args, c / Cg), args, qmax));
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
template <int PACK, bool LU>
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
      const QuantGroup k = quant_group<LU>(args, j / blocks_per_group);
      const float4* s4 = x + ((n * HW + hw) * C16 + j) * 4;
      const float4 a = __ldcs(s4), b = __ldcs(s4 + 1), c = __ldcs(s4 + 2), d = __ldcs(s4 + 3);
      uint4 out;
      out.x = quant4<LU>(a, k, args, qmax);
      out.y = quant4<LU>(b, k, args, qmax);
      out.z = quant4<LU>(c, k, args, qmax);
      out.w = quant4<LU>(d, k, args, qmax);
      if (PACK == 1)
        __stcs(static_cast<uint32_t*>(q) + (n * C16 + j) * HW + hw, pack2_word(out));
      else if (PACK == 2)
        __stcs(static_cast<uint2*>(q) + ((n * (C16 >> 1) + (j >> 1)) * HW + hw) * 2 + (j & 1), pack4_word(out));
      else
        __stcs(static_cast<uint4*>(q) + (n * C16 + j) * HW + hw, out);
    }
  }
}

// Kernel arguments: inv_s (l = 0), or with l non-NULL the learned bounds l, u.
static QuantArgs quant_args(int G, int bits, const float* inv_s, const float* l, const float* u) {
  QuantArgs args{};
  args.qp = static_cast<float>((1 << bits) - 1);
  args.lu = l != nullptr ? 1 : 0;
  for (int g = 0; g < G; ++g) {
    if (l != nullptr) {
      args.l[g] = l[g];
      args.inv_r[g] = 1.0f / (u[g] - l[g]);
    } else {
      args.inv_s[g] = inv_s[g];
    }
  }
  return args;
}

int launch_quantize_c16(const float* x, uint8_t* q, int64_t N, int64_t HW, int G, int Cg, int bits, const float* inv_s,
                        int pack, cudaStream_t stream, const float* l, const float* u) {
  const QuantArgs args = quant_args(G, bits, inv_s, l, u);
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
  const bool lu = args.lu != 0;
  if (pack == 1 && lu)
    pq_quantize_c16<1, true><<<grid, 256, 0, stream>>>(xv, q, N, HW, C16, Cg / 16, qmax, args);
  else if (pack == 1)
    pq_quantize_c16<1, false><<<grid, 256, 0, stream>>>(xv, q, N, HW, C16, Cg / 16, qmax, args);
  else if (pack == 2 && lu)
    pq_quantize_c16<2, true><<<grid, 256, 0, stream>>>(xv, q, N, HW, C16, Cg / 16, qmax, args);
  else if (pack == 2)
    pq_quantize_c16<2, false><<<grid, 256, 0, stream>>>(xv, q, N, HW, C16, Cg / 16, qmax, args);
  else if (lu)
    pq_quantize_c16<0, true><<<grid, 256, 0, stream>>>(xv, q, N, HW, C16, Cg / 16, qmax, args);
  else
    pq_quantize_c16<0, false><<<grid, 256, 0, stream>>>(xv, q, N, HW, C16, Cg / 16, qmax, args);
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
                    cudaStream_t stream, const float* l, const float* u) {
  const QuantArgs args = quant_args(G, bits, inv_s, l, u);
  const int C = G * Cg;
  const int64_t n = P * C;
  const int qmax = (1 << bits) - 1;
  if (n == 0) return 0;
  const bool aligned = (reinterpret_cast<uintptr_t>(x) % 16 == 0) && (reinterpret_cast<uintptr_t>(q) % 16 == 0);
  if (Cg % 16 == 0 && aligned) {
    const int64_t nvec = n / 16;
    const float4* xv = reinterpret_cast<const float4*>(x);
    uint4* qv = reinterpret_cast<uint4*>(q);
    if (args.lu)
      pq_quantize_vec16<true><<<quant_grid(nvec), 256, 0, stream>>>(xv, qv, nvec, C / 16, Cg / 16, qmax, args);
    else
      pq_quantize_vec16<false><<<quant_grid(nvec), 256, 0, stream>>>(xv, qv, nvec, C / 16, Cg / 16, qmax, args);
  } else if (args.lu) {
    pq_quantize_scalar<true><<<quant_grid(n), 256, 0, stream>>>(x, q, n, C, Cg, qmax, args);
  } else {
    pq_quantize_scalar<false><<<quant_grid(n), 256, 0, stream>>>(x, q, n, C, Cg, qmax, args);
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
