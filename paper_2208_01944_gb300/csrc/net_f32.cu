// Full-precision layers around the PalQuant body of a ResNet-18-shaped network:
// the paper keeps the first and the last layer in full precision (Sec. 5).  They
// are off the quantised hot path, but they feed the first quantiser, so every
// output is summed in one fixed order with one fused multiply-add per term
// (__fmaf_rn, a single IEEE rounding); that makes each value independent of how
// the work is spread over threads.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "palquant.h"
#include "pq_internal.h"

namespace pq {
namespace {

constexpr int kCoT = 16;          // output channels per thread
constexpr int kF32Threads = 256;

// Direct NHWC convolution, weights [Cout][k][k][Cin] staged in shared memory as
// [k*k*Cin][Cout] (when they fit) so that the kCoT channels of one term are
// contiguous.  Thread index: pixel fastest, so a warp shares its channel group
// and reads each weight as a broadcast.  Per output: acc = 0, then
// acc = fma(x, w, acc) over (kh, kw, ci) in that order, skipping taps outside
// the image.
template <bool SMEM_W>
__global__ void __launch_bounds__(kF32Threads) pq_conv2d_f32_kernel(const float* __restrict__ x,
                                                                   const float* __restrict__ w, float* __restrict__ y,
                                                                   int64_t N, int H, int W, int Cin, int Cout, int k,
                                                                   int s, int p, int Ho, int Wo, int relu) {
  extern __shared__ float wsm[];
  const int kkc = k * k * Cin;
  if (SMEM_W) {
    for (int i = threadIdx.x; i < kkc * Cout; i += blockDim.x) {
      const int co = i / kkc, r = i - co * kkc;
      wsm[r * Cout + co] = w[i];
    }
    __syncthreads();
  }
  const int64_t P = N * Ho * Wo;
  const int64_t total = P * (Cout / kCoT);
  for (int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int cg = static_cast<int>(idx / P);
    const int64_t pix = idx - cg * P;
    const int ow = static_cast<int>(pix % Wo);
    const int64_t t = pix / Wo;
    const int oh = static_cast<int>(t % Ho);
    const int64_t n = t / Ho;
    const int co0 = cg * kCoT;
    float acc[kCoT];
#pragma unroll
    for (int j = 0; j < kCoT; ++j) acc[j] = 0.0f;
    for (int kh = 0; kh < k; ++kh) {
      const int ih = oh * s - p + kh;
      if (ih < 0 || ih >= H) continue;
      for (int kw = 0; kw < k; ++kw) {
        const int iw = ow * s - p + kw;
        if (iw < 0 || iw >= W) continue;
        const float* xp = x + ((n * H + ih) * W + iw) * Cin;
        const int r0 = (kh * k + kw) * Cin;
        for (int ci = 0; ci < Cin; ++ci) {
          const float xv = xp[ci];
          if (SMEM_W) {
            const float4* wr = reinterpret_cast<const float4*>(wsm + (r0 + ci) * Cout + co0);
#pragma unroll
            for (int q = 0; q < kCoT / 4; ++q) {
              const float4 w4 = wr[q];
              acc[4 * q] = __fmaf_rn(xv, w4.x, acc[4 * q]);
              acc[4 * q + 1] = __fmaf_rn(xv, w4.y, acc[4 * q + 1]);
              acc[4 * q + 2] = __fmaf_rn(xv, w4.z, acc[4 * q + 2]);
              acc[4 * q + 3] = __fmaf_rn(xv, w4.w, acc[4 * q + 3]);
            }
          } else {
#pragma unroll
            for (int j = 0; j < kCoT; ++j) acc[j] = __fmaf_rn(xv, w[static_cast<int64_t>(co0 + j) * kkc + r0 + ci], acc[j]);
          }
        }
      }
    }
    float* yp = y + pix * Cout + co0;
#pragma unroll
    for (int q = 0; q < kCoT / 4; ++q) {
      float4 o = make_float4(acc[4 * q], acc[4 * q + 1], acc[4 * q + 2], acc[4 * q + 3]);
      if (relu) {
        o.x = fmaxf(o.x, 0.0f);
        o.y = fmaxf(o.y, 0.0f);
        o.z = fmaxf(o.z, 0.0f);
        o.w = fmaxf(o.w, 0.0f);
      }
      reinterpret_cast<float4*>(yp)[q] = o;
    }
  }
}

// Max over the in-image taps of each window, fmaxf in (kh, kw) order from -inf.
__global__ void __launch_bounds__(256) pq_maxpool_f32_kernel(const float* __restrict__ x, float* __restrict__ y,
                                                            int64_t N, int H, int W, int C, int k, int s, int p,
                                                            int Ho, int Wo) {
  const int64_t total = N * Ho * Wo * C;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(i % C);
    const int64_t pix = i / C;
    const int ow = static_cast<int>(pix % Wo);
    const int64_t t = pix / Wo;
    const int oh = static_cast<int>(t % Ho);
    const int64_t n = t / Ho;
    float m = -INFINITY;
    for (int kh = 0; kh < k; ++kh) {
      const int ih = oh * s - p + kh;
      if (ih < 0 || ih >= H) continue;
      for (int kw = 0; kw < k; ++kw) {
        const int iw = ow * s - p + kw;
        if (iw < 0 || iw >= W) continue;
        m = fmaxf(m, x[((n * H + ih) * W + iw) * C + c]);
      }
    }
    y[i] = m;
  }
}

// Sum over (h, w) in storage order from 0, then one division by H * W.
__global__ void __launch_bounds__(256) pq_avgpool_f32_kernel(const float* __restrict__ x, float* __restrict__ y,
                                                            int64_t N, int HW, int C) {
  const int64_t total = N * C;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(i % C);
    const int64_t n = i / C;
    float acc = 0.0f;
    for (int j = 0; j < HW; ++j) acc = __fadd_rn(acc, x[(n * HW + j) * C + c]);
    y[i] = __fdiv_rn(acc, static_cast<float>(HW));
  }
}

// y[n, o] = fma over i in order of x[n, i] w[o, i] (no bias).
__global__ void __launch_bounds__(256) pq_linear_f32_kernel(const float* __restrict__ x, const float* __restrict__ w,
                                                           float* __restrict__ y, int64_t N, int Cin, int Cout) {
  const int64_t total = N * Cout;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int o = static_cast<int>(i % Cout);
    const int64_t n = i / Cout;
    const float* xr = x + n * Cin;
    const float* wr = w + static_cast<int64_t>(o) * Cin;
    float acc = 0.0f;
    for (int c = 0; c < Cin; ++c) acc = __fmaf_rn(xr[c], wr[c], acc);
    y[i] = acc;
  }
}

unsigned grid_for(int64_t work, int per_sm) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (work + 255) / 256;
  const int64_t cap = static_cast<int64_t>(sms) * per_sm;
  return static_cast<unsigned>(want < cap ? (want > 0 ? want : 1) : cap);
}

int64_t out_dim(int64_t n, int k, int s, int p) { return (n + 2 * p - k) / s + 1; }

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

}  // namespace
}  // namespace pq

extern "C" {

pq_status palquant_conv2d_f32(const float* x_dev, const float* w_dev, float* y_dev, int64_t N, int32_t H, int32_t W,
                              int32_t Cin, int32_t Cout, int32_t k, int32_t stride, int32_t pad, int32_t relu,
                              pq_stream_t stream) {
  if (N < 0 || H <= 0 || W <= 0 || Cin <= 0 || Cout <= 0 || k <= 0 || stride <= 0 || pad < 0 || pad >= k)
    return PQ_EINVAL;
  if (!x_dev || !w_dev || !y_dev || !pq::aligned16(y_dev) || Cout % pq::kCoT != 0) return PQ_EINVAL;
  const int64_t Ho = pq::out_dim(H, k, stride, pad), Wo = pq::out_dim(W, k, stride, pad);
  if (Ho <= 0 || Wo <= 0) return PQ_EINVAL;
  if (N == 0) return PQ_OK;
  const int64_t wbytes = static_cast<int64_t>(k) * k * Cin * Cout * 4;
  const int64_t work = N * Ho * Wo * (Cout / pq::kCoT);
  auto s = static_cast<cudaStream_t>(stream);
  if (wbytes <= 96 * 1024) {
    static bool attr_set = false;
    if (!attr_set) {
      if (cudaFuncSetAttribute(pq::pq_conv2d_f32_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               96 * 1024) != cudaSuccess)
        return PQ_ECUDA;
      attr_set = true;
    }
    pq::pq_conv2d_f32_kernel<true><<<pq::grid_for(work, 2), pq::kF32Threads, static_cast<size_t>(wbytes), s>>>(
        x_dev, w_dev, y_dev, N, H, W, Cin, Cout, k, stride, pad, static_cast<int>(Ho), static_cast<int>(Wo), relu);
  } else {
    pq::pq_conv2d_f32_kernel<false><<<pq::grid_for(work, 8), pq::kF32Threads, 0, s>>>(
        x_dev, w_dev, y_dev, N, H, W, Cin, Cout, k, stride, pad, static_cast<int>(Ho), static_cast<int>(Wo), relu);
  }
  return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
}

pq_status palquant_maxpool2d_f32(const float* x_dev, float* y_dev, int64_t N, int32_t H, int32_t W, int32_t C,
                                 int32_t k, int32_t stride, int32_t pad, pq_stream_t stream) {
  if (N < 0 || H <= 0 || W <= 0 || C <= 0 || k <= 0 || stride <= 0 || pad < 0 || pad >= k) return PQ_EINVAL;
  if (!x_dev || !y_dev) return PQ_EINVAL;
  const int64_t Ho = pq::out_dim(H, k, stride, pad), Wo = pq::out_dim(W, k, stride, pad);
  if (Ho <= 0 || Wo <= 0) return PQ_EINVAL;
  if (N == 0) return PQ_OK;
  pq::pq_maxpool_f32_kernel<<<pq::grid_for(N * Ho * Wo * C, 8), 256, 0, static_cast<cudaStream_t>(stream)>>>(
      x_dev, y_dev, N, H, W, C, k, stride, pad, static_cast<int>(Ho), static_cast<int>(Wo));
  return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
}

pq_status palquant_avgpool_f32(const float* x_dev, float* y_dev, int64_t N, int32_t H, int32_t W, int32_t C,
                               pq_stream_t stream) {
  if (N < 0 || H <= 0 || W <= 0 || C <= 0 || !x_dev || !y_dev) return PQ_EINVAL;
  if (N == 0) return PQ_OK;
  pq::pq_avgpool_f32_kernel<<<pq::grid_for(N * C, 8), 256, 0, static_cast<cudaStream_t>(stream)>>>(x_dev, y_dev, N,
                                                                                                    H * W, C);
  return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
}

pq_status palquant_linear_f32(const float* x_dev, const float* w_dev, float* y_dev, int64_t N, int32_t Cin,
                              int32_t Cout, pq_stream_t stream) {
  if (N < 0 || Cin <= 0 || Cout <= 0 || !x_dev || !w_dev || !y_dev) return PQ_EINVAL;
  if (N == 0) return PQ_OK;
  pq::pq_linear_f32_kernel<<<pq::grid_for(N * Cout, 8), 256, 0, static_cast<cudaStream_t>(stream)>>>(x_dev, w_dev,
                                                                                                     y_dev, N, Cin, Cout);
  return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
}

}  // extern "C"
