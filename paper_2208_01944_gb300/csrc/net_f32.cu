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

// Two fp32 fused multiply-adds in one packed instruction: (d0, d1) = (a b0 + d0,
// a b1 + d1), each with a single IEEE rounding like __fmaf_rn.
__device__ __forceinline__ void fma2_rn(float& d0, float& d1, float a, float b0, float b1) {
  asm("{\n.reg .b64 x, y, z;\nmov.b64 x, {%2, %2};\nmov.b64 y, {%3, %4};\nmov.b64 z, {%0, %1};\n"
      "fma.rn.f32x2 z, x, y, z;\nmov.b64 {%0, %1}, z;\n}"
      : "+f"(d0), "+f"(d1)
      : "f"(a), "f"(b0), "f"(b1));
}

// The 7x7 stride-2 convolution of a 3-channel image (the network's first layer),
// for Cout = 16 * CG channels (CG <= 8).  A block computes an output tile of
// 8 rows x 16 columns: warp w takes channels [16 w, 16 w + 16) and lane l the
// 4 consecutive pixels (row l / 4, columns 4 (l % 4) .. + 3), so the 16 weights
// of a term are one broadcast read.  The input tile (21 x 37 x 3 floats, zero
// outside the image) and all weights ([147][Cout]) sit in shared memory; the next
// tile's input is copied asynchronously while the current one is computed.
// Per output the terms are added in (kh, kw, ci) order like the generic kernel;
// the zero taps outside the image change nothing: fma(0, w, acc) = acc for
// finite w, since a sum started at +0 is never -0 under round-to-nearest.
constexpr int kStemK = 7, kStemS = 2, kStemP = 3, kStemCin = 3;
constexpr int kStemTH = 8, kStemTW = 16;
constexpr int kStemIR = (kStemTH - 1) * kStemS + kStemK;  // 21
constexpr int kStemIC = (kStemTW - 1) * kStemS + kStemK;  // 37
constexpr int kStemTerms = kStemK * kStemK * kStemCin;    // 147

__device__ __forceinline__ void cp_async4(float* dst, const float* src, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(d), "l"(src), "r"(valid ? 4 : 0) : "memory");
}

__global__ void __launch_bounds__(256, 2) pq_stem7x7s2_kernel(const float* __restrict__ x, const float* __restrict__ w,
                                                           float* __restrict__ y, int64_t N, int H, int W, int Cout,
                                                           int Ho, int Wo, int relu) {
  extern __shared__ float smem[];
  constexpr int kTileFloats = kStemIR * kStemIC * kStemCin;
  float* ws = smem;                          // [147][Cout]
  float* xs0 = smem + kStemTerms * Cout;     // two input tiles [21][37][3]
  const int tiles_h = (Ho + kStemTH - 1) / kStemTH, tiles_w = (Wo + kStemTW - 1) / kStemTW;
  const int64_t n_tiles = N * tiles_h * tiles_w;
  // Input tile t into buffer b with 4-byte asynchronous copies; taps outside the
  // image are zero-filled (source size 0).
  auto load_tile = [&](int64_t t, int b) {
    const int tw = static_cast<int>(t % tiles_w);
    const int64_t r = t / tiles_w;
    const int th = static_cast<int>(r % tiles_h);
    const int64_t n = r / tiles_h;
    const int ih0 = th * kStemTH * kStemS - kStemP, iw0 = tw * kStemTW * kStemS - kStemP;
    float* xs = xs0 + b * kTileFloats;
    for (int i = threadIdx.x; i < kTileFloats; i += blockDim.x) {
      const int ci = i % kStemCin;
      const int rc = i / kStemCin;
      const int c = rc % kStemIC, rr = rc / kStemIC;
      const int ih = ih0 + rr, iw = iw0 + c;
      const bool valid = ih >= 0 && ih < H && iw >= 0 && iw < W;
      cp_async4(xs + i, valid ? x + ((n * H + ih) * W + iw) * kStemCin + ci : x, valid);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  int64_t t = blockIdx.x;
  if (t < n_tiles) load_tile(t, 0);
  // transposed to [term][Cout]: consecutive threads write consecutive words
  // (conflict-free) and gather from the [Cout][term] weights through L2
  for (int i = threadIdx.x; i < kStemTerms * Cout; i += blockDim.x) {
    const int r = i / Cout, co = i - r * Cout;
    ws[i] = w[co * kStemTerms + r];
  }
  const int cg = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ohl = lane >> 2, owl = (lane & 3) * 4;
  const float* wcol = ws + cg * 16;
  int buf = 0;
  for (; t < n_tiles; t += gridDim.x, buf ^= 1) {
    __syncthreads();  // every thread is done with the buffer the next load overwrites
    if (t + gridDim.x < n_tiles) {
      load_tile(t + gridDim.x, buf ^ 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();  // tile t (and the weights) visible to all threads
    const int tw = static_cast<int>(t % tiles_w);
    const int64_t r = t / tiles_w;
    const int th = static_cast<int>(r % tiles_h);
    const int64_t n = r / tiles_h;
    const int oh0 = th * kStemTH, ow0 = tw * kStemTW;
    float acc[4][16];
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int c = 0; c < 16; ++c) acc[j][c] = 0.0f;
    const float* xrow = xs0 + buf * kTileFloats + ((ohl * kStemS) * kStemIC + owl * kStemS) * kStemCin;
#pragma unroll 1
    for (int kh = 0; kh < kStemK; ++kh) {
#pragma unroll
      for (int kw = 0; kw < kStemK; ++kw) {
#pragma unroll
        for (int ci = 0; ci < kStemCin; ++ci) {
          const int term = (kh * kStemK + kw) * kStemCin + ci;
          const float4* w4 = reinterpret_cast<const float4*>(wcol + term * Cout);
          const float4 wa = w4[0], wb = w4[1], wc = w4[2], wd = w4[3];
          const float wv[16] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w,
                                wc.x, wc.y, wc.z, wc.w, wd.x, wd.y, wd.z, wd.w};
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const float xv = xrow[(kh * kStemIC + kw + j * kStemS) * kStemCin + ci];
#pragma unroll
            for (int c = 0; c < 16; c += 2) fma2_rn(acc[j][c], acc[j][c + 1], xv, wv[c], wv[c + 1]);
          }
        }
      }
    }
    const int oh = oh0 + ohl;
    if (oh < Ho) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int ow = ow0 + owl + j;
        if (ow < Wo) {
          float4* yp = reinterpret_cast<float4*>(y + ((n * Ho + oh) * Wo + ow) * Cout + cg * 16);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float4 o = make_float4(acc[j][4 * q], acc[j][4 * q + 1], acc[j][4 * q + 2], acc[j][4 * q + 3]);
            if (relu) {
              o.x = fmaxf(o.x, 0.0f);
              o.y = fmaxf(o.y, 0.0f);
              o.z = fmaxf(o.z, 0.0f);
              o.w = fmaxf(o.w, 0.0f);
            }
            yp[q] = o;
          }
        }
      }
    }
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}

// Max over the in-image taps of each window, fmaxf in (kh, kw) order from -inf.
// One block per output row (n, oh); its threads take (ow, 4 channels) with
// 16-byte loads and stores (C % 4 == 0), so all index arithmetic is 32-bit.
__global__ void __launch_bounds__(256) pq_maxpool_f32_kernel(const float4* __restrict__ x, float4* __restrict__ y,
                                                            int H, int W, int C4, int k, int s, int p, int Ho,
                                                            int Wo) {
  const int64_t row = blockIdx.x;  // n * Ho + oh
  const int oh = static_cast<int>(row % Ho);
  const int64_t n = row / Ho;
  const float4* xi = x + n * H * W * C4;
  float4* yr = y + row * Wo * C4;
  for (int e = threadIdx.x; e < Wo * C4; e += blockDim.x) {
    const int ow = e / C4, c = e - ow * C4;
    float4 m = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    for (int kh = 0; kh < k; ++kh) {
      const int ih = oh * s - p + kh;
      if (ih < 0 || ih >= H) continue;
      for (int kw = 0; kw < k; ++kw) {
        const int iw = ow * s - p + kw;
        if (iw < 0 || iw >= W) continue;
        const float4 v = xi[(static_cast<int64_t>(ih) * W + iw) * C4 + c];
        m.x = fmaxf(m.x, v.x);
        m.y = fmaxf(m.y, v.y);
        m.z = fmaxf(m.z, v.z);
        m.w = fmaxf(m.w, v.w);
      }
    }
    yr[e] = m;
  }
}

// Any C: one thread per output element.
__global__ void __launch_bounds__(256) pq_maxpool_f32_scalar_kernel(const float* __restrict__ x, float* __restrict__ y,
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

// y[n, o] = fma over i in order of x[n, i] w[o, i] (no bias).  A block computes
// 32 outputs x 8 images (warp = one image, lane = one output); 64-wide chunks of
// x and w are staged in shared memory (w rows at pitch 65, so the lanes' reads of
// one column fall in distinct banks).  Every output keeps one running sum in
// register across the chunks, so the order of its terms is i = 0, 1, 2, ...
constexpr int kFcO = 32, kFcN = 8, kFcK = 64;

__global__ void __launch_bounds__(kFcO * kFcN) pq_linear_f32_kernel(const float* __restrict__ x,
                                                                   const float* __restrict__ w,
                                                                   float* __restrict__ y, int64_t N, int Cin,
                                                                   int Cout) {
  __shared__ float xs[kFcN][kFcK];
  __shared__ float wsh[kFcO][kFcK + 1];
  const int lane = threadIdx.x & 31, wn = threadIdx.x >> 5;
  const int o = blockIdx.x * kFcO + lane;
  const int64_t n = static_cast<int64_t>(blockIdx.y) * kFcN + wn;
  float acc = 0.0f;
  for (int c0 = 0; c0 < Cin; c0 += kFcK) {
    const int kc = min(kFcK, Cin - c0);
    __syncthreads();
    for (int i = threadIdx.x; i < kFcN * kFcK; i += blockDim.x) {
      const int r = i / kFcK, c = i - r * kFcK;
      const int64_t nn = static_cast<int64_t>(blockIdx.y) * kFcN + r;
      xs[r][c] = (c < kc && nn < N) ? x[nn * Cin + c0 + c] : 0.0f;
    }
    for (int i = threadIdx.x; i < kFcO * kFcK; i += blockDim.x) {
      const int r = i / kFcK, c = i - r * kFcK;
      const int oo = blockIdx.x * kFcO + r;
      wsh[r][c] = (c < kc && oo < Cout) ? w[static_cast<int64_t>(oo) * Cin + c0 + c] : 0.0f;
    }
    __syncthreads();
    for (int c = 0; c < kc; ++c) acc = __fmaf_rn(xs[wn][c], wsh[lane][c], acc);
  }
  if (o < Cout && n < N) y[n * Cout + o] = acc;
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
  const size_t stem_smem =
      static_cast<size_t>(pq::kStemTerms * Cout + 2 * pq::kStemIR * pq::kStemIC * pq::kStemCin) * sizeof(float);
  if (k == pq::kStemK && stride == pq::kStemS && pad == pq::kStemP && Cin == pq::kStemCin && Cout <= 128 &&
      stem_smem <= 200 * 1024) {
    static bool stem_attr = false;
    if (!stem_attr) {
      if (cudaFuncSetAttribute(pq::pq_stem7x7s2_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024) !=
          cudaSuccess)
        return PQ_ECUDA;
      stem_attr = true;
    }
    const int64_t tiles = N * ((Ho + pq::kStemTH - 1) / pq::kStemTH) * ((Wo + pq::kStemTW - 1) / pq::kStemTW);
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int per_sm = stem_smem <= 100 * 1024 ? 2 : 1;
    const unsigned grid = static_cast<unsigned>(tiles < static_cast<int64_t>(sms) * per_sm ? tiles : sms * per_sm);
    pq::pq_stem7x7s2_kernel<<<grid, 32 * (Cout / 16), stem_smem, s>>>(x_dev, w_dev, y_dev, N, H, W, Cout,
                                                                       static_cast<int>(Ho), static_cast<int>(Wo), relu);
    return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
  }
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
  auto st = static_cast<cudaStream_t>(stream);
  if (C % 4 == 0 && pq::aligned16(x_dev) && pq::aligned16(y_dev) && N * Ho <= 0x7fffffffLL) {
    pq::pq_maxpool_f32_kernel<<<static_cast<unsigned>(N * Ho), 256, 0, st>>>(
        reinterpret_cast<const float4*>(x_dev), reinterpret_cast<float4*>(y_dev), H, W, C / 4, k, stride, pad,
        static_cast<int>(Ho), static_cast<int>(Wo));
  } else {
    pq::pq_maxpool_f32_scalar_kernel<<<pq::grid_for(N * Ho * Wo * C, 8), 256, 0, st>>>(
        x_dev, y_dev, N, H, W, C, k, stride, pad, static_cast<int>(Ho), static_cast<int>(Wo));
  }
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
  const int64_t gy = (N + pq::kFcN - 1) / pq::kFcN;
  if (gy > 65535) return PQ_EUNSUPPORTED;
  const dim3 grid(static_cast<unsigned>((Cout + pq::kFcO - 1) / pq::kFcO), static_cast<unsigned>(gy));
  pq::pq_linear_f32_kernel<<<grid, pq::kFcO * pq::kFcN, 0, static_cast<cudaStream_t>(stream)>>>(x_dev, w_dev, y_dev,
                                                                                               N, Cin, Cout);
  return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
}

}  // extern "C"
