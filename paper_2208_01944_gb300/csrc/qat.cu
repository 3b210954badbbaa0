// Quantisation-aware training forward and backward of PalQuant's quantiser
// (Sec. 3.2 Eq. 2-3 with learned per-group bounds l, u; Sec. 5: the rounding is
// passed by the straight-through estimator).  Elementwise over x [P][G*Cg]
// (group g = channel / Cg), bound by HBM: the forward reads 4 and writes 4
// bytes per element, the backward reads 8 and writes 4; the backward also sums
// the gradients of l and u per group in a fixed partition (deterministic).
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstring>

#include "palquant.h"
#include "pq_internal.h"

namespace pq {
namespace {

constexpr int kQatThreads = 256;
constexpr int kQatMaxBlocks = 512;  // blocks per group (partition of the backward sums)

struct QatParams {
  float l[kMaxG];
  float u[kMaxG];
  float inv_r[kMaxG];  // fl(1 / fl(u - l))
  float k[kMaxG];      // c * inv_r: the input gradient's factor
  float qp, inv_qp;    // 2^b - 1 and fl(1 / (2^b - 1))
  int kind;            // 0 activations (x_hat in [0, 1]), 1 weights ([-1, 1])
  int64_t C4;          // float4s per row (G * Cg / 4)
  uint32_t cq;         // float4s of one group in a row (Cg / 4)
  uint32_t cq_magic;   // ceil(2^32 / cq) (cq > 1)
  uint32_t quads;      // P * cq, float4s of one group
};

// e / cq for e < 2^32: umulhi(e, ceil(2^32 / cq)) is e / cq or one more, so one
// correction makes it exact.
__device__ __forceinline__ uint32_t div_cq(uint32_t e, const QatParams& q) {
  if (q.cq == 1) return e;
  uint32_t d = __umulhi(e, q.cq_magic);
  if (static_cast<uint64_t>(d) * q.cq > e) --d;
  return d;
}

// Round half to even of 0 <= y <= 2^22: the fp32 add of 1.5 * 2^23 rounds the
// sum to an integer (IEEE round to nearest even), the subtraction is exact.
__device__ __forceinline__ float round_small(float y) {
  return __fsub_rn(__fadd_rn(y, 12582912.0f), 12582912.0f);
}

// float4 index of quad e (of group g's P * cq quads, row-major) in x [P][G*Cg].
__device__ __forceinline__ int64_t quad_index(uint32_t e, int g, const QatParams& q) {
  const uint32_t p = div_cq(e, q);
  return static_cast<int64_t>(p) * q.C4 + static_cast<int64_t>(g) * q.cq + (e - p * q.cq);
}

// t = fl(fl(x - l) * inv_r), one rounding per operation.
__device__ __forceinline__ float qat_t(float x, float l, float inv_r) { return __fmul_rn(__fsub_rn(x, l), inv_r); }

__device__ __forceinline__ float qat_fwd1(float x, float l, float inv_r, const QatParams& q) {
  const float xn = fminf(fmaxf(qat_t(x, l, inv_r), 0.0f), 1.0f);  // NaN -> 0
  const float xq = round_small(__fmul_rn(xn, q.qp));
  const float v = __fmul_rn(xq, q.inv_qp);
  return q.kind ? __fmul_rn(2.0f, __fsub_rn(v, 0.5f)) : v;
}

// Blocks: G per part of the row range, the groups fastest in launch order, so
// the blocks that run together read whole rows (DRAM pages), not one group's
// slice of every row.
__global__ void __launch_bounds__(kQatThreads) pq_fake_quant_fwd(const float4* __restrict__ x, float4* __restrict__ y,
                                                                 int G, const __grid_constant__ QatParams q) {
  const int g = static_cast<int>(blockIdx.x % G);
  const uint32_t b = blockIdx.x / G, nb = gridDim.x / G;
  const float l = q.l[g], inv_r = q.inv_r[g];
  const uint32_t e0 = static_cast<uint32_t>(static_cast<uint64_t>(b) * q.quads / nb);
  const uint32_t e1 = static_cast<uint32_t>(static_cast<uint64_t>(b + 1) * q.quads / nb);
  // two float4s per thread and pass, both loads issued before either is used
  for (uint32_t e = e0 + threadIdx.x; e < e1; e += 2 * kQatThreads) {
    const bool two = e + kQatThreads < e1;
    const int64_t i0 = quad_index(e, g, q);
    const int64_t i1 = two ? quad_index(e + kQatThreads, g, q) : i0;
    const float4 v0 = __ldcs(x + i0);
    const float4 v1 = two ? __ldcs(x + i1) : v0;
    __stcs(y + i0, make_float4(qat_fwd1(v0.x, l, inv_r, q), qat_fwd1(v0.y, l, inv_r, q), qat_fwd1(v0.z, l, inv_r, q),
                               qat_fwd1(v0.w, l, inv_r, q)));
    if (two)
      __stcs(y + i1, make_float4(qat_fwd1(v1.x, l, inv_r, q), qat_fwd1(v1.y, l, inv_r, q),
                                 qat_fwd1(v1.z, l, inv_r, q), qat_fwd1(v1.w, l, inv_r, q)));
  }
}

// Compensated fp32 sum (Kahan): s + c carries the exact running sum to within
// about two roundings of the sum of magnitudes, whatever the number of terms.
struct KahanF {
  float s = 0.0f, c = 0.0f;
  __device__ __forceinline__ void add(float v) {
    const float y = __fsub_rn(v, c);
    const float t = __fadd_rn(s, y);
    c = __fsub_rn(__fsub_rn(t, s), y);
    s = t;
  }
};

// Backward: dx = dy * k inside 0 < t < 1, else 0; per block the sums of
// dy (x - u) and dy (x - l) over the inside elements of the block's range (fp32
// products, four summed in fp32, the thread's quads in a compensated fp32 sum,
// the threads in double), written to partial[g][block].  (Double arithmetic per
// element would cost more than the memory traffic: the FP64 rate is low here.)
// At most 32 registers per thread (12 bytes of spills): eight blocks per SM, so
// the grid runs in as few waves as the forward's.
__global__ void __launch_bounds__(kQatThreads, 8) pq_fake_quant_bwd(const float4* __restrict__ x,
                                                                 const float4* __restrict__ dy,
                                                                 float4* __restrict__ dx, double2* __restrict__ partial,
                                                                 int G, const __grid_constant__ QatParams q) {
  const int g = static_cast<int>(blockIdx.x % G);
  const uint32_t b = blockIdx.x / G, nb = gridDim.x / G;
  const float l = q.l[g], u = q.u[g], inv_r = q.inv_r[g], k = q.k[g];
  const uint32_t e0 = static_cast<uint32_t>(static_cast<uint64_t>(b) * q.quads / nb);
  const uint32_t e1 = static_cast<uint32_t>(static_cast<uint64_t>(b + 1) * q.quads / nb);
  KahanF ka, kb;
  auto quad = [&](int64_t i, const float4& xv, const float4& dv) {
    const float xs[4] = {xv.x, xv.y, xv.z, xv.w};
    const float ds[4] = {dv.x, dv.y, dv.z, dv.w};
    float o[4];
    float a = 0.0f, b = 0.0f;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const float t = qat_t(xs[c], l, inv_r);
      const bool in = t > 0.0f && t < 1.0f;
      o[c] = in ? __fmul_rn(ds[c], k) : 0.0f;
      a = __fadd_rn(a, in ? __fmul_rn(ds[c], __fsub_rn(xs[c], u)) : 0.0f);
      b = __fadd_rn(b, in ? __fmul_rn(ds[c], __fsub_rn(xs[c], l)) : 0.0f);
    }
    __stcs(dx + i, make_float4(o[0], o[1], o[2], o[3]));
    ka.add(a);
    kb.add(b);
  };
  // two float4s of x and dy per thread and pass, all four loads issued first
  for (uint32_t e = e0 + threadIdx.x; e < e1; e += 2 * kQatThreads) {
    const bool two = e + kQatThreads < e1;
    const int64_t i0 = quad_index(e, g, q);
    const int64_t i1 = two ? quad_index(e + kQatThreads, g, q) : i0;
    const float4 x0 = __ldcs(x + i0), d0 = __ldcs(dy + i0);
    const float4 x1 = two ? __ldcs(x + i1) : x0;
    const float4 d1 = two ? __ldcs(dy + i1) : d0;
    quad(i0, x0, d0);
    if (two) quad(i1, x1, d1);
  }
  double sa = static_cast<double>(ka.s) - static_cast<double>(ka.c);
  double sb = static_cast<double>(kb.s) - static_cast<double>(kb.c);
  // fixed-order block reduction: warps by shuffles, then warp 0 over the warps
  __shared__ double2 red[kQatThreads / 32];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    sa += __shfl_down_sync(0xffffffffu, sa, off);
    sb += __shfl_down_sync(0xffffffffu, sb, off);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = make_double2(sa, sb);
  __syncthreads();
  if (threadIdx.x == 0) {
    double ta = 0.0, tb = 0.0;
    for (int w = 0; w < kQatThreads / 32; ++w) {
      ta += red[w].x;
      tb += red[w].y;
    }
    partial[static_cast<int64_t>(g) * nb + b] = make_double2(ta, tb);
  }
}

// dl[g] = c / r^2 * sum_a, du[g] = -c / r^2 * sum_b (r = u - l in double): one
// block per group; thread t adds block sums t, t + 256, ... in order, then a
// fixed tree over the threads (deterministic).
__global__ void __launch_bounds__(kQatThreads) pq_fake_quant_bwd_finish(const double2* __restrict__ partial,
                                                                        int nblocks, double c,
                                                                        const __grid_constant__ QatParams q,
                                                                        double* __restrict__ dl,
                                                                        double* __restrict__ du) {
  const int g = blockIdx.x;
  double sa = 0.0, sb = 0.0;
  for (int b = threadIdx.x; b < nblocks; b += kQatThreads) {
    const double2 v = partial[static_cast<int64_t>(g) * nblocks + b];
    sa += v.x;
    sb += v.y;
  }
  __shared__ double2 red[kQatThreads];
  red[threadIdx.x] = make_double2(sa, sb);
  __syncthreads();
  for (int w = kQatThreads / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) {
      red[threadIdx.x].x += red[threadIdx.x + w].x;
      red[threadIdx.x].y += red[threadIdx.x + w].y;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const double r = static_cast<double>(q.u[g]) - static_cast<double>(q.l[g]);
    dl[g] = c / (r * r) * red[0].x;
    du[g] = -c / (r * r) * red[0].y;
  }
}

// Blocks per group: enough to fill the GPU at the benchmark sizes, fixed by the
// problem size only (so the partition, and the sums, do not depend on the device).
int qat_blocks(uint32_t quads) {
  const uint64_t per = kQatThreads * 8u;  // about eight float4s per thread
  uint64_t nb = (static_cast<uint64_t>(quads) + per - 1) / per;
  if (nb < 1) nb = 1;
  if (nb > kQatMaxBlocks) nb = kQatMaxBlocks;
  return static_cast<int>(nb);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

pq_status qat_params(int64_t P, int32_t G, int32_t Cg, int32_t bits, int32_t kind, const float* l_host,
                     const float* u_host, QatParams* q) {
  if (P < 0 || G < 1 || G > kMaxG || Cg < 4 || Cg % 4 != 0 || bits < 1 || bits > 8 || (kind != 0 && kind != 1))
    return PQ_EINVAL;
  if (l_host == nullptr || u_host == nullptr) return PQ_EINVAL;
  const uint64_t quads = static_cast<uint64_t>(P) * static_cast<uint64_t>(Cg / 4);
  if (quads >= (1ull << 32)) return PQ_EUNSUPPORTED;
  std::memset(q, 0, sizeof(*q));
  const float c = kind ? 2.0f : 1.0f;
  for (int g = 0; g < G; ++g) {
    const float l = l_host[g], u = u_host[g];
    if (!std::isfinite(l) || !std::isfinite(u) || !(u > l)) return PQ_EINVAL;
    const float r = u - l;
    if (!std::isfinite(r) || !(r > 0.0f)) return PQ_EINVAL;
    q->l[g] = l;
    q->u[g] = u;
    q->inv_r[g] = 1.0f / r;
    if (!std::isfinite(q->inv_r[g])) return PQ_EINVAL;
    q->k[g] = c * q->inv_r[g];
  }
  q->qp = static_cast<float>((1 << bits) - 1);
  q->inv_qp = 1.0f / q->qp;
  q->kind = kind;
  q->C4 = static_cast<int64_t>(G) * (Cg / 4);
  q->cq = static_cast<uint32_t>(Cg / 4);
  q->cq_magic = q->cq > 1 ? static_cast<uint32_t>(((1ull << 32) + q->cq - 1) / q->cq) : 0u;
  q->quads = static_cast<uint32_t>(quads);
  return PQ_OK;
}

}  // namespace
}  // namespace pq

extern "C" {

pq_status palquant_fake_quant_forward(const float* x_dev, float* xhat_dev, int64_t P, int32_t G, int32_t Cg,
                                      int32_t bits, int32_t kind, const float* l_host, const float* u_host,
                                      pq_stream_t stream) {
  pq::QatParams q;
  const pq_status st = pq::qat_params(P, G, Cg, bits, kind, l_host, u_host, &q);
  if (st != PQ_OK) return st;
  if (P == 0) return PQ_OK;  // no elements (the pointers may be NULL)
  if (x_dev == nullptr || xhat_dev == nullptr || !pq::aligned16(x_dev) || !pq::aligned16(xhat_dev)) return PQ_EINVAL;
  const unsigned grid = static_cast<unsigned>(pq::qat_blocks(q.quads)) * G;
  pq::pq_fake_quant_fwd<<<grid, pq::kQatThreads, 0, static_cast<cudaStream_t>(stream)>>>(
      reinterpret_cast<const float4*>(x_dev), reinterpret_cast<float4*>(xhat_dev), G, q);
  return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
}

size_t palquant_fake_quant_scratch_bytes(int64_t P, int32_t G, int32_t Cg) {
  if (P < 0 || G < 1 || Cg < 4) return 0;
  const uint64_t quads = static_cast<uint64_t>(P) * static_cast<uint64_t>(Cg / 4);
  if (quads >= (1ull << 32)) return 0;
  return sizeof(double2) * static_cast<size_t>(G) * static_cast<size_t>(pq::qat_blocks(static_cast<uint32_t>(quads)));
}

pq_status palquant_fake_quant_backward(const float* x_dev, const float* dy_dev, float* dx_dev, double* dl_dev,
                                       double* du_dev, int64_t P, int32_t G, int32_t Cg, int32_t bits, int32_t kind,
                                       const float* l_host, const float* u_host, void* scratch_dev,
                                       size_t scratch_bytes, pq_stream_t stream) {
  pq::QatParams q;
  const pq_status st = pq::qat_params(P, G, Cg, bits, kind, l_host, u_host, &q);
  if (st != PQ_OK) return st;
  if (dl_dev == nullptr || du_dev == nullptr || (reinterpret_cast<uintptr_t>(dl_dev) & 7u) ||
      (reinterpret_cast<uintptr_t>(du_dev) & 7u))
    return PQ_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const double c = kind ? 2.0 : 1.0;
  if (P == 0) {  // no elements: zero gradients (the element pointers and the scratch may be NULL)
    pq::pq_fake_quant_bwd_finish<<<G, pq::kQatThreads, 0, s>>>(nullptr, 0, c, q, dl_dev, du_dev);
    return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
  }
  if (x_dev == nullptr || dy_dev == nullptr || dx_dev == nullptr || scratch_dev == nullptr) return PQ_EINVAL;
  if (!pq::aligned16(x_dev) || !pq::aligned16(dy_dev) || !pq::aligned16(dx_dev) || !pq::aligned16(scratch_dev))
    return PQ_EINVAL;
  if (scratch_bytes < palquant_fake_quant_scratch_bytes(P, G, Cg)) return PQ_EINVAL;
  const int nb = pq::qat_blocks(q.quads);
  double2* partial = static_cast<double2*>(scratch_dev);
  pq::pq_fake_quant_bwd<<<static_cast<unsigned>(nb) * G, pq::kQatThreads, 0, s>>>(
      reinterpret_cast<const float4*>(x_dev), reinterpret_cast<const float4*>(dy_dev),
      reinterpret_cast<float4*>(dx_dev), partial, G, q);
  if (cudaGetLastError() != cudaSuccess) return PQ_ECUDA;
  pq::pq_fake_quant_bwd_finish<<<G, pq::kQatThreads, 0, s>>>(partial, nb, c, q, dl_dev, du_dev);
  return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
}

}  // extern "C"
