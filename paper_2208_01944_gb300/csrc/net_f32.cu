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

// The 7x7 stride-2 convolution of a 3-channel image to 128 channels (the
// network's first layer).  One block of 256 threads per SM computes output
// tiles of 16 rows x 16 columns; thread (row r, channel group g) holds the 16
// pixels of tile row r and the 8 channels 8 g .. 8 g + 7: 128 sums, so that a
// term costs four 16-byte input loads, two 16-byte weight loads and 64 packed
// FMAs, with the registers to load the next term's operands while the current
// one's FMAs run.  The input window of a tile (37 x 37 x 3 floats, zero outside
// the image) is held split by column parity, channel-planar, in four copies
// shifted by 0..3 positions: copy s of parity b holds at row i, position k the
// window's column 2 (k + s) + b, so the 16 inputs of a thread for tap (kh, kw)
// are positions 0..15, aligned, of copy kw / 2, parity kw % 2, row 2 r + kh.
// The next tile's window comes into a plain copy in shared memory by cp.async
// while the current one is computed, and is split into the copies between the
// tile's two barriers.  The weights of a term are stored as two
// halves of 4 channels per group ([147][2][16][4]): the 16 groups of a warp
// read 256 contiguous bytes.  Per output the terms are added in (kh, kw, ci)
// order like the generic kernel; the zero taps outside the image change
// nothing: fma(0, w, acc) = acc for finite w, since a sum started at +0 is
// never -0 under round-to-nearest.
constexpr int kStemK = 7, kStemS = 2, kStemP = 3, kStemCin = 3, kStemCout = 128;
constexpr int kStemTH = 16, kStemTW = 16;
constexpr int kStemThreads = 256;
constexpr int kStemIR = (kStemTH - 1) * kStemS + kStemK;  // 37 input rows
constexpr int kStemIC = (kStemTW - 1) * kStemS + kStemK;  // 37 input columns
constexpr int kStemTerms = kStemK * kStemK * kStemCin;    // 147
constexpr int kStemRowF = 16;                             // positions per copy row
constexpr int kStemPlaneF = kStemIR * kStemRowF;          // one (copy, parity, channel) plane
constexpr int kStemCopyF = 2 * kStemCin * kStemPlaneF;    // one shifted copy
constexpr int kStemXFloats = 4 * kStemCopyF;              // one window
constexpr int kStemTileElems = kStemIR * kStemIC * kStemCin;                     // 4107
constexpr int kStemLoads = (kStemTileElems + kStemThreads - 1) / kStemThreads;  // 17 per thread
constexpr int kStemPoolRowF = 9 * kStemCout;  // a staged row of pooled columns (max pooling)
constexpr int kStemRawF = (kStemTileElems + 3) / 4 * 4;  // the next window as it lies in the image
constexpr size_t kStemSmem = (static_cast<size_t>(kStemTerms) * kStemCout + kStemXFloats + kStemRawF +
                              (kStemTH / 2) * kStemPoolRowF) * sizeof(float);

// Packed fp32 pairs in one 64-bit register (the low half first), and the packed
// fused multiply-add on them: d = a b + d lane by lane, each lane with a single
// IEEE rounding like __fmaf_rn.
__device__ __forceinline__ unsigned long long f32x2_pair(float lo, float hi) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f32x2_unpair(unsigned long long v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ void ffma2(unsigned long long& d, unsigned long long a, unsigned long long b) {
  asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(d) : "l"(a), "l"(b));
}

// One 4-byte asynchronous copy global -> shared, zero-filled when !valid.
__device__ __forceinline__ void cp_async4(float* dst, const float* src, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(d), "l"(src), "r"(valid ? 4 : 0) : "memory");
}

// 3x3 stride-2 pad-1 max pooling of the stem tile held in registers (ReLU
// outputs, so every value is >= 0, and pixels outside the output are 0).
// Pooled row pr (0..8) of the tile covers stem rows 2 pr - 1 .. 2 pr + 1 and
// pooled column pc (0..8) stem columns 2 pc - 1 .. 2 pc + 1 (tile-relative).
// Columns: each thread reduces its row's 16 pixels to the 9 windows it sees.
// Rows: the odd rows go through shared memory (`stage`) to the even rows'
// threads, which complete pooled rows 1..7.  Windows that reach into a
// neighbouring tile (pooled row 0 and 8, pooled column 0 and 8) are combined
// across tiles by an integer atomic maximum on the float bits (the order of
// non-negative floats), into an output the launcher zeroed; the others are
// stored.  The maximum is exact, so the result does not depend on the order.
// `staged` runs between the caller's two barriers: odd rows write, even rows read.
__device__ __forceinline__ void stem_pool_rows(const float (&acc)[16][8], float (&h)[9][8]) {
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    h[0][c] = fmaxf(acc[0][c], acc[1][c]);
#pragma unroll
    for (int k = 1; k < 8; ++k) h[k][c] = fmaxf(fmaxf(acc[2 * k - 1][c], acc[2 * k][c]), acc[2 * k + 1][c]);
    h[8][c] = acc[15][c];
  }
}

__global__ void __launch_bounds__(kStemThreads, 1) pq_stem7x7s2_kernel(const float* __restrict__ x,
                                                                     const float* __restrict__ w,
                                                                     float* __restrict__ y, float* __restrict__ pool,
                                                                     int64_t N, int H, int W, int Ho, int Wo, int Hp,
                                                                     int Wp, int relu) {
  extern __shared__ float4 smem4[];
  float* ws = reinterpret_cast<float*>(smem4);  // [147][2][16][4]
  float* xs = ws + kStemTerms * kStemCout;      // the window [copy 4][parity 2][ci 3][row 37][16]
  float* raw = xs + kStemXFloats;               // the next window [row 37][column 37][ci 3]
  float* pstage = raw + kStemRawF;              // odd rows' pooled columns [8][9][128]
  const int tiles_h = (Ho + kStemTH - 1) / kStemTH, tiles_w = (Wo + kStemTW - 1) / kStemTW;
  const int64_t n_tiles = N * tiles_h * tiles_w;
  // Tile t's window (element i = (row, column, channel) of the 37 x 37 x 3
  // window, i = threadIdx.x + 256 e) into `raw` by 4-byte cp.async, zero-filled
  // outside the image.
  auto fetch = [&](int64_t t) {
    const int tw = static_cast<int>(t % tiles_w);
    const int64_t r = t / tiles_w;
    const int th = static_cast<int>(r % tiles_h);
    const int64_t n = r / tiles_h;
    const int ih0 = th * kStemTH * kStemS - kStemP, iw0 = tw * kStemTW * kStemS - kStemP;
#pragma unroll
    for (int e = 0; e < kStemLoads; ++e) {
      const int i = threadIdx.x + e * kStemThreads;
      const int rr = i / (kStemIC * kStemCin), rem = i - rr * (kStemIC * kStemCin);
      const int c = rem / kStemCin, ci = rem - c * kStemCin;
      const int ih = ih0 + rr, iw = iw0 + c;
      const bool valid = ih >= 0 && ih < H && iw >= 0 && iw < W;
      if (i < kStemTileElems) cp_async4(raw + i, valid ? x + ((n * H + ih) * W + iw) * kStemCin + ci : x, valid);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  // The fetched window into the four shifted copies of its parity planes.
  auto scatter = [&]() {
#pragma unroll
    for (int e = 0; e < kStemLoads; ++e) {
      const int i = threadIdx.x + e * kStemThreads;
      if (i < kStemTileElems) {
        const float v = raw[i];
        const int rr = i / (kStemIC * kStemCin), rem = i - rr * (kStemIC * kStemCin);
        const int c = rem / kStemCin, ci = rem - c * kStemCin;
        const int k0 = c >> 1;
        float* dst = xs + ((c & 1) * kStemCin + ci) * kStemPlaneF + rr * kStemRowF + k0;
#pragma unroll
        for (int sh = 0; sh < 4; ++sh)
          if (k0 - sh >= 0 && k0 - sh < kStemRowF) dst[sh * kStemCopyF - sh] = v;
      }
    }
  };
  int64_t t = blockIdx.x;
  if (t < n_tiles) fetch(t);
  // weights [Cout][147] to [147][2][16][4]: channel co = 8 g + 4 h + k at
  // term * 128 + h * 64 + g * 4 + k (consecutive threads write consecutive words)
  for (int i = threadIdx.x; i < kStemTerms * kStemCout; i += kStemThreads) {
    const int term = i >> 7, rem = i & 127;
    const int h = rem >> 6, g = (rem >> 2) & 15, k = rem & 3;
    ws[i] = w[(g * 8 + h * 4 + k) * kStemTerms + term];
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();  // the first window landed
  scatter();
  __syncthreads();  // the first window's copies and the weights visible to all threads
  const int cg = threadIdx.x & 15, r = threadIdx.x >> 4;  // channel group, tile row
  const float* wthr = ws + cg * 4;
  const float* xthr = xs + (2 * r) * kStemRowF;
  for (; t < n_tiles; t += gridDim.x) {
    const bool more = t + gridDim.x < n_tiles;
    if (more) fetch(t + gridDim.x);  // in flight during the FMAs
    // the sums of pixel j, channels 2 k and 2 k + 1, as one 64-bit register pair
    unsigned long long a2[16][4];
#pragma unroll
    for (int j = 0; j < 16; ++j)
#pragma unroll
      for (int k = 0; k < 4; ++k) a2[j][k] = 0ull;
#pragma unroll 1
    for (int kh = 0; kh < kStemK; ++kh) {
      const float* xk = xthr + kh * kStemRowF;
      const float* wk = wthr + kh * (kStemK * kStemCin) * kStemCout;
#pragma unroll
      for (int kw = 0; kw < kStemK; ++kw) {
#pragma unroll
        for (int ci = 0; ci < kStemCin; ++ci) {
          const float4* xp =
              reinterpret_cast<const float4*>(xk + (kw >> 1) * kStemCopyF + ((kw & 1) * kStemCin + ci) * kStemPlaneF);
          const float4 x0 = xp[0], x1 = xp[1], x2 = xp[2], x3 = xp[3];
          const float* wt = wk + (kw * kStemCin + ci) * kStemCout;
          // the weight pairs (channels 2 k, 2 k + 1) as they lie in shared memory
          const ulonglong2 wa = *reinterpret_cast<const ulonglong2*>(wt);
          const ulonglong2 wb = *reinterpret_cast<const ulonglong2*>(wt + 64);
          const float xv[16] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w,
                                x2.x, x2.y, x2.z, x2.w, x3.x, x3.y, x3.z, x3.w};
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const unsigned long long xx = f32x2_pair(xv[j], xv[j]);
            ffma2(a2[j][0], xx, wa.x);
            ffma2(a2[j][1], xx, wa.y);
            ffma2(a2[j][2], xx, wb.x);
            ffma2(a2[j][3], xx, wb.y);
          }
        }
      }
    }
    float acc[16][8];
#pragma unroll
    for (int j = 0; j < 16; ++j)
#pragma unroll
      for (int k = 0; k < 4; ++k) f32x2_unpair(a2[j][k], acc[j][2 * k], acc[j][2 * k + 1]);
    const int tw = static_cast<int>(t % tiles_w);
    const int64_t rt = t / tiles_w;
    const int th = static_cast<int>(rt % tiles_h);
    const int64_t n = rt / tiles_h;
    const int oh = th * kStemTH + r;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const bool in_out = oh < Ho && tw * kStemTW + j < Wo;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        if (relu) acc[j][c] = fmaxf(acc[j][c], 0.0f);
        // a pixel outside the output takes no part in a pooling window (with
        // ReLU every value is >= 0, and 0 leaves a window's maximum unchanged)
        if (pool != nullptr && !in_out) acc[j][c] = 0.0f;
      }
      if (y != nullptr && in_out) {
        float4* yp = reinterpret_cast<float4*>(y + ((n * Ho + oh) * Wo + tw * kStemTW + j) * kStemCout + cg * 8);
        yp[0] = make_float4(acc[j][0], acc[j][1], acc[j][2], acc[j][3]);
        yp[1] = make_float4(acc[j][4], acc[j][5], acc[j][6], acc[j][7]);
      }
    }
    // Every warp is done with this window and, from the previous tile, with the
    // pooling stage, and every thread's copies of the next window have landed.
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    if (more) scatter();
    if (pool != nullptr) {
      float h[9][8];
      stem_pool_rows(acc, h);
      if (r & 1) {
#pragma unroll
        for (int pc = 0; pc < 9; ++pc) {
          float4* d = reinterpret_cast<float4*>(pstage + (r >> 1) * kStemPoolRowF + pc * kStemCout + cg * 8);
          d[0] = make_float4(h[pc][0], h[pc][1], h[pc][2], h[pc][3]);
          d[1] = make_float4(h[pc][4], h[pc][5], h[pc][6], h[pc][7]);
        }
      }
      __syncthreads();  // the odd rows staged and the next window's copies written
      if ((r & 1) == 0 || r == kStemTH - 1) {
        const int pr = (r + 1) >> 1;  // even rows: r / 2; the last row: pooled row 8
        const int64_t pi = static_cast<int64_t>(th) * (kStemTH / 2) + pr;
        if (pi < Hp) {
#pragma unroll
          for (int pc = 0; pc < 9; ++pc) {
            const int pj = tw * (kStemTW / 2) + pc;
            if (pj >= Wp) continue;
            float v[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) v[c] = h[pc][c];
            if ((r & 1) == 0) {
#pragma unroll
              for (int rr = -1; rr <= 1; rr += 2) {
                const int ro = r + rr;
                if (ro < 0) continue;
                const float4* sp = reinterpret_cast<const float4*>(pstage + (ro >> 1) * kStemPoolRowF + pc * kStemCout + cg * 8);
                const float4 pa = sp[0], pb = sp[1];
                v[0] = fmaxf(v[0], pa.x); v[1] = fmaxf(v[1], pa.y); v[2] = fmaxf(v[2], pa.z); v[3] = fmaxf(v[3], pa.w);
                v[4] = fmaxf(v[4], pb.x); v[5] = fmaxf(v[5], pb.y); v[6] = fmaxf(v[6], pb.z); v[7] = fmaxf(v[7], pb.w);
              }
            }
            float* dst = pool + ((n * Hp + pi) * Wp + pj) * kStemCout + cg * 8;
            const bool whole = pr >= 1 && pr <= kStemTH / 2 - 1 && pc >= 1 && pc <= 7;
            if (whole) {
              reinterpret_cast<float4*>(dst)[0] = make_float4(v[0], v[1], v[2], v[3]);
              reinterpret_cast<float4*>(dst)[1] = make_float4(v[4], v[5], v[6], v[7]);
            } else {
#pragma unroll
              for (int c = 0; c < 8; ++c) atomicMax(reinterpret_cast<unsigned int*>(dst) + c, __float_as_uint(v[c]));
            }
          }
        }
      }
    } else {
      __syncthreads();  // the next window's copies written
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

// The same sums for four consecutive channels per thread (C % 4 == 0, 16-byte
// aligned rows): each channel's terms are still added in (h, w) order from 0; the
// loop is unrolled so that the loads of several positions are in flight at once.
__global__ void __launch_bounds__(128) pq_avgpool_f32_vec4_kernel(const float4* __restrict__ x,
                                                                 float4* __restrict__ y, int64_t N, int HW, int C4) {
  const int64_t total = N * C4;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t n = i / C4;
    const int64_t c4 = i - n * C4;
    const float4* p = x + n * HW * C4 + c4;
    float4 a = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll 7
    for (int j = 0; j < HW; ++j) {
      const float4 v = __ldg(p + static_cast<int64_t>(j) * C4);
      a.x = __fadd_rn(a.x, v.x);
      a.y = __fadd_rn(a.y, v.y);
      a.z = __fadd_rn(a.z, v.z);
      a.w = __fadd_rn(a.w, v.w);
    }
    const float hw = static_cast<float>(HW);
    y[i] = make_float4(__fdiv_rn(a.x, hw), __fdiv_rn(a.y, hw), __fdiv_rn(a.z, hw), __fdiv_rn(a.w, hw));
  }
}

// y[n, o] = fma over i in order of x[n, i] w[o, i] (no bias).  A block computes
// 32 outputs x 16 images: lane = output, warp w = images 2w and 2w + 1, so a
// thread keeps two running sums, each over i = 0, 1, 2, ... in order.  128-wide
// chunks of x (as image pairs) and w (rows at pitch 129, so the lanes' reads of
// one column fall in distinct banks) are staged in shared memory; the next
// chunk's global loads are issued into registers before the current chunk's
// FMAs and stored after them.
constexpr int kFcO = 32, kFcN = 16, kFcK = 128, kFcThreads = 256;
constexpr int kFcXPer = kFcN * kFcK / kFcThreads;  // 8 x values a thread loads per chunk
constexpr int kFcWPer = kFcO * kFcK / kFcThreads;  // 16 w values a thread loads per chunk

__global__ void __launch_bounds__(kFcThreads) pq_linear_f32_kernel(const float* __restrict__ x,
                                                                  const float* __restrict__ w,
                                                                  float* __restrict__ y, int64_t N, int Cin,
                                                                  int Cout) {
  __shared__ float2 xs[kFcN / 2][kFcK];
  __shared__ float wsh[kFcO][kFcK + 1];
  const int t = threadIdx.x, lane = t & 31, wn = t >> 5;
  const int o = blockIdx.x * kFcO + lane;
  const int64_t n0 = static_cast<int64_t>(blockIdx.y) * kFcN;
  float xr[kFcXPer], wr[kFcWPer];
  // element e = t + kFcThreads * r of a chunk: x row e / kFcK (an image), w row
  // e / kFcK (an output), column e % kFcK; consecutive threads read consecutive
  // columns of one row.
  auto load = [&](int c0) {
#pragma unroll
    for (int r = 0; r < kFcXPer; ++r) {
      const int e = t + kFcThreads * r, img = e / kFcK, c = e % kFcK;
      xr[r] = (c0 + c < Cin && n0 + img < N) ? __ldg(x + (n0 + img) * Cin + c0 + c) : 0.0f;
    }
#pragma unroll
    for (int r = 0; r < kFcWPer; ++r) {
      const int e = t + kFcThreads * r, row = e / kFcK, c = e % kFcK;
      const int oo = blockIdx.x * kFcO + row;
      wr[r] = (c0 + c < Cin && oo < Cout) ? __ldg(w + static_cast<int64_t>(oo) * Cin + c0 + c) : 0.0f;
    }
  };
  auto store = [&]() {
#pragma unroll
    for (int r = 0; r < kFcXPer; ++r) {
      const int e = t + kFcThreads * r, img = e / kFcK, c = e % kFcK;
      float* p = reinterpret_cast<float*>(&xs[img >> 1][c]);
      p[img & 1] = xr[r];
    }
#pragma unroll
    for (int r = 0; r < kFcWPer; ++r) {
      const int e = t + kFcThreads * r, row = e / kFcK, c = e % kFcK;
      wsh[row][c] = wr[r];
    }
  };
  float acc0 = 0.0f, acc1 = 0.0f;
  load(0);
  for (int c0 = 0; c0 < Cin; c0 += kFcK) {
    __syncthreads();  // the previous chunk's reads are done
    store();
    __syncthreads();
    if (c0 + kFcK < Cin) load(c0 + kFcK);
    const int kc = min(kFcK, Cin - c0);
    if (kc == kFcK) {
#pragma unroll 16
      for (int c = 0; c < kFcK; ++c) {
        const float2 xv = xs[wn][c];
        const float wv = wsh[lane][c];
        acc0 = __fmaf_rn(xv.x, wv, acc0);
        acc1 = __fmaf_rn(xv.y, wv, acc1);
      }
    } else {
      for (int c = 0; c < kc; ++c) {
        const float2 xv = xs[wn][c];
        const float wv = wsh[lane][c];
        acc0 = __fmaf_rn(xv.x, wv, acc0);
        acc1 = __fmaf_rn(xv.y, wv, acc1);
      }
    }
  }
  const int64_t na = n0 + 2 * wn;
  if (o < Cout) {
    if (na < N) y[na * Cout + o] = acc0;
    if (na + 1 < N) y[(na + 1) * Cout + o] = acc1;
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
// The stem kernel's dynamic shared memory above the default limit, once per
// process (the network runs on one device).
bool stem_smem_attribute() {
  static bool done = false;
  if (!done) {
    if (cudaFuncSetAttribute(pq_stem7x7s2_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kStemSmem)) != cudaSuccess)
      return false;
    done = true;
  }
  return true;
}

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
  if (k == pq::kStemK && stride == pq::kStemS && pad == pq::kStemP && Cin == pq::kStemCin && Cout == pq::kStemCout &&
      pq::aligned16(y_dev)) {
    if (!pq::stem_smem_attribute()) return PQ_ECUDA;
    const int64_t tiles = N * ((Ho + pq::kStemTH - 1) / pq::kStemTH) * ((Wo + pq::kStemTW - 1) / pq::kStemTW);
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const unsigned grid = static_cast<unsigned>(tiles < static_cast<int64_t>(sms) ? tiles : sms);
    pq::pq_stem7x7s2_kernel<<<grid, pq::kStemThreads, pq::kStemSmem, s>>>(
        x_dev, w_dev, y_dev, nullptr, N, H, W, static_cast<int>(Ho), static_cast<int>(Wo), 0, 0, relu);
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

pq_status palquant_stem_pool_f32(const float* x_dev, const float* w_dev, float* stem_dev, float* pool_dev, int64_t N,
                                 int32_t H, int32_t W, int32_t Cout, pq_stream_t stream) {
  if (N < 0 || H <= 0 || W <= 0 || Cout <= 0 || !x_dev || !w_dev || !pool_dev) return PQ_EINVAL;
  if (!pq::aligned16(pool_dev) || (stem_dev && !pq::aligned16(stem_dev))) return PQ_EINVAL;
  if (Cout != pq::kStemCout) return PQ_EUNSUPPORTED;
  const int64_t Ho = pq::out_dim(H, pq::kStemK, pq::kStemS, pq::kStemP), Wo = pq::out_dim(W, pq::kStemK, pq::kStemS, pq::kStemP);
  if (Ho <= 0 || Wo <= 0) return PQ_EINVAL;
  const int64_t Hp = pq::out_dim(Ho, 3, 2, 1), Wp = pq::out_dim(Wo, 3, 2, 1);
  if (N == 0) return PQ_OK;
  auto s = static_cast<cudaStream_t>(stream);
  if (!pq::stem_smem_attribute()) return PQ_ECUDA;
  // border windows are combined by atomic maxima over non-negative values: start from 0
  if (cudaMemsetAsync(pool_dev, 0, static_cast<size_t>(N * Hp * Wp * Cout) * sizeof(float), s) != cudaSuccess)
    return PQ_ECUDA;
  const int64_t tiles = N * ((Ho + pq::kStemTH - 1) / pq::kStemTH) * ((Wo + pq::kStemTW - 1) / pq::kStemTW);
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const unsigned grid = static_cast<unsigned>(tiles < static_cast<int64_t>(sms) ? tiles : sms);
  pq::pq_stem7x7s2_kernel<<<grid, pq::kStemThreads, pq::kStemSmem, s>>>(
      x_dev, w_dev, stem_dev, pool_dev, N, H, W, static_cast<int>(Ho), static_cast<int>(Wo), static_cast<int>(Hp),
      static_cast<int>(Wp), 1);
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
  if (C % 4 == 0 && pq::aligned16(x_dev) && pq::aligned16(y_dev)) {
    const int64_t work = N * (C / 4);
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (work + 127) / 128, cap = static_cast<int64_t>(sms) * 16;
    pq::pq_avgpool_f32_vec4_kernel<<<static_cast<unsigned>(want < cap ? want : cap), 128, 0,
                                     static_cast<cudaStream_t>(stream)>>>(reinterpret_cast<const float4*>(x_dev),
                                                                          reinterpret_cast<float4*>(y_dev), N, H * W,
                                                                          C / 4);
  } else {
    pq::pq_avgpool_f32_kernel<<<pq::grid_for(N * C, 8), 256, 0, static_cast<cudaStream_t>(stream)>>>(x_dev, y_dev, N,
                                                                                                      H * W, C);
  }
  return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
}

pq_status palquant_linear_f32(const float* x_dev, const float* w_dev, float* y_dev, int64_t N, int32_t Cin,
                              int32_t Cout, pq_stream_t stream) {
  if (N < 0 || Cin <= 0 || Cout <= 0 || !x_dev || !w_dev || !y_dev) return PQ_EINVAL;
  if (N == 0) return PQ_OK;
  const int64_t gy = (N + pq::kFcN - 1) / pq::kFcN;
  if (gy > 65535) return PQ_EUNSUPPORTED;
  const dim3 grid(static_cast<unsigned>((Cout + pq::kFcO - 1) / pq::kFcO), static_cast<unsigned>(gy));
  pq::pq_linear_f32_kernel<<<grid, pq::kFcThreads, 0, static_cast<cudaStream_t>(stream)>>>(x_dev, w_dev, y_dev,
                                                                                               N, Cin, Cout);
  return cudaGetLastError() == cudaSuccess ? PQ_OK : PQ_ECUDA;
}

}  // extern "C"
