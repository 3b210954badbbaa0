// Bit-level decomposition of an M-bit layer into B-bit slices (Sec. 3.3, Eq. 4):
// the activation codes x = sum_i x_i 2^(iB) are split into their B-bit slices,
// laid out as the input of one convolution: channel block i carries x_i, each
// slice stored once.  The convolution gives every input code Gw weight slices
// per tap (pq_layer_desc.wslices), 2^((i+j)B) w_j for slice j, packed on the
// host, so the Ga Gw shifted B-bit products of Eq. 4 accumulate in one pass of
// the tensor-core kernel while the activation slices are read once each.
#include <cuda_runtime.h>

#include <cstdint>

#include "pq_internal.h"

namespace pq {

// One thread per 16-byte unit (16 codes of one position and 16-channel chunk):
// slice i of every byte is (v >> iB) & (2^B - 1), computed on 32-bit words (a
// bit shifted in from the next byte lands above the mask as long as (i+1) B <= 8).
// Channel-blocked layout: input [N][C/16][HW][16], output [N][Ga C/16][HW][16]
// with output chunk i C/16 + cb = slice i of input chunk cb.  NHWC layout:
// input [P][C], output [P][Ga C], channel i C + c.
__global__ void __launch_bounds__(256) pq_bitsplit_act_kernel(const uint4* __restrict__ q, uint4* __restrict__ xs,
                                                             int64_t N, int64_t HW, int C16, int Ga, int B, int c16) {
  const int64_t units = N * HW * C16;
  const uint32_t mask = ((1u << B) - 1u) * 0x01010101u;
  for (int64_t u = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; u < units;
       u += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    // c16: u = (n * C16 + cb) * HW + hw;  nhwc: u = p * C16 + cb
    int64_t n_or_p, hw = 0;
    int cb;
    if (c16) {
      hw = u % HW;
      const int64_t r = u / HW;
      cb = static_cast<int>(r % C16);
      n_or_p = r / C16;
    } else {
      cb = static_cast<int>(u % C16);
      n_or_p = u / C16;
    }
    const uint4 v = q[u];
    const int64_t oc16 = static_cast<int64_t>(Ga) * C16;  // output chunks per image / pixel
    for (int i = 0; i < Ga; ++i) {
      const int s = i * B;
      const uint4 o = make_uint4((v.x >> s) & mask, (v.y >> s) & mask, (v.z >> s) & mask, (v.w >> s) & mask);
      const int64_t ob = static_cast<int64_t>(i) * C16 + cb;  // output chunk
      xs[c16 ? (n_or_p * oc16 + ob) * HW + hw : n_or_p * oc16 + ob] = o;
    }
  }
}

int launch_bitsplit_act(const uint8_t* q, uint8_t* xs, int64_t N, int64_t HW, int C, int Ga, int B, int c16,
                        cudaStream_t stream) {
  const int C16 = C / 16;
  const int64_t units = N * HW * C16;
  if (units == 0) return 0;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (units + 255) / 256, cap = static_cast<int64_t>(sms) * 8;
  pq_bitsplit_act_kernel<<<static_cast<unsigned>(want < cap ? want : cap), 256, 0, stream>>>(
      reinterpret_cast<const uint4*>(q), reinterpret_cast<uint4*>(xs), N, HW, C16, Ga, B, c16);
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // namespace pq
