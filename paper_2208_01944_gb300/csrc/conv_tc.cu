// PalQuant B-bit group convolution with the fused epilogue, on the sm_103a
// 5th-generation tensor cores.
//
// What it computes (Sec. 3.1 Eq. 1 lowered per group, Sec. 4.1 "B-bit group
// convolution", Sec. 3.2 de-quantisation with the output scale alpha, Sec. 4.2
// Eq. 6-8 output permutation, Eq. 2 requantisation):
//   acc[pix, g, co] = sum_{tap, ci} q[in_pix(pix, tap), g*Cin_g + ci] * w[g, co, tap, ci]
//   y = (float)acc * m_out[g] (+ shortcut) (ReLU);  q' = clamp(rint(t * m_req[g]), 0, Qp)
// all written at the destination channel of (g, co).
//
// How (one persistent CTA per SM, warp-specialised):
//  * warp 0 (one lane) loads, per tile, the activation codes a tile needs with
//    TMA straight into the tensor core's no-swizzle K-major operand layout: for
//    each 16-byte chunk of input channels a plane of consecutive positions, one
//    position per 16-byte row.  A "position" is a pixel of the zero-padded input
//    tile (rows mode) or a pixel of the flattened batch (flat mode, 1x1 layers).
//    Out-of-range pixels are zero-filled by TMA, which is exactly the zero
//    padding (code 0).  Stride-2 layers load the four stride phases of the input
//    through strided tensor views, so every tap is again a contiguous run of
//    positions.
//  * The int8 codes are NOT converted: a byte v <= 15 is the FP8 E4M3 encoding of
//    v * 2^-9 (subnormal and first binade are linear), so the tensor core reads
//    the codes in place and every product and sum is exact in the fp32
//    accumulator; the epilogue multiplies by 2^9 (exact).
//  * Weights are packed on the host as E4M3 of the signed integer codes in the
//    same layout, and either stay resident in shared memory for the CTA's whole
//    (group, output-block) unit or stream through a ring of (K block, tap) slices.
//  * warp 1 (one lane) issues tcgen05.mma kind::f8f6f4 (M = 128, N = the output
//    block): for every tap the A operand is the same planes with the start
//    address moved by the tap's position offset (16 bytes per position), so a
//    3x3 convolution needs no im2col copy.  Accumulators live in tensor memory,
//    double-buffered so the epilogue of tile i overlaps the MMAs of tile i+1.
//  * warps 2-5 read the accumulators (tcgen05.ld), apply the rescale, shortcut,
//    ReLU, output permutation and requantisation in registers, stage rows in
//    shared memory and write them with coalesced 16-byte stores.
//  * every wait is bounded (failure detection): a wait that runs out records
//    PQ_ERR_TIMEOUT in the device error word, raises a CTA-wide abort flag, and
//    every role drains what it has in flight and returns.
#include <cuda_runtime.h>

#include "pq_device.cuh"
#include "pq_internal.h"

namespace pq {

namespace {

struct Ring {
  uint32_t stage = 0, phase = 0, n = 1;
  __device__ __forceinline__ void advance() {
    if (++stage == n) {
      stage = 0;
      phase ^= 1u;
    }
  }
};

struct Item {
  int64_t unit, tile;
  int g, nb;
  int n, oh0;   // rows mode
  int64_t p0;   // flat mode
};

__device__ __forceinline__ Item decode_item(const ConvParams& p, int64_t it) {
  Item r;
  r.unit = it / p.tiles;
  r.tile = it - r.unit * p.tiles;
  r.g = static_cast<int>(r.unit / p.NB);
  r.nb = static_cast<int>(r.unit - static_cast<int64_t>(r.g) * p.NB);
  if (p.mode == kModeFlat) {
    r.p0 = r.tile * p.flat_box;
    r.n = 0;
    r.oh0 = 0;
  } else {
    r.n = static_cast<int>(r.tile / p.tiles_per_img);
    r.oh0 = static_cast<int>(r.tile - static_cast<int64_t>(r.n) * p.tiles_per_img) * p.Ht;
    r.p0 = 0;
  }
  return r;
}

// Shared-memory barrier block layout (64-bit words):
//   [0, A)           a_full       [A, 2A)        a_empty
//   [2A, 2A+B)       b_full       [2A+B, 2A+2B)  b_empty
//   +0,+1 acc_full, +2,+3 acc_empty, +4 drain, then int abort flag, u32 TMEM base.
struct Bars {
  uint32_t base;
  int A, B;
  __device__ uint32_t a_full(int s) const { return base + 8u * s; }
  __device__ uint32_t a_empty(int s) const { return base + 8u * (A + s); }
  __device__ uint32_t b_full(int s) const { return base + 8u * (2 * A + s); }
  __device__ uint32_t b_empty(int s) const { return base + 8u * (2 * A + B + s); }
  __device__ uint32_t acc_full(int s) const { return base + 8u * (2 * A + 2 * B + s); }
  __device__ uint32_t acc_empty(int s) const { return base + 8u * (2 * A + 2 * B + 2 + s); }
  __device__ uint32_t drain() const { return base + 8u * (2 * A + 2 * B + 4); }
  __device__ uint32_t words() const { return 2 * A + 2 * B + 5; }
};

// --------------------------------------------------------------------------
// Copy role (warp 0, lane 0).
// --------------------------------------------------------------------------
__device__ void producer_role(const ConvParams& p, const TensorMaps& tm, const Bars& bars, uint32_t a_base,
                              uint32_t b_base, int64_t it0, int64_t it1, const WaitCtx& ctx) {
  Ring ra{0, 0, static_cast<uint32_t>(p.a_stages)};
  Ring rb{0, 0, static_cast<uint32_t>(p.b_resident ? 1 : p.b_stages)};
  int64_t a_issued = 0, b_issued = 0;
  int64_t cur_unit = -1;
  bool ok = true;
  for (int64_t it = it0; it < it1 && ok; ++it) {
    const Item item = decode_item(p, it);
    if (p.b_resident && item.unit != cur_unit) {
      if (!mbar_wait(bars.b_empty(rb.stage), rb.phase ^ 1u, ctx)) { ok = false; break; }
      const uint32_t bar = bars.b_full(rb.stage);
      mbar_arrive_expect_tx(bar, p.b_unit_bytes);
      const uint8_t* src = p.w_packed + static_cast<size_t>(item.unit) * p.b_unit_bytes;
      // Copy in pieces of at most 64 KB.
      for (uint32_t off = 0; off < p.b_unit_bytes; off += 65536u) {
        const uint32_t len = min(65536u, p.b_unit_bytes - off);
        bulk_load(b_base + off, src + off, len, bar);
      }
      rb.advance();
      ++b_issued;
      cur_unit = item.unit;
    }
    for (int kb = 0; kb < p.n_kb; ++kb) {
      if (!mbar_wait(bars.a_empty(ra.stage), ra.phase ^ 1u, ctx)) { ok = false; break; }
      const uint32_t full = bars.a_full(ra.stage);
      mbar_arrive_expect_tx(full, p.a_tx_bytes);
      const uint32_t dst = a_base + ra.stage * p.a_stage_bytes;
      const int chi = (item.g * p.Cin_g + kb * p.KC) >> 4;
      if (p.mode == kModeFlat) {
        tma_load_3d(dst, &tm.a[0], 0, static_cast<int>(item.p0), chi, full);
      } else {
        for (int ph = 0; ph < p.nph; ++ph)
          tma_load_5d(dst + ph * p.a_phase_bytes, &tm.a[ph], 0, p.w_coord, item.oh0 + p.h_off, chi, item.n, full);
      }
      ra.advance();
      ++a_issued;
      if (!p.b_resident) {
        for (int t = 0; t < p.taps; ++t) {
          if (!mbar_wait(bars.b_empty(rb.stage), rb.phase ^ 1u, ctx)) { ok = false; break; }
          const uint32_t bar = bars.b_full(rb.stage);
          mbar_arrive_expect_tx(bar, p.b_slice_bytes);
          const size_t slice = (static_cast<size_t>(item.unit) * p.n_kb + kb) * p.taps + t;
          bulk_load(b_base + rb.stage * p.b_slice_bytes, p.w_packed + slice * p.b_slice_bytes, p.b_slice_bytes, bar);
          rb.advance();
          ++b_issued;
        }
        if (!ok) break;
      }
    }
  }
  // Drain: the last min(stages, issued) copies of each ring may still be in flight.
  const int64_t na = p.a_stages, nbs = p.b_resident ? 1 : p.b_stages;
  for (int64_t k = (a_issued > na ? a_issued - na : 0); k < a_issued; ++k)
    mbar_wait_drain(bars.a_full(static_cast<int>(k % na)), static_cast<uint32_t>((k / na) & 1), ctx.limit_ns, ctx.err);
  for (int64_t k = (b_issued > nbs ? b_issued - nbs : 0); k < b_issued; ++k)
    mbar_wait_drain(bars.b_full(static_cast<int>(k % nbs)), static_cast<uint32_t>((k / nbs) & 1), ctx.limit_ns, ctx.err);
}

// --------------------------------------------------------------------------
// Tensor-core issue role (warp 1, lane 0).
// --------------------------------------------------------------------------
__device__ void mma_role(const ConvParams& p, const Bars& bars, uint32_t a_base, uint32_t b_base, uint32_t tmem_base,
                         int64_t it0, int64_t it1, const WaitCtx& ctx) {
  Ring ra{0, 0, static_cast<uint32_t>(p.a_stages)};
  Ring rb{0, 0, static_cast<uint32_t>(p.b_resident ? 1 : p.b_stages)};
  Ring racc{0, 0, static_cast<uint32_t>(p.acc_stages)};
  const uint32_t idesc = idesc_e4m3_f32(128, p.Nblk);
  const int ksteps = p.nch >> 1;
  int64_t cur_unit = -1;
  bool ok = true;
  for (int64_t it = it0; it < it1 && ok; ++it) {
    const int64_t unit = it / p.tiles;
    if (p.b_resident && unit != cur_unit) {
      if (!mbar_wait(bars.b_full(rb.stage), rb.phase, ctx)) { ok = false; break; }
      cur_unit = unit;
    }
    if (!mbar_wait(bars.acc_empty(racc.stage), racc.phase ^ 1u, ctx)) { ok = false; break; }
    tc_fence_after();
    const uint32_t d0 = tmem_base + racc.stage * p.MT * p.Npow2;
    for (int kb = 0; kb < p.n_kb && ok; ++kb) {
      if (!mbar_wait(bars.a_full(ra.stage), ra.phase, ctx)) { ok = false; break; }
      tc_fence_after();
      const uint32_t a_stage = a_base + ra.stage * p.a_stage_bytes;
      for (int t = 0; t < p.taps; ++t) {
        uint32_t bslice;
        if (p.b_resident) {
          bslice = b_base + (kb * p.taps + t) * p.b_slice_bytes;
        } else {
          if (!mbar_wait(bars.b_full(rb.stage), rb.phase, ctx)) { ok = false; break; }
          tc_fence_after();
          bslice = b_base + rb.stage * p.b_slice_bytes;
        }
        const uint32_t a_tap = a_stage + p.tap_phase[t] * p.a_phase_bytes + static_cast<uint32_t>(p.tap_off[t]) * 16u;
        for (int ks = 0; ks < ksteps; ++ks) {
          const uint64_t bdesc = smem_desc(bslice + 2u * ks * p.lbo_b, p.lbo_b, 128u);
          for (int mt = 0; mt < p.MT; ++mt) {
            const uint64_t adesc = smem_desc(a_tap + mt * 2048u + 2u * ks * p.lbo_a, p.lbo_a, 128u);
            tc_mma_e4m3(d0 + mt * p.Npow2, adesc, bdesc, idesc, (kb | t | ks) != 0 ? 1u : 0u);
          }
        }
        if (!p.b_resident) {
          tc_commit(bars.b_empty(rb.stage));
          rb.advance();
        }
      }
      if (!ok) break;
      tc_commit(bars.a_empty(ra.stage));
      ra.advance();
    }
    if (!ok) break;
    tc_commit(bars.acc_full(racc.stage));
    racc.advance();
    if (p.b_resident) {
      const int64_t next_unit = (it + 1 < it1) ? (it + 1) / p.tiles : -1;
      if (next_unit != unit) {
        tc_commit(bars.b_empty(rb.stage));
        rb.advance();
      }
    }
  }
  // Drain: wait until every MMA this thread issued has completed.
  tc_commit(bars.drain());
  mbar_wait_drain(bars.drain(), 0, ctx.limit_ns, ctx.err);
}

// --------------------------------------------------------------------------
// Epilogue role (warps 2-5).
// --------------------------------------------------------------------------
// 32 rows of `row_bytes` (multiple of 16) staged at `pitch`: lane r's row goes to
// global byte offset row_off (negative: row not stored).
__device__ __forceinline__ void warp_store_rows(const uint8_t* stg, uint32_t pitch, int row_bytes, uint8_t* gdst,
                                                long long row_off, int lane) {
  __syncwarp();
  const int cpr = row_bytes >> 4;
  const int total = 32 * cpr;
  for (int idx = lane; idx < total; idx += 32) {
    const int r = idx / cpr;
    const int c = idx - r * cpr;
    const long long off = __shfl_sync(0xffffffffu, row_off, r);
    if (off >= 0) *reinterpret_cast<uint4*>(gdst + off + c * 16) = *reinterpret_cast<const uint4*>(stg + r * pitch + c * 16);
  }
  __syncwarp();
}

__device__ void epilogue_role(const ConvParams& p, const Bars& bars, uint32_t tmem_base, uint8_t* stage_base,
                              int64_t it0, int64_t it1, const WaitCtx& ctx) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quarter = warp & 3;  // TMEM lanes this warp may access
  uint8_t* stg_q = stage_base + (warp - 2) * p.stage_warp_bytes;
  uint8_t* stg_f = stg_q + 32 * p.stage_q_pitch;
  Ring racc{0, 0, static_cast<uint32_t>(p.acc_stages)};
  const int nchunks = p.Nblk >> 4;
  const float qmax = static_cast<float>(p.qmax_out);
  for (int64_t it = it0; it < it1; ++it) {
    const Item item = decode_item(p, it);
    if (!mbar_wait(bars.acc_full(racc.stage), racc.phase, ctx)) break;
    tc_fence_after();
    const int g = item.g;
    const float m_out = p.m_out[g];
    const float m_req = p.m_req[g];
    const int src_c0 = g * p.Cout_g + item.nb * p.Nblk;          // source channel of column 0
    const int dst_c0 = p.dst_group[g] * p.Cout_g + item.nb * p.Nblk;  // destination channel of column 0
    for (int mt = 0; mt < p.MT; ++mt) {
      const int m = mt * 128 + quarter * 32 + lane;
      long long pix;
      bool valid;
      if (p.mode == kModeFlat) {
        pix = item.p0 + m;
        valid = pix < p.P_out;
      } else {
        const int r = m / p.Wh;
        const int c = m - r * p.Wh;
        const int oh = item.oh0 + r;
        valid = (r < p.Ht) && (c < p.Wo) && (oh < p.Ho);
        pix = (static_cast<long long>(item.n) * p.Ho + oh) * p.Wo + c;
      }
      const long long row_elem = valid ? pix * p.C_out_total : -1;
      const uint32_t tcol = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + racc.stage * p.MT * p.Npow2 +
                            mt * p.Npow2;
      for (int ch = 0; ch < nchunks; ++ch) {
        uint32_t v[16];
        tmem_ld16(tcol + ch * 16, v);
        tmem_wait_ld();
        float accf[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) accf[j] = __uint_as_float(v[j]) * 512.0f;  // exact: codes were read as v * 2^-9
        float sc[16];
        if (p.shortcut != nullptr) {
          if (valid) {
            const float4* s4 = reinterpret_cast<const float4*>(p.shortcut + pix * p.C_out_total + src_c0 + ch * 16);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const float4 t = s4[j];
              sc[4 * j] = t.x; sc[4 * j + 1] = t.y; sc[4 * j + 2] = t.z; sc[4 * j + 3] = t.w;
            }
          } else {
#pragma unroll
            for (int j = 0; j < 16; ++j) sc[j] = 0.0f;
          }
        }
        float y[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          float t = __fmul_rn(accf[j], m_out);
          if (p.shortcut != nullptr) t = __fadd_rn(t, sc[j]);
          if (p.relu) t = fmaxf(t, 0.0f);
          y[j] = t;
        }
        if (p.channel_shuffle) {
          // Per-channel scatter (destination channel co * G + g); rarely used, unstaged.
          if (valid) {
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int co = item.nb * p.Nblk + ch * 16 + j;
              const long long o = pix * p.C_out_total + static_cast<long long>(co) * p.G + g;
              if (p.acc_out) p.acc_out[o] = __float2int_rn(accf[j]);
              if (p.y_out) p.y_out[o] = y[j];
              if (p.q_out) {
                float r = rintf(__fmul_rn(p.shortcut != nullptr ? y[j] : accf[j], m_req));
                r = fminf(fmaxf(r, 0.0f), qmax);
                p.q_out[o] = static_cast<uint8_t>(static_cast<int>(r));
              }
            }
          }
          continue;
        }
        if (p.acc_out) {
          uint32_t* row = reinterpret_cast<uint32_t*>(stg_f + lane * p.stage_f_pitch);
#pragma unroll
          for (int j = 0; j < 16; j += 4)
            *reinterpret_cast<uint4*>(row + j) =
                make_uint4(__float2int_rn(accf[j]), __float2int_rn(accf[j + 1]), __float2int_rn(accf[j + 2]),
                           __float2int_rn(accf[j + 3]));
          warp_store_rows(stg_f, p.stage_f_pitch, 64, reinterpret_cast<uint8_t*>(p.acc_out),
                          row_elem < 0 ? -1 : (row_elem + dst_c0 + ch * 16) * 4, lane);
        }
        if (p.y_out) {
          float* row = reinterpret_cast<float*>(stg_f + lane * p.stage_f_pitch);
#pragma unroll
          for (int j = 0; j < 16; j += 4) *reinterpret_cast<float4*>(row + j) = make_float4(y[j], y[j + 1], y[j + 2], y[j + 3]);
          warp_store_rows(stg_f, p.stage_f_pitch, 64, reinterpret_cast<uint8_t*>(p.y_out),
                          row_elem < 0 ? -1 : (row_elem + dst_c0 + ch * 16) * 4, lane);
        }
        if (p.q_out) {
          uint32_t w[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            uint32_t packed = 0;
#pragma unroll
            for (int b = 0; b < 4; ++b) {
              const float src = p.shortcut != nullptr ? y[4 * j + b] : accf[4 * j + b];
              float r = rintf(__fmul_rn(src, m_req));
              r = fminf(fmaxf(r, 0.0f), qmax);
              packed |= static_cast<uint32_t>(static_cast<int>(r)) << (8 * b);
            }
            w[j] = packed;
          }
          *reinterpret_cast<uint4*>(stg_q + lane * p.stage_q_pitch + (ch & 3) * 16) = make_uint4(w[0], w[1], w[2], w[3]);
          // Codes go out in segments of up to 64 channels (4 chunks) per row.
          if ((ch & 3) == 3 || ch == nchunks - 1) {
            const int seg0 = ch & ~3;
            warp_store_rows(stg_q, p.stage_q_pitch, (ch - seg0 + 1) * 16, p.q_out,
                            row_elem < 0 ? -1 : row_elem + dst_c0 + seg0 * 16, lane);
          }
        }
      }
    }
    tc_fence_before();
    mbar_arrive(bars.acc_empty(racc.stage));
    racc.advance();
  }
}

}  // namespace

__global__ void __launch_bounds__(kConvThreads, 1)
    pq_conv_tc_kernel(const __grid_constant__ ConvParams p, const __grid_constant__ TensorMaps tm) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  Bars bars{base + p.smem_bar_off, p.a_stages, p.b_resident ? 1 : p.b_stages};
  uint8_t* bar_block = gbase + p.smem_bar_off;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bar_block + 8 * bars.words());
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_block + 8 * bars.words() + 8);

  if (threadIdx.x == 0) {
    for (int s = 0; s < bars.A; ++s) {
      mbar_init(bars.a_full(s), 1);
      mbar_init(bars.a_empty(s), 1);
    }
    for (int s = 0; s < bars.B; ++s) {
      mbar_init(bars.b_full(s), 1);
      mbar_init(bars.b_empty(s), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(bars.acc_full(s), 1);
      mbar_init(bars.acc_empty(s), kEpiWarps * 32);
    }
    mbar_init(bars.drain(), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    for (int ph = 0; ph < p.nph; ++ph) prefetch_tmap(&tm.a[ph]);
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), p.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int64_t it0 = static_cast<int64_t>(blockIdx.x) * p.items / gridDim.x;
  const int64_t it1 = static_cast<int64_t>(blockIdx.x + 1) * p.items / gridDim.x;
  const uint32_t a_base = base;
  const uint32_t b_base = base + p.smem_b_off;

  if (warp == 0) {
    if (lane == 0) producer_role(p, tm, bars, a_base, b_base, it0, it1, WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_PRODUCER});
  } else if (warp == 1) {
    if (lane == 0) mma_role(p, bars, a_base, b_base, tmem_base, it0, it1, WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_MMA});
    __syncwarp();
  } else {
    epilogue_role(p, bars, tmem_base, gbase + p.smem_stage_off, it0, it1,
                  WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_EPILOGUE});
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

int launch_conv_tc(const ConvParams& p, const TensorMaps& tm, int grid, cudaStream_t stream) {
  static int attr_set_for_device[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  const int need = static_cast<int>(p.smem_bytes) + 1024;
  if (dev < 64 && attr_set_for_device[dev] < need) {
    if (cudaFuncSetAttribute(pq_conv_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem) != cudaSuccess)
      return -1;
    attr_set_for_device[dev] = kMaxSmem;
  }
  pq_conv_tc_kernel<<<grid, kConvThreads, need, stream>>>(p, tm);
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // namespace pq
