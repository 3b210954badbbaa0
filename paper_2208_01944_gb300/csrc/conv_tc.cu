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
//  * warps 2-5 copy, per tile, the activation codes the tile needs with 16-byte
//    cp.async straight into the tensor core's no-swizzle K-major operand layout:
//    for each 16-byte chunk of input channels a plane of consecutive positions,
//    one position per 16-byte row.  A "position" is a pixel of the zero-padded
//    input tile (rows mode) or a pixel of the flattened batch (flat mode, 1x1
//    layers).  Out-of-range pixels are zero-filled, which is exactly the zero
//    padding (code 0).  Stride-2 layers get one plane set per stride phase of
//    the input, so every tap is again a contiguous run of positions.  (A TMA box
//    with a 16-byte inner extent moves one element per several cycles per SM and
//    starved the tensor core; the LSU path moves 512 bytes per warp instruction.)
//  * The int8 codes are NOT converted: a byte v <= 15 is the FP8 E4M3 encoding of
//    v * 2^-9 (subnormal and first binade are linear), so the tensor core reads
//    the codes in place and every product and sum is exact in the fp32
//    accumulator; the epilogue multiplies by 2^9 (exact).
//  * Weights are packed on the host as E4M3 of the signed integer codes in the
//    same layout; warp 0 bulk-copies them (cp.async.bulk) so they either stay
//    resident in shared memory for the CTA's whole (group, output-block) unit or
//    stream through a ring of (K block, tap) slices.
//  * warp 1 (one lane) issues tcgen05.mma kind::f8f6f4 (M = 128, N = the output
//    block): for every tap the A operand is the same planes with the start
//    address moved by the tap's position offset (16 bytes per position), so a
//    3x3 convolution needs no im2col copy.  Accumulators live in tensor memory,
//    double-buffered so the epilogue of tile i overlaps the MMAs of tile i+1.
//  * warps 6-13 (two warpgroups, each taking half of the output columns) read the
//    accumulators (tcgen05.ld), apply the rescale, shortcut,
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

// Position in the CTA's contiguous range of work items, advanced without
// divisions (64-bit divisions per item cost every role hundreds of cycles).
struct Item {
  int64_t it;   // global item index
  int unit;     // (group, output block) unit = g * NB + nb
  int tile;     // tile within the unit
  int g, nb;
  int n, rb;    // image and tile within it (rows mode: oh0 = rb * Ht; flat mode: first pixel rb * flat_box)
  __device__ __forceinline__ int oh0(int Ht) const { return rb * Ht; }
};

__device__ __forceinline__ Item item_begin(const ConvParams& p, int64_t it) {
  Item r;
  r.it = it;
  const int64_t unit = it / p.tiles;
  r.unit = static_cast<int>(unit);
  r.tile = static_cast<int>(it - unit * p.tiles);
  r.g = r.unit / p.NB;
  r.nb = r.unit - r.g * p.NB;
  r.n = r.tile / p.tiles_per_img;
  r.rb = r.tile - r.n * p.tiles_per_img;
  return r;
}

__device__ __forceinline__ void item_next(const ConvParams& p, Item& r) {
  ++r.it;
  if (++r.tile == p.tiles) {
    r.tile = 0;
    r.n = 0;
    r.rb = 0;
    if (++r.nb == p.NB) {
      r.nb = 0;
      ++r.g;
    }
    ++r.unit;
    return;
  }
  if (++r.rb == p.tiles_per_img) {
    r.rb = 0;
    ++r.n;
  }
}

// Shared-memory barrier block layout (64-bit words):
//   [0, A)           a_full       [A, 2A)        a_empty
//   [2A, 2A+B)       b_full       [2A+B, 2A+2B)  b_empty
//   +0..+3 acc_full, +4..+7 acc_empty (kMaxAccStages), +8 drain, then A pk_full and A pk_empty
//   (packed codes only), then int abort flag, u32 TMEM base.
struct Bars {
  uint32_t base;
  int A, B;
  __device__ uint32_t a_full(int s) const { return base + 8u * s; }
  __device__ uint32_t a_empty(int s) const { return base + 8u * (A + s); }
  __device__ uint32_t b_full(int s) const { return base + 8u * (2 * A + s); }
  __device__ uint32_t b_empty(int s) const { return base + 8u * (2 * A + B + s); }
  __device__ uint32_t acc_full(int s) const { return base + 8u * (2 * A + 2 * B + s); }
  __device__ uint32_t acc_empty(int s) const { return base + 8u * (2 * A + 2 * B + kMaxAccStages + s); }
  __device__ uint32_t drain() const { return base + 8u * (2 * A + 2 * B + 2 * kMaxAccStages); }
  // packed-code staging ring (one stage per operand stage)
  __device__ uint32_t pk_full(int s) const { return base + 8u * (2 * A + 2 * B + 2 * kMaxAccStages + 1 + s); }
  __device__ uint32_t pk_empty(int s) const { return base + 8u * (3 * A + 2 * B + 2 * kMaxAccStages + 1 + s); }
  __device__ uint32_t words() const { return 4 * A + 2 * B + 2 * kMaxAccStages + 1; }
};

// Wait taken by every lane of a converged warp; the lanes agree on the outcome,
// so the warp stays converged (for warp barriers and per-warp arrivals) even when
// a wait times out.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, const WaitCtx& ctx) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, ctx));
}

// --------------------------------------------------------------------------
// Copy role (warp 0, lane 0): bulk copies of the packed weights, either once
// per (group, output-block) unit (resident) or one (K block, tap) slice at a
// time through a ring; and, for channel-blocked codes at stride 1, the
// activation operand of each stage as one TMA load (every plane row is a
// contiguous run there).
// --------------------------------------------------------------------------
__device__ __forceinline__ void producer_role(const ConvParams& p, const CUtensorMap* tmA, const Bars& bars,
                                              uint32_t a_base, uint32_t b_base, uint32_t pk_base, int64_t it0,
                                              int64_t it1, const WaitCtx& ctx) {
  Ring ra{0, 0, static_cast<uint32_t>(p.a_stages)};
  Ring rb{0, 0, static_cast<uint32_t>(p.b_resident ? 1 : p.b_stages)};
  int64_t a_issued = 0, b_issued = 0;
  int64_t cur_unit = -1;
  const bool a_tma = p.a_tma != 0, flat = p.mode == kModeFlat;
  bool ok = true;
  Item item = item_begin(p, it0);
  for (int64_t it = it0; it < it1 && ok; ++it, item_next(p, item)) {
    const int64_t unit = item.unit;
    if (p.b_resident && unit != cur_unit) {
      if (!mbar_wait(bars.b_empty(rb.stage), rb.phase ^ 1u, ctx)) break;
      const uint32_t bar = bars.b_full(rb.stage);
      mbar_arrive_expect_tx(bar, p.b_unit_bytes);
      const uint8_t* src = p.w_packed + static_cast<size_t>(unit) * p.b_unit_bytes;
      for (uint32_t off = 0; off < p.b_unit_bytes; off += 65536u)
        bulk_load(b_base + off, src + off, min(65536u, p.b_unit_bytes - off), bar);
      rb.advance();
      ++b_issued;
      cur_unit = unit;
    }
    if (!a_tma && p.b_resident) continue;
    for (int kb = 0; kb < p.n_kb && ok; ++kb) {
      if (a_tma && p.a_quant) {
        // fp32 activations: a box of 32 channels (one 128-byte swizzled row per
        // position) into the staging ring; the copy warps quantise it.
        if (!mbar_wait(bars.pk_empty(ra.stage), ra.phase ^ 1u, ctx)) { ok = false; break; }
        const uint32_t full = bars.pk_full(ra.stage);
        mbar_arrive_expect_tx(full, p.a_tx_bytes);
        const uint32_t dst = pk_base + ra.stage * p.pk_stage_bytes;
        const int ch0 = p.src_group[item.g] * p.Cin_g + kb * p.KC;
        // one box per 32 channels of the K block, each on a 1024-byte swizzle atom
        for (int b = 0; b < (p.KC >> 5); ++b) {
          const uint32_t db = dst + static_cast<uint32_t>(b) * p.q_box_bytes;
          if (flat)
            tma_load_3d(db, tmA, ch0 + 32 * b, item.rb * p.flat_box, item.n, full);
          else
            tma_load_4d(db, tmA, ch0 + 32 * b, p.w_coord, item.oh0(p.Ht) + p.h_off, item.n, full);
        }
        ra.advance();
        ++a_issued;
      } else if (a_tma && p.a_split) {
        // Stride 2: the tile's whole input window (both stride phases of its rows
        // and columns) into the staging ring; the copy warps split it into the
        // phase planes.
        if (!mbar_wait(bars.pk_empty(ra.stage), ra.phase ^ 1u, ctx)) { ok = false; break; }
        const uint32_t full = bars.pk_full(ra.stage);
        mbar_arrive_expect_tx(full, p.a_tx_bytes);
        const int chi = (p.src_group[item.g] * p.Cin_g + kb * p.KC) >> p.chunk_shift;
        tma_load_4d(pk_base + ra.stage * p.pk_stage_bytes, tmA, 4 * p.w_coord, 2 * (item.oh0(p.Ht) + p.h_off), chi,
                    item.n, full);
        ra.advance();
        ++a_issued;
      } else if (a_tma && p.a_unpack) {
        // Packed codes: the box of 32-bit words into the staging ring; the copy
        // warps unpack it into the operand stage.
        if (!mbar_wait(bars.pk_empty(ra.stage), ra.phase ^ 1u, ctx)) { ok = false; break; }
        const uint32_t full = bars.pk_full(ra.stage);
        mbar_arrive_expect_tx(full, p.a_tx_bytes);
        const uint32_t dst = pk_base + ra.stage * p.pk_stage_bytes;
        const int chi = (p.src_group[item.g] * p.Cin_g + kb * p.KC) >> 4;
        if (flat)
          tma_load_3d(dst, tmA, item.rb * p.flat_box, chi, item.n, full);
        else
          tma_load_4d(dst, tmA, p.w_coord - p.pk_off, item.oh0(p.Ht) + p.h_off, chi, item.n, full);
        ra.advance();
        ++a_issued;
      } else if (a_tma) {
        if (!mbar_wait(bars.a_empty(ra.stage), ra.phase ^ 1u, ctx)) { ok = false; break; }
        const uint32_t full = bars.a_full(ra.stage);
        mbar_arrive_expect_tx(full, p.a_tx_bytes);
        const uint32_t dst = a_base + ra.stage * p.a_stage_bytes;
        const int chi = (p.src_group[item.g] * p.Cin_g + kb * p.KC) >> p.chunk_shift;
        if (flat) {
          // one box of 128 positions per accumulator, each into its own region
          for (int mt = 0; mt < p.MT; ++mt)
            tma_load_3d(dst + static_cast<uint32_t>(mt) * (p.a_mt16 << 4), tmA, 2 * (item.rb * p.flat_box + mt * 128),
                        chi, item.n, full);
        } else {
          tma_load_4d(dst, tmA, 2 * p.w_coord, item.oh0(p.Ht) + p.h_off, chi, item.n, full);
        }
        ra.advance();
        ++a_issued;
      }
      if (p.b_resident) continue;
      for (int t = 0; t < p.taps; ++t) {
        if (!mbar_wait(bars.b_empty(rb.stage), rb.phase ^ 1u, ctx)) { ok = false; break; }
        const uint32_t bar = bars.b_full(rb.stage);
        mbar_arrive_expect_tx(bar, p.b_slice_bytes);
        const size_t slice = (static_cast<size_t>(unit) * p.taps + t) * p.n_kb + kb;  // tap-major packing
        bulk_load(b_base + rb.stage * p.b_slice_bytes, p.w_packed + slice * p.b_slice_bytes, p.b_slice_bytes, bar);
        rb.advance();
        ++b_issued;
      }
    }
  }
  // Drain: the last min(stages, issued) copies of each ring may still be in flight.
  const int64_t na = p.a_stages, nbs = p.b_resident ? 1 : p.b_stages;
  for (int64_t k = (a_issued > na ? a_issued - na : 0); k < a_issued; ++k)
    mbar_wait_drain((p.a_unpack || p.a_quant || p.a_split) ? bars.pk_full(static_cast<int>(k % na)) : bars.a_full(static_cast<int>(k % na)),
                    static_cast<uint32_t>((k / na) & 1), ctx.limit_ns, ctx.err);
  for (int64_t k = (b_issued > nbs ? b_issued - nbs : 0); k < b_issued; ++k)
    mbar_wait_drain(bars.b_full(static_cast<int>(k % nbs)), static_cast<uint32_t>((k / nbs) & 1), ctx.limit_ns, ctx.err);
}

// --------------------------------------------------------------------------
// Activation copy role (warps 2-5): 16-byte cp.async copies of the codes a tile
// needs into the tensor core's no-swizzle K-major layout.  For each stride phase
// and each 16-byte chunk j of the K block's input channels there is a plane of
// Hd x Wd positions (one 16-byte row per position); a position outside the image
// is zero-filled (src-size 0), which is the zero padding.  Flat mode is one row
// of flat_box positions.  The (position, chunk) pattern of a plane row is the same
// for every row, so each thread precomputes its share once.  A thread releases a
// stage after its copies have landed (wait_group) and a proxy fence, so the
// tensor core (async proxy) sees the data; up to `depth` newer stages per thread
// stay in flight meanwhile.
// --------------------------------------------------------------------------
constexpr int kLoaders = 32 * kLoadWarps;
constexpr int kMaxLoadEntries = 8;

// Every thread's copies of the stage have landed (its wait_group); after the
// proxy fence and a warp barrier one lane arrives for the warp.
__device__ __forceinline__ void load_release(const Bars& bars, int64_t k, int stages) {
  fence_proxy_async_smem();
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bars.a_full(static_cast<int>(k % stages)));
}

__device__ __forceinline__ void loader_role(const ConvParams& p, const Bars& bars, uint32_t a_base, int64_t it0, int64_t it1,
                            const WaitCtx& ctx) {
  if (p.a_tma) return;  // warp 0 loads the operand with TMA
  const int tid = threadIdx.x - 32 * kFirstLoadWarp;
  const bool flat = p.mode == kModeFlat;
  const int nch = p.nch;
  const uint32_t plane = p.lbo_a;
  const int64_t ld_pix = p.ld_pix, ld_chunk = p.ld_chunk;
  const int row_len = flat ? p.flat_box : p.Wd;
  const int per_row = row_len * nch;
  const bool tabled = per_row <= kMaxLoadEntries * kLoaders;
  // This thread's (position, chunk) entries of one plane row.
  uint32_t ent_dst[kMaxLoadEntries];
  int ent_iw0[kMaxLoadEntries], ent_jo[kMaxLoadEntries];  // ent_jo: the entry's 16-channel chunk
  int n_ent = 0;
#pragma unroll
  for (int i = 0; i < kMaxLoadEntries; ++i) {
    const int e = tid + i * kLoaders;
    ent_dst[i] = 0;
    ent_iw0[i] = 0;
    ent_jo[i] = 0;
    if (tabled && e < per_row) {
      const int w = static_cast<int>(__umulhi(static_cast<uint32_t>(e), p.nch_magic));
      const int j = e - w * nch;
      ent_dst[i] = static_cast<uint32_t>(j) * plane + static_cast<uint32_t>(w) * 16u;
      ent_iw0[i] = flat ? w : p.stride * (p.w_coord + w);
      ent_jo[i] = j;
      n_ent = i + 1;
    }
  }
  // Per-row values that depend on the stride phase, held in registers (a
  // dynamically indexed kernel-parameter array costs a long-latency load).
  const int pa0 = p.phase_a[0], pa1 = p.phase_a[1], pa2 = p.phase_a[2], pa3 = p.phase_a[3];
  const int pb0 = p.phase_b[0], pb1 = p.phase_b[1], pb2 = p.phase_b[2], pb3 = p.phase_b[3];
  const int depth = min(2, p.a_stages - 1);
  Ring ra{0, 0, static_cast<uint32_t>(p.a_stages)};
  int64_t issued = 0, released = 0;
  bool ok = true;
  const int nph = flat ? 1 : p.nph, Hd = flat ? 1 : p.Hd;
  Item item = item_begin(p, it0);
  for (int64_t it = it0; it < it1 && ok; ++it, item_next(p, item)) {
    for (int kb = 0; kb < p.n_kb; ++kb) {
      if (!warp_wait(bars.a_empty(ra.stage), ra.phase ^ 1u, ctx)) { ok = false; break; }
      const uint32_t stage = a_base + ra.stage * p.a_stage_bytes;
      const int ch0 = p.src_group[item.g] * p.Cin_g + kb * p.KC;  // first input channel of the K block
      const uint8_t* img_src = p.q_in + item.n * p.ld_img + static_cast<int64_t>(ch0) * p.ld_c0_mul / 16;
      for (int ph = 0; ph < nph; ++ph)
      for (int r = 0; r < Hd; ++r) {
        bool row_ok;
        const uint8_t* row_src;
        uint32_t row_dst;
        int b, w_lim;
        if (flat) {
          const int p0 = item.rb * p.flat_box;  // first pixel of the tile in its image
          row_ok = true;
          row_src = img_src + static_cast<int64_t>(p0) * ld_pix;
          row_dst = stage;
          b = 0;
          w_lim = min(p.img_pix - p0, p.flat_box);
        } else {
          const int pa = ph == 0 ? pa0 : ph == 1 ? pa1 : ph == 2 ? pa2 : pa3;
          const int ih = p.stride * (item.oh0(p.Ht) + p.h_off + r) + pa;
          row_ok = ih >= 0 && ih < p.H;
          row_src = img_src + (row_ok ? ih : 0) * p.ld_row;
          row_dst = stage + ph * p.a_phase_bytes + static_cast<uint32_t>(r * p.Wd) * 16u;
          b = ph == 0 ? pb0 : ph == 1 ? pb1 : ph == 2 ? pb2 : pb3;
          w_lim = p.W;
        }
        if (tabled) {
#pragma unroll
          for (int i = 0; i < kMaxLoadEntries; ++i) {
            if (i < n_ent) {
              const int iw = ent_iw0[i] + b;
              const bool valid = row_ok && iw >= 0 && iw < w_lim;
              cp_async_16(row_dst + ent_dst[i], valid ? row_src + iw * ld_pix + ent_jo[i] * ld_chunk : p.q_in,
                          valid ? 16u : 0u);
            }
          }
        } else {
          for (int e = tid; e < per_row; e += kLoaders) {
            const int w = static_cast<int>(__umulhi(static_cast<uint32_t>(e), p.nch_magic));
            const int j = e - w * nch;
            const int iw = (flat ? w : p.stride * (p.w_coord + w)) + b;
            const bool valid = row_ok && iw >= 0 && iw < w_lim;
            cp_async_16(row_dst + static_cast<uint32_t>(j) * plane + static_cast<uint32_t>(w) * 16u,
                        valid ? row_src + iw * ld_pix + j * ld_chunk : p.q_in, valid ? 16u : 0u);
          }
        }
      }
      cp_async_commit();
      ++issued;
      ra.advance();
      // Release the oldest stage once only `depth` newer ones may still be pending.
      if (issued - released > depth) {
        if (depth >= 2) cp_async_wait<2>();
        else cp_async_wait<1>();
        load_release(bars, released, p.a_stages);
        ++released;
      }
    }
  }
  cp_async_wait<0>();
  while (released < issued) {
    load_release(bars, released, p.a_stages);
    ++released;
  }
}

// --------------------------------------------------------------------------
// Unpack role for packed 2-bit codes (warps 2-5): each staged TMA box of
// 32-bit words (16 codes of one position and 16-channel chunk) is expanded into
// the operand stage, one byte per code.  A staged row of chunk j and tile row r
// holds pk_box_w words starting pk_off positions left of the tile's first
// position (the TMA start is rounded down to 16 bytes); positions outside the
// image were zero-filled by the TMA unit, which is the zero padding.  Warp wi
// takes rows wi, wi + 4, ... and its lanes consecutive positions, so the 4-byte
// reads and 16-byte writes of shared memory are conflict-free.  The stage is
// released to the tensor core after a proxy fence (generic writes, async-proxy
// reads), and the staging stage back to the producer.
// --------------------------------------------------------------------------
__device__ __forceinline__ void unpack_role(const ConvParams& p, const Bars& bars, uint32_t a_base, uint32_t pk_base,
                                            int64_t it0, int64_t it1, const WaitCtx& ctx) {
  const int tid = threadIdx.x - 32 * kFirstLoadWarp;
  const int wi = tid >> 5, lane = tid & 31;
  const bool flat = p.mode == kModeFlat;
  const int row_len = flat ? p.flat_box : p.Wd;
  const int n_rows = p.nch * (flat ? 1 : p.Hd);
  const int Hd = flat ? 1 : p.Hd;
  const uint32_t plane = p.lbo_a;  // bytes between 16-channel chunks of the operand stage
  Ring r{0, 0, static_cast<uint32_t>(p.a_stages)};
  bool ok = true;
  for (int64_t it = it0; it < it1 && ok; ++it) {
    for (int kb = 0; kb < p.n_kb; ++kb) {
      if (!warp_wait(bars.pk_full(r.stage), r.phase, ctx)) { ok = false; break; }
      if (!warp_wait(bars.a_empty(r.stage), r.phase ^ 1u, ctx)) { ok = false; break; }
      const uint32_t src = pk_base + r.stage * p.pk_stage_bytes;
      const uint32_t dst = a_base + r.stage * p.a_stage_bytes;
      for (int row = wi; row < n_rows; row += kLoadWarps) {
        const int j = row / Hd, rr = row - j * Hd;
        const uint32_t srow = src + static_cast<uint32_t>(row * p.pk_box_w + p.pk_off) * 4u;
        const uint32_t drow = dst + static_cast<uint32_t>(j) * plane + static_cast<uint32_t>(rr * row_len) * 16u;
        for (int w = lane; w < row_len; w += 32) {
          uint32_t v;
          asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(srow + static_cast<uint32_t>(w) * 4u) : "memory");
          const uint4 u = unpack2_word(v);
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(drow + static_cast<uint32_t>(w) * 16u),
                       "r"(u.x), "r"(u.y), "r"(u.z), "r"(u.w)
                       : "memory");
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bars.a_full(r.stage));
        mbar_arrive(bars.pk_empty(r.stage));
      }
      r.advance();
    }
  }
}

// --------------------------------------------------------------------------
// Split role for stride 2 (warps 2-5): a staged window holds, per 16-byte chunk
// j, 2 Hd input rows of 2 Wd positions (16 bytes each) starting at input row
// 2 (oh0 + h_off) and column 2 w_coord; staged row y = 2 r + a and column
// x = 2 w + b go to row r, position w of the plane of stride phase (a, b) (the
// phases no tap uses are skipped).  Warp wi takes window rows wi, wi + 4, ...
// of every chunk and its lanes consecutive columns: conflict-free 16-byte reads, and 16-byte
// writes in two runs of consecutive positions.  Positions outside the image were
// zero-filled by the TMA unit (the zero padding).  The stage goes to the tensor
// core after a proxy fence, the staging stage back to the producer.
// --------------------------------------------------------------------------
__device__ __forceinline__ void split_role(const ConvParams& p, const Bars& bars, uint32_t a_base, uint32_t pk_base,
                                           int64_t it0, int64_t it1, const WaitCtx& ctx) {
  const int tid = threadIdx.x - 32 * kFirstLoadWarp;
  const int wi = tid >> 5, lane = tid & 31;
  const int Hd = p.Hd, Wd = p.Wd, Ws = 2 * p.Wd, nch = p.nch;
  const uint32_t plane = p.lbo_a;
  // destination offset of phase (a, b), or -1 where no tap reads it, in
  // registers (a dynamically indexed local array would live in local memory,
  // one long-latency load per staged row)
  int o00 = -1, o01 = -1, o10 = -1, o11 = -1;
#pragma unroll
  for (int q = 0; q < kMaxPhases; ++q) {
    if (q >= p.nph) break;
    const int v = q * static_cast<int>(p.a_phase_bytes);
    const int pa = p.phase_a[q] & 1, pb = p.phase_b[q] & 1;
    if (pa == 0) {
      if (pb == 0) o00 = v; else o01 = v;
    } else {
      if (pb == 0) o10 = v; else o11 = v;
    }
  }
  Ring r{0, 0, static_cast<uint32_t>(p.a_stages)};
  bool ok = true;
  for (int64_t it = it0; it < it1 && ok; ++it) {
    for (int kb = 0; kb < p.n_kb; ++kb) {
      if (!warp_wait(bars.pk_full(r.stage), r.phase, ctx)) { ok = false; break; }
      if (!warp_wait(bars.a_empty(r.stage), r.phase ^ 1u, ctx)) { ok = false; break; }
      const uint32_t src = pk_base + r.stage * p.pk_stage_bytes;
      const uint32_t dst = a_base + r.stage * p.a_stage_bytes;
      for (int y = wi; y < 2 * Hd; y += kLoadWarps) {
        const int a = y & 1, rr = y >> 1;
        const int off0 = a ? o10 : o00, off1 = a ? o11 : o01;
        if (off0 < 0 && off1 < 0) continue;
        for (int j = 0; j < nch; ++j) {
          const uint32_t srow = src + static_cast<uint32_t>((j * 2 * Hd + y) * Ws) * 16u;
          const uint32_t drow = dst + static_cast<uint32_t>(j) * plane + static_cast<uint32_t>(rr * Wd) * 16u;
          for (int x = lane; x < Ws; x += 32) {
            const int off = (x & 1) ? off1 : off0;
            if (off < 0) continue;
            uint32_t v0, v1, v2, v3;
            asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(v0), "=r"(v1), "=r"(v2), "=r"(v3)
                         : "r"(srow + static_cast<uint32_t>(x) * 16u)
                         : "memory");
            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(drow + static_cast<uint32_t>(off) +
                                                                           static_cast<uint32_t>(x >> 1) * 16u),
                         "r"(v0), "r"(v1), "r"(v2), "r"(v3)
                         : "memory");
          }
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bars.a_full(r.stage));
        mbar_arrive(bars.pk_empty(r.stage));
      }
      r.advance();
    }
  }
}

// --------------------------------------------------------------------------
// Tensor-core issue role (warp 1).
// --------------------------------------------------------------------------

constexpr int kUnrollTaps = 9;

template <int KSTEPS, int MT, bool F4>
__device__ __forceinline__ void mma_role(const ConvParams& p, const Bars& bars, uint32_t a_base, uint32_t b_base,
                                         uint32_t tmem_base, const uint32_t* tap_a16, int64_t it0, int64_t it1,
                                         const WaitCtx& ctx) {
  // The issue loop must stay lean: the whole warp runs it converged and one
  // elected lane issues each MMA; every extra instruction, branch or
  // long-latency load per MMA lowers tensor-core throughput directly, the more
  // so as the epilogue warps compete for the same schedulers.  So the K steps
  // and accumulators per tap are compile-time (fully unrolled), operand
  // addresses are 32-bit adds of 16-byte-unit offsets onto the low word of
  // precomputed descriptors (shared-memory addresses are below 2^18, so the
  // 14-bit address field never carries), and the per-tap offsets sit in
  // registers.  Waits are taken by all lanes and agreed on with a vote, so the
  // warp stays converged even when a wait times out.
  Ring ra{0, 0, static_cast<uint32_t>(p.a_stages)};
  Ring rb{0, 0, static_cast<uint32_t>(p.b_resident ? 1 : p.b_stages)};
  Ring racc{0, 0, static_cast<uint32_t>(p.acc_stages)};
  const uint32_t idesc = F4 ? idesc_mxf4_f32(128, p.Nblk) : idesc_e4m3_f32(128, p.Nblk);
  // FP4: scale factors of A and B (all 2^-4, so a product is v/2 * w * 2^-8 =
  // v * w * 2^-9, the same raw accumulator as the FP8 path).
  const uint32_t sfa = tmem_base + p.sf_col, sfb = tmem_base + p.sf_col + 16u;
  const uint64_t a_desc0 = smem_desc(a_base, p.lbo_a, 128u);
  const uint64_t b_desc0 = smem_desc(b_base, p.lbo_b, 128u);
  const uint64_t a_hi = a_desc0 & 0xFFFFFFFF00000000ull, b_hi = b_desc0 & 0xFFFFFFFF00000000ull;
  const uint32_t a_lo0 = static_cast<uint32_t>(a_desc0), b_lo0 = static_cast<uint32_t>(b_desc0);
  const uint32_t a_ks16 = (2u * p.lbo_a) >> 4, b_ks16 = (2u * p.lbo_b) >> 4;  // one K step (32 bytes of K)
  const uint32_t a_stage16 = p.a_stage_bytes >> 4, b_slice16 = p.b_slice_bytes >> 4;
  const uint32_t b_tap16 = static_cast<uint32_t>(p.n_kb) * b_slice16;  // one tap of all K blocks
  const uint32_t amt = p.a_mt16;  // A operand of accumulator mt starts mt * amt 16-byte units in
  const int taps = p.taps, n_kb = p.n_kb;
  const uint32_t npow2 = static_cast<uint32_t>(p.Npow2);
  const bool resident = p.b_resident != 0;
  const int64_t tiles = p.tiles;
  uint32_t tap_reg[kUnrollTaps];
#pragma unroll
  for (int t = 0; t < kUnrollTaps; ++t) tap_reg[t] = t < taps ? tap_a16[t] : 0u;
  int unit = -1;
  int tile = static_cast<int>(it0 % tiles);
  int unit_next = static_cast<int>(it0 / tiles);
  bool ok = true;
  for (int64_t it = it0; it < it1 && ok; ++it) {
    const int cur = unit_next;
    if (++tile == tiles) {
      tile = 0;
      ++unit_next;
    }
    if (resident && cur != unit) {
      if (!warp_wait(bars.b_full(rb.stage), rb.phase, ctx)) { ok = false; break; }
      unit = cur;
    }
    if (!warp_wait(bars.acc_empty(racc.stage), racc.phase ^ 1u, ctx)) { ok = false; break; }
    tc_fence_after();
    const uint32_t d0 = tmem_base + racc.stage * static_cast<uint32_t>(MT) * npow2;
    for (int kb = 0; kb < n_kb && ok; ++kb) {
      if (!warp_wait(bars.a_full(ra.stage), ra.phase, ctx)) { ok = false; break; }
      tc_fence_after();
      const uint32_t a_lo_stage = a_lo0 + ra.stage * a_stage16;
      // packed weights are tap-major: tap t of K block kb is slice t * n_kb + kb
      const uint32_t b_lo_kb = b_lo0 + static_cast<uint32_t>(kb) * b_slice16;
      // One tap: KSTEPS x MT MMAs, fully unrolled.
      auto issue_tap = [&](int t, uint32_t a_lo_tap, uint32_t b_lo_tap) {
        const uint32_t acc0 = (kb | t) == 0 ? 0u : 1u;
#pragma unroll
        for (int ks = 0; ks < KSTEPS; ++ks) {
          const uint64_t bdesc = b_hi | (b_lo_tap + static_cast<uint32_t>(ks) * b_ks16);
          const uint32_t a_lo = a_lo_tap + static_cast<uint32_t>(ks) * a_ks16;
          const uint32_t acc = ks == 0 ? acc0 : 1u;
          if constexpr (F4) {
            if constexpr (MT == 4) {
              tc_mma4_f4_warp(d0, d0 + npow2, d0 + 2 * npow2, d0 + 3 * npow2, a_hi | a_lo, a_hi | (a_lo + amt),
                              a_hi | (a_lo + 2u * amt), a_hi | (a_lo + 3u * amt), bdesc, idesc, sfa, sfb, acc);
            } else if constexpr (MT == 3) {
              tc_mma3_f4_warp(d0, d0 + npow2, d0 + 2 * npow2, a_hi | a_lo, a_hi | (a_lo + amt), a_hi | (a_lo + 2u * amt),
                              bdesc, idesc, sfa, sfb, acc);
            } else if constexpr (MT == 2) {
              tc_mma2_f4_warp(d0, d0 + npow2, a_hi | a_lo, a_hi | (a_lo + amt), bdesc, idesc, sfa, sfb, acc);
            } else {
              tc_mma_f4_warp(d0, a_hi | a_lo, bdesc, idesc, sfa, sfb, acc);
            }
          } else if constexpr (MT == 4) {
            tc_mma4_e4m3_warp(d0, d0 + npow2, d0 + 2 * npow2, d0 + 3 * npow2, a_hi | a_lo, a_hi | (a_lo + amt),
                              a_hi | (a_lo + 2u * amt), a_hi | (a_lo + 3u * amt), bdesc, idesc, acc);
          } else if constexpr (MT == 3) {
            tc_mma3_e4m3_warp(d0, d0 + npow2, d0 + 2 * npow2, a_hi | a_lo, a_hi | (a_lo + amt), a_hi | (a_lo + 2u * amt),
                              bdesc, idesc, acc);
          } else if constexpr (MT == 2) {
            tc_mma2_e4m3_warp(d0, d0 + npow2, a_hi | a_lo, a_hi | (a_lo + amt), bdesc, idesc, acc);
          } else {
            tc_mma_e4m3_warp(d0, a_hi | a_lo, bdesc, idesc, acc);
          }
        }
      };
      if (resident && taps <= kUnrollTaps) {
        // Up to 9 taps unrolled with their offsets in registers: no loads or
        // loop branches between the MMAs of a K block.
#pragma unroll
        for (int t = 0; t < kUnrollTaps; ++t)
          if (t < taps) issue_tap(t, a_lo_stage + tap_reg[t], b_lo_kb + static_cast<uint32_t>(t) * b_tap16);
      } else {
        for (int t = 0; t < taps; ++t) {
          uint32_t b_lo_tap;
          if (resident) {
            b_lo_tap = b_lo_kb + static_cast<uint32_t>(t) * b_tap16;
          } else {
            if (!warp_wait(bars.b_full(rb.stage), rb.phase, ctx)) { ok = false; break; }
            tc_fence_after();
            b_lo_tap = b_lo0 + rb.stage * b_slice16;
          }
          issue_tap(t, a_lo_stage + tap_a16[t], b_lo_tap);
          if (!resident) {
            tc_commit_warp(bars.b_empty(rb.stage));
            rb.advance();
          }
        }
      }
      if (!ok) break;
      tc_commit_warp(bars.a_empty(ra.stage));
      ra.advance();
    }
    if (!ok) break;
    tc_commit_warp(bars.acc_full(racc.stage));
    racc.advance();
    if (resident && (it + 1 >= it1 || unit_next != cur)) {
      tc_commit_warp(bars.b_empty(rb.stage));
      rb.advance();
    }
  }
  // Drain: wait until every MMA this warp issued has completed.
  tc_commit_warp(bars.drain());
  mbar_wait_drain(bars.drain(), 0, ctx.limit_ns, ctx.err);
}

// Dispatch to the MMA role compiled for this layer's K steps per tap and
// accumulators per tile (and operand type: F4 for packed FP4 codes).
template <bool F4>
__device__ __forceinline__ void mma_role_dispatch(const ConvParams& p, const Bars& bars, uint32_t a_base, uint32_t b_base,
                                                  uint32_t tmem_base, const uint32_t* tap_a16, int64_t it0, int64_t it1,
                                                  const WaitCtx& ctx) {
  const int ks = p.nch >> 1;  // one MMA takes 32 bytes of K: 32 FP8 or 64 FP4 channels
#define PQ_MMA_CASE(K, M) \
  if (ks == K && p.MT == M) return mma_role<K, M, F4>(p, bars, a_base, b_base, tmem_base, tap_a16, it0, it1, ctx);
  PQ_MMA_CASE(1, 1) PQ_MMA_CASE(1, 2) PQ_MMA_CASE(1, 3) PQ_MMA_CASE(1, 4)
  PQ_MMA_CASE(2, 1) PQ_MMA_CASE(2, 2) PQ_MMA_CASE(2, 3) PQ_MMA_CASE(2, 4)
  PQ_MMA_CASE(3, 1) PQ_MMA_CASE(3, 2) PQ_MMA_CASE(3, 3) PQ_MMA_CASE(3, 4)
  PQ_MMA_CASE(4, 1) PQ_MMA_CASE(4, 2) PQ_MMA_CASE(4, 3) PQ_MMA_CASE(4, 4)
  PQ_MMA_CASE(8, 1) PQ_MMA_CASE(8, 2) PQ_MMA_CASE(8, 3) PQ_MMA_CASE(8, 4)
#undef PQ_MMA_CASE
  // The planner only produces the shapes above; anything else is a planner bug.
  atomicOr(ctx.err, PQ_ERR_TIMEOUT | PQ_ERR_MMA);
  *ctx.abort_flag = 1;
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

// Requantised code of t = clamp(rint(t), 0, qmax) with round-half-to-even, on the
// FMA and integer pipes: clamping t to [-1, qmax + 1] first does not change the
// result (rounding is monotone and the final clamp is integral), and for
// |r| < 2^22 the fp32 sum r + 1.5 * 2^23 is rounded by the adder to the nearest
// integer, ties to even, which then sits in the low mantissa bits.  NaN -> 0.
__device__ __forceinline__ int requant_code(float t, float qmax_f, int qmax) {
  const float r = fminf(fmaxf(t, -1.0f), qmax_f + 1.0f);
  int i = __float_as_int(__fadd_rn(r, 12582912.0f)) - 0x4B400000;
  return min(max(i, 0), qmax);
}

// Item-level constants of the epilogue.
struct EpiItem {
  uint32_t tbase;        // TMEM address of accumulator 0, this warp's lanes
  float m_out512, m_req512, m_req;
  float m_req15;         // m_req * 2^-15 (codes-only conversion through fp16, see epi_codes16_f16)
  int g, src_c0, dst_c0;
  int n, rb, oh0;
  int nb;
};

// Output pixel (within its image) of accumulator row m, and whether it exists.
__device__ __forceinline__ int epi_pos(const ConvParams& p, const EpiItem& e, int m, bool& valid) {
  if (p.mode == kModeFlat) {
    const int pos = e.rb * p.flat_box + m;
    valid = m < p.flat_box && pos < p.img_pix;
    return pos;
  }
  const int r = static_cast<int>(__umulhi(static_cast<uint32_t>(m), p.wh_magic));  // m / Wh
  const int c = m - r * p.Wh;
  const int oh = e.oh0 + r;
  valid = (r < p.Ht) && (c < p.Wo) && (oh < p.Ho);
  return oh * p.Wo + c;
}

// Quantise-on-load with learned bounds: the codes rint(sat((x - l) * inv_r) * Qp)
// of 16 fp32 values, one rounding per operation (x - l as x + (-l), exact), the
// rounding to an integer by the fp32 add of 1.5 * 2^23 (its low 16 bits); sat
// maps NaN to 0, so NaN-filled padding gives code 0 whatever l is.  The product
// with Qp is a scalar __fmul_rn: a packed mul.rn.f32x2 followed by the packed add
// was fused into one FMA by the compiler (the product then not rounded first),
// which changes the rounding at ties.
__device__ __forceinline__ uint4 lu_codes16(const uint32_t (&v)[16], float neg_l, float inv_r, float qp,
                                            uint32_t qmax2) {
  uint32_t h[8];
#pragma unroll
  for (int j = 0; j < 16; j += 2) {
    float d0, d1, y0, y1, r0, r1;
    add2_rn(__uint_as_float(v[j]), __uint_as_float(v[j + 1]), neg_l, d0, d1);
    const float c0 = mul_sat(d0, inv_r), c1 = mul_sat(d1, inv_r);
    y0 = __fmul_rn(c0, qp);
    y1 = __fmul_rn(c1, qp);
    add2_rn(y0, y1, 12582912.0f, r0, r1);
    h[j >> 1] = __vimin_s16x2_relu(__byte_perm(__float_as_uint(r0), __float_as_uint(r1), 0x5410), qmax2);
  }
  uint4 w;
  w.x = __byte_perm(h[0], h[1], 0x6420);
  w.y = __byte_perm(h[2], h[3], 0x6420);
  w.z = __byte_perm(h[4], h[5], 0x6420);
  w.w = __byte_perm(h[6], h[7], 0x6420);
  return w;
}

// Code packing of the channel-blocked output: 0 one code per byte, 1 four 2-bit
// codes per byte, 2 two FP4 nibbles per byte.
__device__ __forceinline__ int codes_pack(const ConvParams& p) { return p.codes_p2 ? 1 : (p.codes_f4 ? 2 : 0); }

// 16 codes (one per byte of w) to global memory: as they are (16 bytes), packed
// four to a byte (4 bytes) or two to a byte (8 bytes, half of a 32-channel row).
__device__ __forceinline__ void store_codes16(uint8_t* dst, uint4 w, int pack) {
  if (pack == 1)
    *reinterpret_cast<uint32_t*>(dst) = pack2_word(w);
  else if (pack == 2)
    *reinterpret_cast<uint2*>(dst) = pack4_word(w);
  else
    *reinterpret_cast<uint4*>(dst) = w;
}

// Byte offset of the 16 codes of output pixel pos (in its image n) and the
// 16-channel chunk k = channel / 16, channel-blocked.
__device__ __forceinline__ long long codes_offset(const ConvParams& p, int pack, int n, long long hw_out, int pos, int k) {
  if (pack == 2)
    return ((static_cast<long long>(n) * (p.C_out_total >> 5) + (k >> 1)) * hw_out + pos) * 16 + (k & 1) * 8;
  return ((static_cast<long long>(n) * (p.C_out_total >> 4) + k) * hw_out + pos) * (pack ? 4 : 16);
}

// --------------------------------------------------------------------------
// Quantise-on-load role (warps 2-5): each staged box holds, per position of the
// stage, the 32 fp32 activations of the K block as one 128-byte row, swizzled
// 128B (16-byte chunk c of row r at chunk c ^ (r & 7), the rows' bank groups
// spread).  Thread items are (position, box): eight 16-byte reads of the row,
// the codes clamp(rint(x * fl(1/s)), 0, Qp) of the input group (one fp32
// multiply, the saturating form of the epilogue's conversion, NaN -> 0), and
// 16-byte writes to the operand planes: one per 16-channel half for byte codes,
// one for the row's 32 FP4 nibbles.  Positions outside the image were
// zero-filled by the TMA unit: code 0, the zero padding.
// --------------------------------------------------------------------------
template <bool F4, bool LU>
__device__ __forceinline__ void quant_role(const ConvParams& p, const Bars& bars, uint32_t a_base, uint32_t st_base,
                                           int64_t it0, int64_t it1, const WaitCtx& ctx) {
  const int tid = threadIdx.x - 32 * kFirstLoadWarp;
  const int lane = tid & 31;
  const int npos = p.mode == kModeFlat ? p.flat_box : p.Hd * p.Wd;
  const uint32_t box_bytes = p.q_box_bytes;  // one 32-channel fp32 box (1024-byte aligned)
  // items (position, box j): one 128-byte row of 32 channels each; the stage
  // holds KC / 32 boxes, a power of two
  const int lg_nbox = __ffs(p.KC >> 5) - 1;
  const int n_items = npos << lg_nbox;
  const uint32_t plane = p.lbo_a;
  const float two_b = p.q_two_b;
  const uint32_t qmax2 = p.q_qmax2;
  Ring r{0, 0, static_cast<uint32_t>(p.a_stages)};
  bool ok = true;
  Item item = item_begin(p, it0);
  const float qp = p.q_qp;
  for (int64_t it = it0; it < it1 && ok; ++it, item_next(p, item)) {
    const int sg = p.src_group[item.g];
    const float m_sat = LU ? p.q_inv_r[sg] : p.q_inv_sat[sg];
    const float neg_l = LU ? p.q_neg_l[sg] : 0.0f;
    auto codes16 = [&](const uint32_t (&x)[16]) {
      if constexpr (LU) return lu_codes16(x, neg_l, m_sat, qp, qmax2);
      else return epi_codes16(x, m_sat, two_b, qmax2);
    };
    for (int kb = 0; kb < p.n_kb; ++kb) {
      if (!warp_wait(bars.pk_full(r.stage), r.phase, ctx)) { ok = false; break; }
      if (!warp_wait(bars.a_empty(r.stage), r.phase ^ 1u, ctx)) { ok = false; break; }
      const uint32_t src = st_base + r.stage * p.pk_stage_bytes;
      const uint32_t dst = a_base + r.stage * p.a_stage_bytes;
      for (int e = tid; e < n_items; e += 32 * kLoadWarps) {
        const int pos = e >> lg_nbox, j = e & ((1 << lg_nbox) - 1);
        const uint32_t row = src + static_cast<uint32_t>(j) * box_bytes + static_cast<uint32_t>(pos) * 128u;
        if (F4) {
          // FP4 nibbles: operand chunk j is box j, the whole row: 32 codes packed
          // two to a byte
          const uint32_t out = dst + static_cast<uint32_t>(j) * plane + static_cast<uint32_t>(pos) * 16u;
          uint32_t v[16];
          uint2 packed[2];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint32_t a = row + ((static_cast<uint32_t>(4 * h + k) ^ static_cast<uint32_t>(pos & 7)) << 4);
              asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                           : "=r"(v[4 * k]), "=r"(v[4 * k + 1]), "=r"(v[4 * k + 2]), "=r"(v[4 * k + 3])
                           : "r"(a)
                           : "memory");
            }
            packed[h] = pack4_word(codes16(v));
          }
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(out), "r"(packed[0].x), "r"(packed[0].y),
                       "r"(packed[1].x), "r"(packed[1].y)
                       : "memory");
        } else {
          // byte codes: the row's two 16-channel halves are operand chunks 2j and
          // 2j + 1 (all eight reads issued before the conversions)
          const uint32_t out = dst + static_cast<uint32_t>(2 * j) * plane + static_cast<uint32_t>(pos) * 16u;
          uint32_t v[16], u[16];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint32_t a = row + ((static_cast<uint32_t>(k) ^ static_cast<uint32_t>(pos & 7)) << 4);
            const uint32_t b = row + ((static_cast<uint32_t>(4 + k) ^ static_cast<uint32_t>(pos & 7)) << 4);
            asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(v[4 * k]), "=r"(v[4 * k + 1]), "=r"(v[4 * k + 2]), "=r"(v[4 * k + 3])
                         : "r"(a)
                         : "memory");
            asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(u[4 * k]), "=r"(u[4 * k + 1]), "=r"(u[4 * k + 2]), "=r"(u[4 * k + 3])
                         : "r"(b)
                         : "memory");
          }
          const uint4 w0 = codes16(v);
          const uint4 w1 = codes16(u);
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(out), "r"(w0.x), "r"(w0.y), "r"(w0.z),
                       "r"(w0.w)
                       : "memory");
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(out + plane), "r"(w1.x), "r"(w1.y), "r"(w1.z),
                       "r"(w1.w)
                       : "memory");
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bars.a_full(r.stage));
        mbar_arrive(bars.pk_empty(r.stage));
      }
      r.advance();
    }
  }
}

// Store 16 codes of 16-column chunk `ch` of the row (output pixel pos).
__device__ __forceinline__ void epi_store_codes(const ConvParams& p, const EpiItem& e, uint8_t* stg, int lane, bool valid,
                                                int pos, int ch, uint4 w) {
  const long long hw_out = static_cast<long long>(p.Ho) * p.Wo;
  if (p.codes_c16) {
    // Channel-blocked codes: lanes hold consecutive pixels, so each store of the
    // warp lands next to its neighbours'.
    if (valid) {
      const int pack = codes_pack(p);
      store_codes16(p.q_out + codes_offset(p, pack, e.n, hw_out, pos, (e.dst_c0 >> 4) + ch), w, pack);
    }
  } else {
    // NHWC: staged, then 16-byte rows written by the warp.
    *reinterpret_cast<uint4*>(stg + lane * p.stage_q_pitch) = w;
    const long long pix = static_cast<long long>(e.n) * hw_out + pos;
    warp_store_rows(stg, p.stage_q_pitch, 16, p.q_out, valid ? pix * p.C_out_total + e.dst_c0 + ch * 16 : -1, lane);
  }
}

// General units (int32 sums, fp32 outputs with or without the shortcut, codes)
// of UC accumulator columns.  TMEM gives each lane one row (pixel), but a global
// access instruction costs about one cycle per cache line it touches, so rows
// of 4 UC bytes per lane would cost 32 lines per instruction.  The shortcut,
// the fp32 outputs and the int32 sums therefore pass through the warp's staging
// buffer (32 rows of 4 UC bytes; 16-byte chunk c of row r at chunk c ^ sw(r),
// which keeps both access patterns conflict-free): a global access instruction
// takes whole rows, 512 bytes in 4 rows of 128 (UC = 32) or 8 rows of 64
// (UC = 16), and each lane reads or writes its own row in shared memory.  The shortcut comes by
// cp.async (zero-filled for rows outside the output).  Codes go through the
// fp16 conversion (epi_codes16_f16) where no NaN can reach it: without a
// shortcut the value is fl(raw * m_req * 2^-15) = fl(acc * m_req) * 2^-24; with
// one, fl(y * m_req * 2^-24) = fl(y * m_req) * 2^-24 (a power-of-two factor,
// exact while the product is normal; both give code 0 below that), and ReLU has
// removed NaN (fmaxf(NaN, 0) = 0).  A shortcut without ReLU keeps the scalar
// form, which maps NaN to code 0.
template <int UC>
__device__ __forceinline__ uint32_t stg_chunk(uint32_t base, int r, int c) {
  constexpr int CPR = UC / 4;  // 16-byte chunks per staged row
  const int sw = (UC == 32 ? r : r >> 1) & (CPR - 1);
  return base + static_cast<uint32_t>(r * (UC * 4) + ((c ^ sw) << 4));
}

template <int UC>
__device__ __forceinline__ void epi_general_units(const ConvParams& p, const EpiItem& e, uint8_t* stg, int wg,
                                                  int n_groups, int quarter, int lane, uint32_t qmax2) {
  constexpr int CPR = UC / 4, RPP = 32 / CPR;  // chunks per row, rows per coalesced pass
  // one staging buffer: 32 rows of 128 bytes whatever UC is, so that the NHWC code
  // rows staged by epi_store_codes (32 rows at an 80-byte pitch) stay inside it
  constexpr uint32_t kBuf = 32u * 128u;
  const bool has_sc = p.shortcut != nullptr;
  // With a shortcut (and no int32 output, which would need the buffer first) the
  // next unit's shortcut rows are fetched into the warp's second buffer while
  // this unit computes and stores: the fetch latency then runs under the stores.
  const bool pre = has_sc && p.acc_out == nullptr;
  const bool f16q = !has_sc || p.relu;
  const float m_q = has_sc ? __fmul_rn(e.m_req, 1.0f / 16777216.0f) : e.m_req15;
  const int qmax = p.qmax_out;
  const float qmax_f = static_cast<float>(qmax);
  const int m_lane = quarter * 32 + lane;
  const long long hw_out = static_cast<long long>(p.Ho) * p.Wo;
  const int per_acc = p.Nblk / UC;
  const int n_units = p.MT * per_acc;
  const int pr = lane / CPR, pc = lane % CPR;  // row within a pass, chunk: coalesced role
  // Channel shuffle (kind 2): column j of the unit goes to destination channel
  // (nb Nblk + col0 + j) G + g, so a staged row leaves as UC values G apart:
  // lane j of a store instruction takes column j of 32 / UC rows.
  const bool shuf = p.channel_shuffle != 0;
  const int sj = lane % UC, sr = lane / UC;
  // this lane's row offset (elements; -1 outside the output) of unit u
  auto row_of = [&](int u, bool& valid, int& pos) -> long long {
    const int mt = u / per_acc;
    pos = epi_pos(p, e, mt * 128 + m_lane, valid);
    return valid ? (static_cast<long long>(e.n) * hw_out + pos) * p.C_out_total : -1;
  };
  // unit u's shortcut rows (its source channels) into buffer `buf` by cp.async,
  // whole rows per instruction, zero-filled outside the output
  auto fetch_sc = [&](int u, long long rc, uint32_t buf) {
    const int col0 = (u - (u / per_acc) * per_acc) * UC;
#pragma unroll
    for (int ps = 0; ps < CPR; ++ps) {
      const int r = ps * RPP + pr;
      const long long off = __shfl_sync(0xffffffffu, rc, r);
      cp_async_16(stg_chunk<UC>(buf, r, pc), off >= 0 ? p.shortcut + off + e.src_c0 + col0 + 4 * pc : p.shortcut,
                  off >= 0 ? 16u : 0u);
    }
    cp_async_commit();
  };
  int cur = 0;
  if (pre && wg < n_units) {
    bool v0;
    int p0;
    fetch_sc(wg, row_of(wg, v0, p0), smem_u32(stg));
  }
  for (int u = wg; u < n_units; u += n_groups, cur ^= 1) {
    const int mt = u / per_acc, col0 = (u - mt * per_acc) * UC;
    bool valid;
    int pos;
    const long long rowc = row_of(u, valid, pos);
    const uint32_t sbase = smem_u32(stg) + (pre ? static_cast<uint32_t>(cur) * kBuf : 0u);
    uint8_t* const stg_cur = stg + (pre ? cur * kBuf : 0u);
    if (pre) {
      if (u + n_groups < n_units) {
        bool vn;
        int pn;
        fetch_sc(u + n_groups, row_of(u + n_groups, vn, pn), smem_u32(stg) + static_cast<uint32_t>(cur ^ 1) * kBuf);
        cp_async_wait<1>();  // this unit's rows have landed; the next unit's may still be in flight
      } else {
        cp_async_wait<0>();
      }
      __syncwarp();
    }
    uint32_t v[UC];
    if constexpr (UC == 32)
      tmem_ld32(e.tbase + mt * p.Npow2 + col0, v);
    else
      tmem_ld16(e.tbase + mt * p.Npow2 + col0, v);
    // Whole staged rows to global memory (row r's element offset is lane r's rowc).
    auto store_rows = [&](void* out, int c0) {
      __syncwarp();
      if (shuf) {
        const long long dcl = static_cast<long long>(e.nb * p.Nblk + col0 + sj) * p.G + e.g;
#pragma unroll 4
        for (int r0 = 0; r0 < 32; r0 += 32 / UC) {
          const int r = r0 + sr;
          const long long off = __shfl_sync(0xffffffffu, rowc, r);
          uint32_t x;
          asm volatile("ld.shared.b32 %0, [%1];" : "=r"(x) : "r"(stg_chunk<UC>(sbase, r, sj >> 2) + 4u * (sj & 3)) : "memory");
          if (off >= 0) reinterpret_cast<uint32_t*>(out)[off + dcl] = x;
        }
        __syncwarp();
        return;
      }
#pragma unroll
      for (int ps = 0; ps < CPR; ++ps) {
        const int r = ps * RPP + pr;
        const long long off = __shfl_sync(0xffffffffu, rowc, r);
        uint32_t x0, x1, x2, x3;
        asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(x0), "=r"(x1), "=r"(x2), "=r"(x3)
                     : "r"(stg_chunk<UC>(sbase, r, pc))
                     : "memory");
        if (off >= 0)
          *reinterpret_cast<uint4*>(reinterpret_cast<uint32_t*>(out) + off + c0 + col0 + 4 * pc) =
              make_uint4(x0, x1, x2, x3);
      }
      __syncwarp();
    };
    // This lane's row of UC 32-bit values into the staging buffer.
    auto stage_row = [&](const uint32_t (&x)[UC]) {
#pragma unroll
      for (int c = 0; c < CPR; ++c)
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(stg_chunk<UC>(sbase, lane, c)), "r"(x[4 * c]),
                     "r"(x[4 * c + 1]), "r"(x[4 * c + 2]), "r"(x[4 * c + 3])
                     : "memory");
    };
    if (p.acc_out) {
      tmem_wait_ld();
      uint32_t a[UC];
#pragma unroll
      for (int j = 0; j < UC; ++j) a[j] = static_cast<uint32_t>(__float2int_rn(__fmul_rn(__uint_as_float(v[j]), 512.0f)));
      __syncwarp();
      stage_row(a);
      store_rows(p.acc_out, e.dst_c0);
    }
    if (has_sc && !pre) {
      // the rows' shortcut values into the staging buffer, after the int32 sums left it
      fetch_sc(u, rowc, sbase);
      cp_async_wait<0>();
      __syncwarp();
    }
    tmem_wait_ld();
    uint4 w[UC / 16];
    if (p.q_out && !has_sc) {
      w[0] = epi_codes16_f16<UC, 0>(v, m_q, qmax2);
      if constexpr (UC == 32) w[1] = epi_codes16_f16<UC, 16>(v, m_q, qmax2);
    }
    // y = relu(fl(acc * m_out) + shortcut), in place
#pragma unroll
    for (int c = 0; c < CPR; ++c) {
      float sc0 = 0.0f, sc1 = 0.0f, sc2 = 0.0f, sc3 = 0.0f;
      if (has_sc)
        asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                     : "=f"(sc0), "=f"(sc1), "=f"(sc2), "=f"(sc3)
                     : "r"(stg_chunk<UC>(sbase, lane, c))
                     : "memory");
      const float scv[4] = {sc0, sc1, sc2, sc3};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        float t = __fmul_rn(__uint_as_float(v[4 * c + k]), e.m_out512);  // = (float)acc * m_out, one rounding
        if (has_sc) t = __fadd_rn(t, scv[k]);
        if (p.relu) t = fmaxf(t, 0.0f);
        v[4 * c + k] = __float_as_uint(t);
      }
    }
    if (p.q_out && has_sc) {
      if (f16q) {
        w[0] = epi_codes16_f16<UC, 0>(v, m_q, qmax2);
        if constexpr (UC == 32) w[1] = epi_codes16_f16<UC, 16>(v, m_q, qmax2);
      } else {
#pragma unroll
        for (int h = 0; h < UC / 16; ++h) {
          int code[16];
#pragma unroll
          for (int j = 0; j < 16; ++j)
            code[j] = requant_code(__fmul_rn(__uint_as_float(v[16 * h + j]), e.m_req), qmax_f, qmax);
          w[h].x = __byte_perm(__byte_perm(code[0], code[1], 0x0040), __byte_perm(code[2], code[3], 0x0040), 0x5410);
          w[h].y = __byte_perm(__byte_perm(code[4], code[5], 0x0040), __byte_perm(code[6], code[7], 0x0040), 0x5410);
          w[h].z = __byte_perm(__byte_perm(code[8], code[9], 0x0040), __byte_perm(code[10], code[11], 0x0040), 0x5410);
          w[h].w = __byte_perm(__byte_perm(code[12], code[13], 0x0040), __byte_perm(code[14], code[15], 0x0040), 0x5410);
        }
      }
    }
    if (p.y_out) {
      __syncwarp();  // every lane has read its shortcut row
      stage_row(v);
      store_rows(p.y_out, e.dst_c0);
    }
    if (p.q_out && !shuf) {
      __syncwarp();
#pragma unroll
      for (int h = 0; h < UC / 16; ++h) epi_store_codes(p, e, stg_cur, lane, valid, pos, col0 / 16 + h, w[h]);
    } else if (p.q_out && valid) {
      // byte codes scattered one by one (the API takes no packed codes here)
#pragma unroll
      for (int h = 0; h < UC / 16; ++h) {
        const uint32_t wd[4] = {w[h].x, w[h].y, w[h].z, w[h].w};
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const long long dc = static_cast<long long>(e.nb * p.Nblk + col0 + 16 * h + j) * p.G + e.g;
          const long long o = p.codes_c16 ? ((static_cast<long long>(e.n) * (p.C_out_total >> 4) + (dc >> 4)) * hw_out + pos) * 16 + (dc & 15)
                                          : rowc + dc;
          p.q_out[o] = static_cast<uint8_t>(wd[j >> 2] >> (8 * (j & 3)));
        }
      }
    }
  }
}

// The epilogue's work per tile is a list of units, one per (accumulator mt,
// 16-column chunk); epilogue warpgroup wg of n_groups takes units wg,
// wg + n_groups, ...  Each warp handles the 32 TMEM lanes (rows) it may access.
// On the codes-only path the TMEM loads are double-buffered: the next unit's
// load is in flight while the current one is computed and stored.
template <bool F4>
__device__ __forceinline__ void epilogue_role(const ConvParams& p, const Bars& bars, uint32_t tmem_base,
                                              uint8_t* stage_base, int first_warp, int n_groups, int64_t it0,
                                              int64_t it1, const WaitCtx& ctx) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ew = warp - first_warp;  // epilogue warp index
  const int wg = ew >> 2;            // warpgroup
  const int quarter = warp & 3;      // TMEM lanes this warp may access
  uint8_t* stg = stage_base + ew * p.stage_warp_bytes;
  Ring racc{0, 0, static_cast<uint32_t>(p.acc_stages)};
  const int nchunks = p.Nblk >> 4;
  const int n_units = p.MT * nchunks;
  const bool codes_only = p.shortcut == nullptr && p.y_out == nullptr && p.acc_out == nullptr && !p.channel_shuffle;
  // The group's multipliers and destination stay in registers while consecutive
  // items share the group (items run group by group); a dynamically indexed
  // kernel-parameter array costs a long-latency constant load.
  int cur_g = -1, dst_g = 0;
  float g_m_out512 = 0.0f, g_m_req512 = 0.0f, g_m_req = 0.0f, g_m_req15 = 0.0f;
  const uint32_t qmax2 = static_cast<uint32_t>(p.qmax_out) * 0x00010001u;
  Item item = item_begin(p, it0);
  for (int64_t it = it0; it < it1; ++it, item_next(p, item)) {
    if (item.g != cur_g) {
      cur_g = item.g;
      g_m_out512 = p.m_out512[cur_g];
      g_m_req512 = p.m_req512[cur_g];
      g_m_req = p.m_req[cur_g];
      g_m_req15 = __fmul_rn(g_m_req, 1.0f / 32768.0f);  // exact: |m_req| is 0 or above 1e-30
      dst_g = p.dst_group[cur_g];
    }
    if (!warp_wait(bars.acc_full(racc.stage), racc.phase, ctx)) break;
    tc_fence_after();
    EpiItem e;
    e.g = item.g;
    e.nb = item.nb;
    e.n = item.n;
    e.rb = item.rb;
    e.oh0 = item.oh0(p.Ht);
    e.m_out512 = g_m_out512;
    e.m_req512 = g_m_req512;
    e.m_req = g_m_req;
    e.m_req15 = g_m_req15;
    e.src_c0 = e.g * p.Cout_g + item.nb * p.Nblk;     // source channel of column 0
    e.dst_c0 = dst_g * p.Cout_g + item.nb * p.Nblk;  // destination channel of column 0
    e.tbase = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + racc.stage * p.MT * p.Npow2;
    if (F4 && codes_only && (p.Nblk & 31) == 0) {
      // FP4 nibbles, units of 32 columns: a lane's 32 codes are one whole 16-byte
      // row of a 32-channel block, so a unit costs one store instruction (the
      // epilogue's time goes mostly to store instructions, not bytes).
      const int nb32 = p.Nblk >> 5;
      const long long blk_bytes = static_cast<long long>(p.Ho) * p.Wo * 16;
      uint8_t* const blk0 =
          p.q_out + (static_cast<long long>(e.n) * (p.C_out_total >> 5) + (e.dst_c0 >> 5)) * blk_bytes;
      const int m_lane = quarter * 32 + lane;
      const int MT = p.MT;
      auto row_ptr = [&](int mt) -> uint8_t* {
        if (mt >= MT) return nullptr;
        bool valid;
        const int pos = epi_pos(p, e, mt * 128 + m_lane, valid);
        return valid ? blk0 + static_cast<long long>(pos) * 16 : nullptr;
      };
      auto step = [&](int& mt, int& b) {
        b += n_groups;
        while (b >= nb32) {
          b -= nb32;
          ++mt;
        }
      };
      auto col = [&](int mt, int b) { return e.tbase + static_cast<uint32_t>(mt) * p.Npow2 + b * 32; };
      // Two 16-column buffers: the unit's first half (va) is converted while its
      // second half (vb) loads, and the next unit's first half loads while the
      // second half is converted and the row is stored.
      uint32_t va[16], vb[16];
      int c_mt = 0, c_b = wg - n_groups;
      step(c_mt, c_b);
      uint8_t* c_row = row_ptr(c_mt);
      if (c_mt < MT) {
        tmem_ld16(col(c_mt, c_b), va);
        tmem_wait_ld();
      }
      while (c_mt < MT) {
        tmem_ld16(col(c_mt, c_b) + 16, vb);
        const uint2 lo = pack4_word(epi_codes16_f16(va, e.m_req15, qmax2));
        tmem_wait_ld();
        int n_mt = c_mt, n_b = c_b;
        step(n_mt, n_b);
        if (n_mt < MT) tmem_ld16(col(n_mt, n_b), va);
        const uint2 hi = pack4_word(epi_codes16_f16(vb, e.m_req15, qmax2));
        tmem_wait_ld();  // before the store: a TMEM-load wait right after a store stalls on the store
        if (c_row) *reinterpret_cast<uint4*>(c_row + c_b * blk_bytes) = make_uint4(lo.x, lo.y, hi.x, hi.y);
        c_row = n_mt == c_mt ? c_row : row_ptr(n_mt);
        c_mt = n_mt;
        c_b = n_b;
      }
    } else if (codes_only && p.codes_c16) {
      // Channel-blocked codes only (the timed path).  A warp's units run in
      // increasing (mt, ch) order; the destination of this lane's row is
      // computed once per accumulator, and 16-channel block ch of that row lies
      // ch * H_out * W_out * 16 bytes further on.
      // FP4 nibbles: 32-channel blocks of 16 bytes per position, a chunk writes
      // one half of its block's row.
      const int pack = codes_pack(p);
      const int code_bytes = pack == 1 ? 4 : 16;  // bytes per position of a channel block
      const long long chunk_bytes = static_cast<long long>(p.Ho) * p.Wo * code_bytes;
      const int k0 = e.dst_c0 >> 4;
      uint8_t* const blk0 =
          p.q_out + (pack == 2 ? static_cast<long long>(e.n) * (p.C_out_total >> 5) * chunk_bytes
                               : (static_cast<long long>(e.n) * (p.C_out_total >> 4) + k0) * chunk_bytes);
      auto coff = [&](int ch) -> long long {
        if (pack != 2) return ch * chunk_bytes;
        const int k = k0 + ch;
        return (k >> 1) * chunk_bytes + (k & 1) * 8;
      };
      const int m_lane = quarter * 32 + lane;
      const int MT = p.MT;
      auto row_ptr = [&](int mt) -> uint8_t* {
        if (mt >= MT) return nullptr;
        bool valid;
        const int pos = epi_pos(p, e, mt * 128 + m_lane, valid);
        return valid ? blk0 + static_cast<long long>(pos) * code_bytes : nullptr;
      };
      auto step = [&](int& mt, int& ch) {
        ch += n_groups;
        while (ch >= nchunks) {
          ch -= nchunks;
          ++mt;
        }
      };
      auto col = [&](int mt, int ch) { return e.tbase + static_cast<uint32_t>(mt) * p.Npow2 + ch * 16; };
      uint32_t va[16], vb[16];
      int c_mt = 0, c_ch = wg - n_groups;
      step(c_mt, c_ch);
      // Units in pairs: both TMEM loads in flight together, one wait, then both
      // conversions in one stretch of code (independent work the scheduler can
      // interleave) and two stores.
      while (c_mt < MT) {
        int n_mt = c_mt, n_ch = c_ch;
        step(n_mt, n_ch);
        const bool two = n_mt < MT;
        tmem_ld16(col(c_mt, c_ch), va);
        if (two) tmem_ld16(col(n_mt, n_ch), vb);
        uint8_t* c_row = row_ptr(c_mt);
        uint8_t* n_row = two ? (n_mt == c_mt ? c_row : row_ptr(n_mt)) : nullptr;
        tmem_wait_ld();
        const uint4 w0 = epi_codes16_f16(va, e.m_req15, qmax2);
        const uint4 w1 = epi_codes16_f16(vb, e.m_req15, qmax2);
        if (c_row) store_codes16(c_row + coff(c_ch), w0, pack);
        if (n_row) store_codes16(n_row + coff(n_ch), w1, pack);
        if (!two) break;
        step(n_mt, n_ch);
        c_mt = n_mt;
        c_ch = n_ch;
      }
    } else {
      if ((p.Nblk & 31) == 0)
        epi_general_units<32>(p, e, stg, wg, n_groups, quarter, lane, qmax2);
      else
        epi_general_units<16>(p, e, stg, wg, n_groups, quarter, lane, qmax2);
    }
    // One arrival per warp: the warp's tensor-memory reads are complete (each
    // thread waited for its loads) and ordered before the arrive by the fence
    // and the warp barrier.
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(bars.acc_empty(racc.stage));
    racc.advance();
  }
}

}  // namespace

// One instance per operand type (F4: packed FP4 codes and block-scaled FP4 MMAs;
// else one code per byte or packed 2-bit codes, FP8 MMAs), so that each carries
// only its own MMA loops and epilogue paths (a smaller instruction footprint).
template <bool F4, bool LU>
__global__ void __launch_bounds__(kConvThreads, 1)
    pq_conv_tc_kernel(const __grid_constant__ ConvParams p, const __grid_constant__ CUtensorMap tmA) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  Bars bars{base + p.smem_bar_off, p.a_stages, p.b_resident ? 1 : p.b_stages};
  uint8_t* bar_block = gbase + p.smem_bar_off;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bar_block + 8 * bars.words());
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_block + 8 * bars.words() + 8);
  uint32_t* tap_a16 = reinterpret_cast<uint32_t*>(bar_block + 8 * bars.words() + 16);  // p.taps entries
  for (int t = threadIdx.x; t < p.taps; t += blockDim.x) tap_a16[t] = p.tap_a16[t];

  if (threadIdx.x == 0) {
    for (int s = 0; s < bars.A; ++s) {
      // TMA, or one arrival per copy warp
      mbar_init(bars.a_full(s), (p.a_tma && !p.a_unpack && !p.a_quant && !p.a_split) ? 1 : kLoadWarps);
      mbar_init(bars.a_empty(s), 1);
      if (p.a_unpack || p.a_quant || p.a_split) {
        mbar_init(bars.pk_full(s), 1);
        mbar_init(bars.pk_empty(s), kLoadWarps);
      }
    }
    for (int s = 0; s < bars.B; ++s) {
      mbar_init(bars.b_full(s), 1);
      mbar_init(bars.b_empty(s), 1);
    }
    for (int s = 0; s < p.acc_stages; ++s) {
      mbar_init(bars.acc_full(s), 1);
      mbar_init(bars.acc_empty(s),
                (p.a_tma && !p.a_unpack && !p.a_quant && !p.a_split) ? kEpiWarps + kLoadWarps : kEpiWarps);  // one per warp
    }
    mbar_init(bars.drain(), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), p.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  if (F4) {
    // Block scale factors of the FP4 MMAs: 32 columns of every lane set to 2^-4
    // (UE8M0 byte 123); warps 2-5 cover the four lane quarters.
    if (warp >= kFirstLoadWarp && warp < kFirstLoadWarp + 4) {
      const uint32_t t = tmem_base + (static_cast<uint32_t>((warp & 3) * 32) << 16) + p.sf_col;
#pragma unroll
      for (int c = 0; c < 32; c += 8) tmem_st8_fill(t + c, 0x7B7B7B7Bu);
      tmem_wait_st();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
  }

  // A programmatic dependent launch: the set-up above (barriers, tensor memory,
  // scale factors) overlaps the previous grid's last CTAs; every global read and
  // write below waits for that grid to complete (it may produce this launch's
  // inputs or read its outputs), so stream order holds.  Where the caller has
  // promised that the previous kernel writes neither the activations nor the
  // weights (pdl_early_loads), only the epilogue warps wait: the others' global
  // accesses are those loads (the producer's copies, the loader warps' reads),
  // and the quantiser and MMA warps work in shared and tensor memory.
  const bool third_epi = p.a_tma && !p.a_unpack && !p.a_quant && !p.a_split;  // warps 2-5 run the epilogue too
  const bool epi_warp = warp >= kFirstEpiWarp || (third_epi && warp >= kFirstLoadWarp);
  if (p.pdl && (epi_warp || !p.pdl_early_loads)) asm volatile("griddepcontrol.wait;" ::: "memory");
  // Let the next dependent launch on the stream start its CTAs as SMs free up, but
  // only once this CTA's own wait has returned: a launch that depends on this one
  // then starts only after the kernel before this one has completed, so an early
  // loader two launches on never reads what that kernel is still writing.  The
  // signal comes from a thread that waited (the first epilogue warp's lane 0).
  const int first_epi_warp = third_epi ? kFirstLoadWarp : kFirstEpiWarp;
  if (p.pdl && threadIdx.x == 32 * first_epi_warp) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int64_t it0 = static_cast<int64_t>(blockIdx.x) * p.items / gridDim.x;
  const int64_t it1 = static_cast<int64_t>(blockIdx.x + 1) * p.items / gridDim.x;
  const uint32_t a_base = base;
  const uint32_t b_base = base + p.smem_b_off;

  if (warp == 0) {
    if (lane == 0) {
      if (p.a_tma) prefetch_tmap(&tmA);
      producer_role(p, &tmA, bars, a_base, b_base, base + p.smem_pk_off, it0, it1,
                    WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_PRODUCER});
    }
    __syncwarp();
  } else if (warp == 1) {
    mma_role_dispatch<F4>(p, bars, a_base, b_base, tmem_base, tap_a16, it0, it1,
                      WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_MMA});
    __syncwarp();
  } else if (warp < kFirstEpiWarp && !p.a_tma) {
    loader_role(p, bars, a_base, it0, it1, WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_PRODUCER});
  } else if (warp < kFirstEpiWarp && p.a_quant) {
    quant_role<F4, LU>(p, bars, a_base, base + p.smem_pk_off, it0, it1,
               WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_PRODUCER});
  } else if (warp < kFirstEpiWarp && p.a_split) {
    split_role(p, bars, a_base, base + p.smem_pk_off, it0, it1,
               WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_PRODUCER});
  } else if (warp < kFirstEpiWarp && p.a_unpack) {
    unpack_role(p, bars, a_base, base + p.smem_pk_off, it0, it1,
                WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_PRODUCER});
  } else {
    // With TMA loading the activations as they are, the copy warps form a third
    // epilogue warpgroup.
    const bool third = p.a_tma && !p.a_unpack && !p.a_quant && !p.a_split;
    const int first = third ? kFirstLoadWarp : kFirstEpiWarp;

    epilogue_role<F4>(p, bars, tmem_base, gbase + p.smem_stage_off, first, third ? kEpiGroups + 1 : kEpiGroups, it0, it1,
                  WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_EPILOGUE});
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

int launch_conv_tc(const ConvParams& p, const CUtensorMap& tma_a, int grid, cudaStream_t stream) {
  // one instance per operand type (FP4 or byte codes) and quantiser form (learned
  // bounds or not); the attribute is set once per instance and device
  static int attr_set_for_device[4][64] = {{0}};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  const int need = static_cast<int>(p.smem_bytes) + 1024;
  const int f4 = p.codes_f4 ? 1 : 0, lu = p.q_lu ? 1 : 0;
  const int v = f4 * 2 + lu;
  const void* fn = f4 ? (lu ? reinterpret_cast<const void*>(pq_conv_tc_kernel<true, true>)
                            : reinterpret_cast<const void*>(pq_conv_tc_kernel<true, false>))
                      : (lu ? reinterpret_cast<const void*>(pq_conv_tc_kernel<false, true>)
                            : reinterpret_cast<const void*>(pq_conv_tc_kernel<false, false>));
  if (dev < 64 && attr_set_for_device[v][dev] < need) {
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem) != cudaSuccess) return -1;
    attr_set_for_device[v][dev] = kMaxSmem;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kConvThreads);
  cfg.dynamicSmemBytes = static_cast<size_t>(need);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.pdl ? 1 : 0;
  cudaError_t e;
  if (f4 && lu)
    e = cudaLaunchKernelEx(&cfg, pq_conv_tc_kernel<true, true>, p, tma_a);
  else if (f4)
    e = cudaLaunchKernelEx(&cfg, pq_conv_tc_kernel<true, false>, p, tma_a);
  else if (lu)
    e = cudaLaunchKernelEx(&cfg, pq_conv_tc_kernel<false, true>, p, tma_a);
  else
    e = cudaLaunchKernelEx(&cfg, pq_conv_tc_kernel<false, false>, p, tma_a);
  return e == cudaSuccess && cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // namespace pq
