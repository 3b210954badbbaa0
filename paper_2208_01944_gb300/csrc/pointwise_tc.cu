// PalQuant 1x1 group convolution with the codes-only epilogue on the sm_103a
// tensor cores: the memory-bound member of the layer family (a pointwise layer
// reads and writes one byte per code and does few operations per byte).
//
// What it computes (Sec. 4.1's B-bit group convolution with a 1x1 kernel, the
// Sec. 3.2 rescale, the Sec. 4.2 Eq. 6-8 output permutation and the Eq. 2
// requantisation):
//   q'[n, p, dst(g) Cout_g + co] = clamp(rint(m_req[g] sum_ci q[n, p, g Cin_g + ci] w[g, co, ci]), 0, Qp)
// with channel-blocked codes [N][C/16][H*W][16] in and out.
//
// How (persistent CTAs, two per SM where each fits half the SM, warp-specialised):
//  * A work item is (image, tile of up to 256 pixels, group), the group
//    fastest, and a CTA takes a contiguous range of items, so its loads walk
//    through consecutive bytes of each image.  With two CTAs per SM, a CTA of
//    the next launch starts loading as soon as one of the two finishes.
//  * Warp 0 (one lane) bulk-copies every group's packed weights into shared
//    memory once, then loads each item's input codes with one TMA box per
//    128-row accumulator (the group's 16-channel planes x 128 positions;
//    positions past the image are zero-filled and never stored) into a ring of
//    stages, several items ahead.
//  * Warp 1 (converged, one elected lane issuing) runs MT x Cin_g/32 MMAs per
//    item, tcgen05.mma kind::f8f6f4 with M = 128 and N = Cout_g on the codes read
//    in place as E4M3 subnormals (a code byte v <= 15 is the E4M3 encoding of
//    v 2^-9, so every sum is exact), into a tensor-memory accumulator stage.
//  * Two epilogue warpgroups take the accumulators in turn: tcgen05.ld (the
//    next 32 columns in flight while the current ones are converted), the
//    requantisation in registers (through the fp16 conversion, two values per
//    instruction), and the codes stored straight from registers
//    at the destination group's planes: the 32 lanes of a warp are 32
//    consecutive pixels of one 16-channel plane, 512 contiguous bytes.
//  * Every wait is bounded (failure detection): a wait that runs out records
//    PQ_ERR_TIMEOUT in the device error word, raises a CTA-wide abort flag, and
//    every role drains what it has in flight and returns.
#include <cuda_runtime.h>

#include "pq_device.cuh"
#include "pq_internal.h"

namespace pq {

namespace {

// Shared-memory barrier block (64-bit words): [0, S) a_full, [S, 2S) a_empty,
// then kMaxAccStages acc_full, kMaxAccStages acc_empty, w_full, drain,
// tmem_ready; after them the abort flag and the tensor-memory base.
struct PwBars {
  uint32_t base;
  int S;
  __device__ uint32_t a_full(int s) const { return base + 8u * s; }
  __device__ uint32_t a_empty(int s) const { return base + 8u * (S + s); }
  __device__ uint32_t acc_full(int s) const { return base + 8u * (2 * S + s); }
  __device__ uint32_t acc_empty(int s) const { return base + 8u * (2 * S + kMaxAccStages + s); }
  __device__ uint32_t w_full() const { return base + 8u * (2 * S + 2 * kMaxAccStages); }
  __device__ uint32_t drain() const { return base + 8u * (2 * S + 2 * kMaxAccStages + 1); }
  __device__ uint32_t tmem_ready() const { return base + 8u * (2 * S + 2 * kMaxAccStages + 2); }
  __device__ uint32_t words() const { return 2 * S + 2 * kMaxAccStages + 3; }
};

// Item index -> (image, tile, group); the group is fastest.  32-bit divisions
// (the planner keeps the item count below 2^31).
struct PwItem {
  int n, t, g;
};

__device__ __forceinline__ PwItem pw_item(const PwParams& p, int it) {
  PwItem r;
  const int q = it / p.G;
  r.g = it - q * p.G;
  r.n = q / p.tiles_per_img;
  r.t = q - r.n * p.tiles_per_img;
  return r;
}

// Wait taken by every lane of a converged warp; the lanes agree on the outcome.
__device__ __forceinline__ bool pw_warp_wait(uint32_t bar, uint32_t parity, const WaitCtx& ctx) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, ctx));
}

// Copy role (warp 0, lane 0).
__device__ __forceinline__ void pw_producer(const PwParams& p, const CUtensorMap* tm, const PwBars& bars,
                                            uint32_t a_base, uint32_t w_base, int it0, int it1, const WaitCtx& ctx) {
  // every group's weights, once for the whole launch, right after the first
  // item's codes (the weights come from L2, the codes from DRAM)
  bool w_issued = false;
  auto issue_weights = [&]() {
    mbar_arrive_expect_tx(bars.w_full(), p.w_bytes);
    for (uint32_t off = 0; off < p.w_bytes; off += 65536u)
      bulk_load(w_base + off, p.w_packed + off, min(65536u, p.w_bytes - off), bars.w_full());
    w_issued = true;
  };
  uint32_t stage = 0, phase = 0;
  int issued = 0;
  for (int it = it0; it < it1; ++it) {
    if (issued == 1 && !w_issued) issue_weights();
    const PwItem c = pw_item(p, it);
    if (!mbar_wait(bars.a_empty(stage), phase ^ 1u, ctx)) break;
    const uint32_t full = bars.a_full(stage);
    mbar_arrive_expect_tx(full, p.a_tx_bytes);
    const uint32_t dst = a_base + stage * p.a_stage_bytes;
    // x counts 8-byte elements, two per 16-byte position: always even, so every
    // box starts on a 16-byte boundary
    const int x0 = 2 * c.t * p.T;
    for (int mt = 0; mt < p.MT; ++mt)
      tma_load_3d(dst + static_cast<uint32_t>(mt * p.nch) * 2048u, tm, x0 + 256 * mt, c.g * p.nch, c.n, full);
    ++issued;
    if (++stage == static_cast<uint32_t>(p.a_stages)) {
      stage = 0;
      phase ^= 1u;
    }
  }
  if (!w_issued) issue_weights();  // one item, or none after an abort: the drain below finds them
  // Drain: the last min(stages, issued) loads and the weights may still be in flight.
  for (int k = max(0, issued - p.a_stages); k < issued; ++k)
    mbar_wait_drain(bars.a_full(k % p.a_stages), static_cast<uint32_t>((k / p.a_stages) & 1), ctx.limit_ns, ctx.err);
  mbar_wait_drain(bars.w_full(), 0, ctx.limit_ns, ctx.err);
}

// Tensor-core issue role (warp 1, converged; one elected lane issues).  The
// issue loop is compiled for the accumulators per item (MT) and the K steps
// (KS, 0: a runtime loop), so that an item's MMAs go out back to back: the
// warp shares its scheduler with busy epilogue warps, and every
// instruction per MMA delays the next item's accumulator.
template <int MT, int KS>
__device__ __forceinline__ void pw_mma(const PwParams& p, const PwBars& bars, uint32_t a_base, uint32_t w_base,
                                       uint32_t tmem_base, int it0, int it1, const WaitCtx& ctx) {
  const uint32_t idesc = idesc_e4m3_f32(128, p.Cout_g);
  // A: K-major planes of 128 positions x 16 bytes (core matrices 8 rows apart by
  // 128 bytes, 16-byte K chunks a plane, 2048 bytes, apart).  B: the group's
  // weights, per 16-channel chunk Cout_g rows of 16 bytes.
  const uint64_t a_desc0 = smem_desc(a_base, 2048u, 128u);
  const uint64_t b_desc0 = smem_desc(w_base, static_cast<uint32_t>(p.Cout_g) * 16u, 128u);
  const uint64_t a_hi = a_desc0 & 0xFFFFFFFF00000000ull, b_hi = b_desc0 & 0xFFFFFFFF00000000ull;
  const uint32_t a_lo0 = static_cast<uint32_t>(a_desc0), b_lo0 = static_cast<uint32_t>(b_desc0);
  // offsets in 16-byte units
  const uint32_t a_stage16 = p.a_stage_bytes >> 4;
  const uint32_t a_mt16 = static_cast<uint32_t>(p.nch) * 128u;           // next accumulator's box
  const uint32_t b_g16 = static_cast<uint32_t>(p.Cin_g * p.Cout_g) >> 4;  // next group's weights
  const uint32_t b_ks16 = 2u * static_cast<uint32_t>(p.Cout_g);           // one K step: two 16-channel chunks
  const uint32_t npow2 = static_cast<uint32_t>(p.Npow2);
  const uint32_t acc_cols = static_cast<uint32_t>(MT) * npow2;
  const int ksteps = KS > 0 ? KS : p.ksteps;
  const int G = p.G, AS = p.acc_stages, S = p.a_stages;
  bool ok = pw_warp_wait(bars.w_full(), 0, ctx);
  uint32_t stage = 0, phase = 0, as = 0, as_phase = 0;
  int g = it0 % G;
  for (int it = it0; ok && it < it1; ++it) {
    if (!pw_warp_wait(bars.acc_empty(as), as_phase ^ 1u, ctx)) break;
    tc_fence_after();
    if (!pw_warp_wait(bars.a_full(stage), phase, ctx)) break;
    tc_fence_after();
    const uint32_t d0 = tmem_base + as * acc_cols;
    const uint32_t a_lo = a_lo0 + stage * a_stage16;
    const uint32_t b_lo = b_lo0 + static_cast<uint32_t>(g) * b_g16;
    if constexpr (KS > 0) {
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        const uint64_t bdesc = b_hi | (b_lo + static_cast<uint32_t>(ks) * b_ks16);
        const uint32_t ak = a_lo + static_cast<uint32_t>(ks) * 256u;
        if constexpr (MT == 2)
          tc_mma2_e4m3_warp(d0, d0 + npow2, a_hi | ak, a_hi | (ak + a_mt16), bdesc, idesc, ks > 0 ? 1u : 0u);
        else
          tc_mma_e4m3_warp(d0, a_hi | ak, bdesc, idesc, ks > 0 ? 1u : 0u);
      }
    } else {
      for (int mt = 0; mt < MT; ++mt)
        for (int ks = 0; ks < ksteps; ++ks)
          tc_mma_e4m3_warp(d0 + static_cast<uint32_t>(mt) * npow2,
                           a_hi | (a_lo + static_cast<uint32_t>(mt) * a_mt16 + static_cast<uint32_t>(ks) * 256u),
                           b_hi | (b_lo + static_cast<uint32_t>(ks) * b_ks16), idesc, ks > 0 ? 1u : 0u);
    }
    tc_commit_warp(bars.a_empty(stage));
    tc_commit_warp(bars.acc_full(as));
    if (++stage == static_cast<uint32_t>(S)) {
      stage = 0;
      phase ^= 1u;
    }
    if (++as == static_cast<uint32_t>(AS)) {
      as = 0;
      as_phase ^= 1u;
    }
    if (++g == G) g = 0;
  }
  // Drain: wait until every MMA this warp issued has completed.
  tc_commit_warp(bars.drain());
  mbar_wait_drain(bars.drain(), 0, ctx.limit_ns, ctx.err);
}

__device__ __forceinline__ void pw_mma_dispatch(const PwParams& p, const PwBars& bars, uint32_t a_base,
                                                uint32_t w_base, uint32_t tmem_base, int it0, int it1,
                                                const WaitCtx& ctx) {
#define PQ_PW_CASE(M, K) \
  if (p.MT == M && p.ksteps == K) return pw_mma<M, K>(p, bars, a_base, w_base, tmem_base, it0, it1, ctx);
  PQ_PW_CASE(2, 1) PQ_PW_CASE(2, 2) PQ_PW_CASE(2, 3) PQ_PW_CASE(2, 4)
  PQ_PW_CASE(1, 1) PQ_PW_CASE(1, 2) PQ_PW_CASE(1, 3) PQ_PW_CASE(1, 4)
#undef PQ_PW_CASE
  if (p.MT == 2) return pw_mma<2, 0>(p, bars, a_base, w_base, tmem_base, it0, it1, ctx);
  return pw_mma<1, 0>(p, bars, a_base, w_base, tmem_base, it0, it1, ctx);
}

// Epilogue role (warps 2-9: two warpgroups).  The tasks are the items'
// accumulators in order (item i, accumulator mt is task i MT + mt), and
// warpgroup w takes tasks w, w + 2, ... (only warpgroup 0 when the CTA's tensor
// memory holds a single accumulator): with two accumulators per item, the two
// warpgroups share each item.  Warp w reads
// tensor-memory lanes 32 (w % 4) .. 32 (w % 4) + 31, the accumulator rows that
// are consecutive pixels of the tile, and takes the accumulator 32 columns at a
// time (two 16-channel planes of codes), the next 32 columns loading while the
// current ones are converted and stored.
__device__ __forceinline__ void pw_epilogue(const PwParams& p, const PwBars& bars, const uint32_t* tmem_slot,
                                            int it0, int it1, const WaitCtx& ctx) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the tensor memory is allocated by warp 1 once the SM has it free
  if (!pw_warp_wait(bars.tmem_ready(), 0, ctx)) return;
  tc_fence_after();
  const uint32_t tmem_base = *reinterpret_cast<const volatile uint32_t*>(tmem_slot);
  const int eg = (warp - kPwFirstEpiWarp) >> 2;
  const int quarter = warp & 3;
  const uint32_t qmax2 = p.qmax2;
  const int nco = p.Cout_g >> 4;   // 16-channel planes of codes per item
  const int npc = (nco + 1) >> 1;  // 32-column pieces (the planner's Npow2 >= 32 holds the last one)
  const int MT = p.MT, AS = p.acc_stages, T = p.T, HW = p.HW, Npow2 = p.Npow2;
  const int plane = HW * 16;  // bytes of one 16-channel plane of an image (the planner keeps HW <= 2^22)
  const uint32_t lane_base = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16);
  // Every use of an accumulator stage must go to the same warpgroups: a wait on
  // a stage's phase parity cannot tell its next phase from the one after, so a
  // warpgroup may only wait for a stage's next use after it has taken the
  // previous one.  Task k = i MT + mt uses stage i % AS, so with n_egs
  // warpgroups taking tasks k % n_egs, AS MT must be a multiple of n_egs.
  const int n_egs = min(kPwEpiGroups, AS * MT);
  if (eg >= n_egs) return;
  for (int k = eg;; k += n_egs) {
    const int i = MT == 2 ? (k >> 1) : k;
    const int mt = k - i * MT;
    if (it0 + i >= it1) break;
    const PwItem c = pw_item(p, it0 + i);
    const int as = i % AS;
    const uint32_t use = static_cast<uint32_t>(i / AS);
    if (!pw_warp_wait(bars.acc_full(as), use & 1u, ctx)) break;
    tc_fence_after();
    const int p0 = c.t * T;
    const int tv = min(T, HW - p0);         // rows of this tile inside the image
    const int r0 = mt * 128 + quarter * 32;  // this warp's first row
    if (r0 < tv) {                           // warp-uniform
      const float m_req15 = p.m_req15[c.g];
      const int m = r0 + lane;
      uint8_t* const row = m < tv ? p.q_out +
                                        (static_cast<long long>(c.n) * p.C16_out +
                                         static_cast<long long>(p.dst_group[c.g]) * nco) *
                                            static_cast<long long>(plane) +
                                        static_cast<long long>(p0 + m) * 16
                                  : nullptr;
      const uint32_t tcol = lane_base + static_cast<uint32_t>((as * MT + mt) * Npow2);
      auto store = [&](int j, uint4 lo, uint4 hi) {  // piece j: planes 2j and 2j + 1
        if (row == nullptr) return;
        *reinterpret_cast<uint4*>(row + (2 * j) * plane) = lo;
        if (2 * j + 1 < nco) *reinterpret_cast<uint4*>(row + (2 * j + 1) * plane) = hi;
      };
      // every TMEM-load wait comes before a store (a wait right after a store
      // stalls on the store)
      uint32_t va[32], vb[32];
      tmem_ld32(tcol, va);
      tmem_wait_ld();
      for (int j = 0; j < npc; j += 2) {
        const bool nb = j + 1 < npc, na = j + 2 < npc;
        if (nb) tmem_ld32(tcol + static_cast<uint32_t>(j + 1) * 32u, vb);
        const uint4 w0 = epi_codes16_f16<32, 0>(va, m_req15, qmax2);
        const uint4 w1 = epi_codes16_f16<32, 16>(va, m_req15, qmax2);
        if (nb) tmem_wait_ld();
        store(j, w0, w1);
        if (na) tmem_ld32(tcol + static_cast<uint32_t>(j + 2) * 32u, va);
        if (!nb) break;
        const uint4 w2 = epi_codes16_f16<32, 0>(vb, m_req15, qmax2);
        const uint4 w3 = epi_codes16_f16<32, 16>(vb, m_req15, qmax2);
        if (na) tmem_wait_ld();
        store(j + 1, w2, w3);
      }
    }
    // One arrival per warp and task: its tensor-memory reads are complete (each
    // lane waited for its loads) and ordered before the arrive by the fence and
    // the warp barrier.
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(bars.acc_empty(as));
  }
}

}  // namespace

// At most 102 registers a thread, so that two CTAs fit an SM's register file.
__global__ void __launch_bounds__(kPwThreads, 2)
    pq_pointwise_tc_kernel(const __grid_constant__ PwParams p, const __grid_constant__ CUtensorMap tmA) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  PwBars bars{base + p.smem_bar_off, p.a_stages};
  uint8_t* bar_block = gbase + p.smem_bar_off;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bar_block + 8 * bars.words());
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_block + 8 * bars.words() + 8);
  if (threadIdx.x == 0) {
    for (int s = 0; s < p.a_stages; ++s) {
      mbar_init(bars.a_full(s), 1);   // the producer's expect_tx arrival; the TMA completes the bytes
      mbar_init(bars.a_empty(s), 1);  // the MMA warp's commit
    }
    for (int s = 0; s < p.acc_stages; ++s) {
      mbar_init(bars.acc_full(s), 1);   // the MMA warp's commit
      mbar_init(bars.acc_empty(s), 4 * p.MT);  // one arrival per warp and accumulator
    }
    mbar_init(bars.w_full(), 1);
    mbar_init(bars.drain(), 1);
    mbar_init(bars.tmem_ready(), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  // A programmatic dependent launch: the set-up above overlaps the previous
  // grid's last CTAs; every global access below waits for that grid, except,
  // under the caller's inputs-ready promise, the loads of the codes and weights
  // (warps 0 and 1 then start at once; the epilogue, which makes every store,
  // always waits).  The dependent launch after this one is let in only once
  // this CTA's own wait has returned, from a thread that waited.
  //
  // The planner keeps a CTA under half an SM's shared memory, so a CTA of the
  // next launch can share the SM with this launch's CTA while that one finishes.
  // The tensor memory is therefore allocated by the MMA warp after the set-up,
  // not before it: tcgen05.alloc waits until the other CTA has released its
  // columns, while this CTA's producer already loads its first items.
  const bool epi_warp = warp >= kPwFirstEpiWarp;
  if (p.pdl && (epi_warp || !p.pdl_early_loads)) asm volatile("griddepcontrol.wait;" ::: "memory");
  if (p.pdl && threadIdx.x == 32 * kPwFirstEpiWarp) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  // a contiguous range of items, sizes differing by at most one (32-bit arithmetic)
  const int per = p.items / static_cast<int>(gridDim.x), rem = p.items - per * static_cast<int>(gridDim.x);
  const int bx = static_cast<int>(blockIdx.x);
  const int it0 = bx * per + min(bx, rem);
  const int it1 = it0 + per + (bx < rem ? 1 : 0);
  const uint32_t a_base = base;
  const uint32_t w_base = base + p.smem_w_off;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&tmA);
      pw_producer(p, &tmA, bars, a_base, w_base, it0, it1, WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_PRODUCER});
    }
    __syncwarp();
  } else if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), p.tmem_cols);
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(bars.tmem_ready());
    tc_fence_after();
    const uint32_t tmem_base = *reinterpret_cast<volatile uint32_t*>(tmem_slot);
    pw_mma_dispatch(p, bars, a_base, w_base, tmem_base, it0, it1,
                    WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_MMA});
    __syncwarp();
  } else {
    pw_epilogue(p, bars, tmem_slot, it0, it1, WaitCtx{abort_flag, p.err, p.wait_limit_ns, PQ_ERR_EPILOGUE});
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(*reinterpret_cast<volatile uint32_t*>(tmem_slot), p.tmem_cols);
  }
}

int launch_pointwise_tc(const PwParams& p, const CUtensorMap& tma_a, int grid, cudaStream_t stream) {
  static int attr_set_for_device[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  const int need = static_cast<int>(p.smem_bytes) + 1024;  // + the 1024-byte alignment of the base
  if (dev >= 64 || attr_set_for_device[dev] < need) {
    if (cudaFuncSetAttribute(pq_pointwise_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem) !=
        cudaSuccess)
      return -1;
    if (dev < 64) attr_set_for_device[dev] = kMaxSmem;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kPwThreads);
  cfg.dynamicSmemBytes = static_cast<size_t>(need);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.pdl ? 1 : 0;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, pq_pointwise_tc_kernel, p, tma_a);
  return e == cudaSuccess && cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // namespace pq
