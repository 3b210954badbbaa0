// Device-side building blocks for sm_103a: mbarriers with bounded waits, bulk and
// 16-byte asynchronous copies into shared memory, and the tcgen05 (5th-generation tensor core)
// operations used by the PalQuant kernels.  All inline PTX is written here; the
// kernels call these helpers only.
#pragma once

#include <cstdint>

#include "pq_internal.h"

namespace pq {

// ---------------------------------------------------------------- addresses
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ---------------------------------------------------------------- mbarriers
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\n"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      "selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// As mbar_try_wait, but the thread may stay suspended (without taking issue
// slots) for up to `suspend_ns` while the phase is incomplete; it resumes as
// soon as the phase completes.
__device__ __forceinline__ bool mbar_try_wait_suspend(uint32_t bar, uint32_t parity, uint32_t suspend_ns) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\n"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
      "selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(suspend_ns)
      : "memory");
  return ok != 0;
}

struct WaitCtx {
  volatile int* abort_flag;  // shared memory
  unsigned int* err;         // device error word (global)
  uint64_t limit_ns;
  unsigned int err_bits;     // bits recorded by this role on timeout
};

// Wait limits are kept in SM clock cycles: the cycle counter costs a few cycles
// to read, while %globaltimer reads cost on the order of a microsecond, which
// stalled every role of the pipeline when read on each blocking wait.  The
// conversion assumes 2.5 cycles per ns, above the highest SM clock (2.07 GHz),
// so a limit never ends earlier than asked.
__device__ __forceinline__ uint64_t limit_cycles(uint64_t limit_ns) { return limit_ns * 5u / 2u; }

// Suspension per try_wait of a blocking wait: waiting warps leave the issue
// slots to working ones, and the abort flag and the limit are still checked
// every few microseconds.
constexpr uint32_t kSuspendNs = 4000;

// Wait until the phase with the given parity of `bar` has completed.  Returns
// false (after recording PQ_ERR_TIMEOUT and raising the abort flag) when the
// wait exceeds ctx.limit_ns, or when another role of the CTA already aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, const WaitCtx& ctx) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_try_wait_suspend(bar, parity, kSuspendNs)) return true;
    if (*ctx.abort_flag) return false;
    if (static_cast<uint64_t>(clock64() - t0) > limit_cycles(ctx.limit_ns)) {
      atomicOr(ctx.err, PQ_ERR_TIMEOUT | ctx.err_bits);
      *ctx.abort_flag = 1;
      return false;
    }
  }
}

// Bounded wait that ignores the abort flag (teardown: drain what is in flight).
__device__ __forceinline__ bool mbar_wait_drain(uint32_t bar, uint32_t parity, uint64_t limit_ns, unsigned int* err) {
  const long long t0 = clock64();
  uint32_t n = 0;
  while (!mbar_try_wait(bar, parity)) {
    if ((++n & 63u) == 0 && static_cast<uint64_t>(clock64() - t0) > limit_cycles(limit_ns)) {
      atomicOr(err, PQ_ERR_TIMEOUT | PQ_ERR_TEARDOWN);
      return false;
    }
  }
  return true;
}

// ------------------------------------------------------------ async copies
// Order this thread's generic-proxy shared-memory accesses before later
// async-proxy (bulk copy / tensor core) accesses.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Tiled TMA loads (global -> shared), completion counted on `bar` in bytes.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const void* tmap, int c0, int c1, int c2, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const void* tmap, int c0, int c1, int c2, int c3,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], [%6];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void prefetch_tmap(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}

// Plain bulk copy of `bytes` (multiple of 16, both addresses 16-byte aligned).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
               : "memory");
}

// 16-byte asynchronous copy global -> shared through the LSU path; src_bytes = 0
// writes 16 zero bytes and reads nothing.
__device__ __forceinline__ void cp_async_16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(reinterpret_cast<uint64_t>(src)),
               "r"(src_bytes)
               : "memory");
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

// Wait until at most N of this thread's most recent copy groups are pending.
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// ------------------------------------------------------------ packed fp32
// Two IEEE fp32 round-to-nearest multiplies / adds in one instruction
// (sm_100+ f32x2 arithmetic); lane-wise identical to __fmul_rn / __fadd_rn.
__device__ __forceinline__ void mul2_rn(float a, float b, float m, float& x, float& y) {
  asm("{\n.reg .b64 s, t, r;\nmov.b64 s, {%2, %3};\nmov.b64 t, {%4, %4};\nmul.rn.f32x2 r, s, t;\nmov.b64 {%0, %1}, r;\n}"
      : "=f"(x), "=f"(y)
      : "f"(a), "f"(b), "f"(m));
}

__device__ __forceinline__ void add2_rn(float a, float b, float m, float& x, float& y) {
  asm("{\n.reg .b64 s, t, r;\nmov.b64 s, {%2, %3};\nmov.b64 t, {%4, %4};\nadd.rn.f32x2 r, s, t;\nmov.b64 {%0, %1}, r;\n}"
      : "=f"(x), "=f"(y)
      : "f"(a), "f"(b), "f"(m));
}

// x = fl(a * b) clamped to [0, 1] (saturation; NaN -> +0).
__device__ __forceinline__ float mul_sat(float a, float b) {
  float x;
  asm("mul.rn.sat.f32 %0, %1, %2;" : "=f"(x) : "f"(a), "f"(b));
  return x;
}

// (x, y) = (fl(a * m + c), fl(b * m + c)), each one rounding (packed fp32 FMA).
__device__ __forceinline__ void fma2_rn(float a, float b, float m, float c, float& x, float& y) {
  asm("{\n.reg .b64 s, t, u, r;\nmov.b64 s, {%2, %3};\nmov.b64 t, {%4, %4};\nmov.b64 u, {%5, %5};\n"
      "fma.rn.f32x2 r, s, t, u;\nmov.b64 {%0, %1}, r;\n}"
      : "=f"(x), "=f"(y)
      : "f"(a), "f"(b), "f"(m), "f"(c));
}

// Codes-only unit (the timed path): the codes clamp(rint(t), 0, Qp) of
// t = acc * m_req = raw * (m_req * 2^9), Qp = 2^b - 1, as
//   c = sat(raw * m_sat), m_sat = m_req * 2^9 / 2^b (a power-of-two scaling, so
//       c = clamp(t, 0, 2^b) / 2^b exactly; NaN -> 0);
//   r = c * 2^b + 1.5 * 2^23, one rounding half to even: the low 16 bits of r
//       hold k = rint(clamp(t, 0, 2^b)), in [0, 2^b];
//   code = min(k, Qp), two 16-bit halves per instruction.
// Clamping to [0, 2^b] before rounding and to Qp after it equals clamping the
// rounded value to [0, Qp] (integer bounds, monotone rounding).
// (v: 16 accumulator columns, or 16 of a larger array starting at OFF.)
template <int NV = 16, int OFF = 0>
__device__ __forceinline__ uint4 epi_codes16(const uint32_t (&v)[NV], float m_sat, float two_b, uint32_t qmax2) {
  static_assert(OFF + 16 <= NV, "16 columns of the array");
  uint32_t h[8];
#pragma unroll
  for (int j = 0; j < 16; j += 2) {
    const float c0 = mul_sat(__uint_as_float(v[OFF + j]), m_sat);
    const float c1 = mul_sat(__uint_as_float(v[OFF + j + 1]), m_sat);
    float r0, r1;
    fma2_rn(c0, c1, two_b, 12582912.0f, r0, r1);
    h[j >> 1] = __vimin_s16x2_relu(__byte_perm(__float_as_uint(r0), __float_as_uint(r1), 0x5410), qmax2);
  }
  uint4 w;
  w.x = __byte_perm(h[0], h[1], 0x6420);
  w.y = __byte_perm(h[2], h[3], 0x6420);
  w.z = __byte_perm(h[4], h[5], 0x6420);
  w.w = __byte_perm(h[6], h[7], 0x6420);
  return w;
}

// Requantised codes of 16 accumulator columns through the fp16 conversion, for
// output codes of at most 8 bits:
//   y = fl(raw * m_req 2^-15) with raw = acc * 2^-9, so y = fl(acc * m_req) * 2^-24
//       = t * 2^-24 exactly (power-of-two scalings commute with rounding; where y
//       would be an fp32 subnormal, |t| < 2^-102 and the code is 0 either way);
//   the fp16 conversion with .relu rounds y half to even onto the fp16 grid,
//       which below 2^-14 is the integers times 2^-24 (the subnormals), so the
//       16-bit pattern is rint(t) for t in [0, 1024], any larger t gives a larger
//       pattern (the positive encodings are ordered, up to +inf), and negative t
//       gives +0;
//   code = min(pattern, Qp) on both 16-bit halves in one instruction.
// This equals clamp(rint(t), 0, Qp): integer bounds, monotone rounding.  Per
// pair of values: one packed multiply, one packed conversion, one packed min,
// against two multiplies, a packed multiply-add and two integer steps in
// epi_codes16.  m_req15 = m_req * 2^-15 (the caller's exact scaling).
__device__ __forceinline__ uint32_t cvt_f16x2_relu(float hi, float lo) {
  uint32_t r;
  asm("cvt.rn.relu.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

template <int NV = 16, int OFF = 0>
__device__ __forceinline__ uint4 epi_codes16_f16(const uint32_t (&v)[NV], float m_req15, uint32_t qmax2) {
  static_assert(OFF + 16 <= NV, "16 columns of the array");
  uint32_t h[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    float y0, y1;
    mul2_rn(__uint_as_float(v[OFF + 2 * q]), __uint_as_float(v[OFF + 2 * q + 1]), m_req15, y0, y1);
    h[q] = __vimin_s16x2_relu(cvt_f16x2_relu(y1, y0), qmax2);
  }
  return make_uint4(__byte_perm(h[0], h[1], 0x6420), __byte_perm(h[2], h[3], 0x6420), __byte_perm(h[4], h[5], 0x6420),
                    __byte_perm(h[6], h[7], 0x6420));
}

// ------------------------------------------------------------- packed codes
// Sixteen 2-bit codes (one per byte of w, each <= 3) packed into one 32-bit word,
// code k at bits 2k: the product of a byte quadruple with 2^24 + 2^18 + 2^12 + 2^6
// moves byte k's value to bits 24 + 2k without carries (every partial product
// occupies its own bit pair), and the top byte holds the four codes.
__device__ __forceinline__ uint32_t pack2_quad(uint32_t x) { return (x * 0x01041040u) >> 24; }

__device__ __forceinline__ uint32_t pack2_word(uint4 w) {
  return pack2_quad(w.x) | (pack2_quad(w.y) << 8) | (pack2_quad(w.z) << 16) | (pack2_quad(w.w) << 24);
}

// Inverse: the 16 codes of a packed word, one per byte.  Even codes sit in the
// low two bits of the nibbles of (v & 0x33333333), odd codes in those of
// ((v >> 2) & 0x33333333); byte permutes interleave them back in order.
__device__ __forceinline__ uint4 unpack2_word(uint32_t v) {
  const uint32_t e = v & 0x33333333u, o = (v >> 2) & 0x33333333u;
  const uint32_t e_lo = e & 0x0F0F0F0Fu, e_hi = (e >> 4) & 0x0F0F0F0Fu;  // codes 0,4,8,12 | 2,6,10,14
  const uint32_t o_lo = o & 0x0F0F0F0Fu, o_hi = (o >> 4) & 0x0F0F0F0Fu;  // codes 1,5,9,13 | 3,7,11,15
  const uint32_t a = __byte_perm(e_lo, o_lo, 0x5140);  // 0 1 4 5
  const uint32_t b = __byte_perm(e_hi, o_hi, 0x5140);  // 2 3 6 7
  const uint32_t c = __byte_perm(e_lo, o_lo, 0x7362);  // 8 9 12 13
  const uint32_t d = __byte_perm(e_hi, o_hi, 0x7362);  // 10 11 14 15
  return make_uint4(__byte_perm(a, b, 0x5410), __byte_perm(a, b, 0x7632), __byte_perm(c, d, 0x5410),
                    __byte_perm(c, d, 0x7632));
}

// ------------------------------------------------------------------ tcgen05
// Shared-memory matrix descriptor, no swizzle, K-major: core matrices of
// 8 rows x 16 bytes; `lbo` = byte distance between core matrices adjacent in K,
// `sbo` = byte distance between core matrices adjacent in M/N.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((addr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;  // descriptor version for tcgen05
  return d;
}

// Instruction descriptor of kind::f8f6f4 with E4M3 A and B, fp32 accumulator,
// both operands K-major, M = 128.
__host__ __device__ constexpr uint32_t idesc_e4m3_f32(int M, int N) {
  return (1u << 4)                                 // D format: f32
         | (0u << 7) | (0u << 10)                  // A, B: E4M3
         | (static_cast<uint32_t>(N >> 3) << 17)   // N / 8
         | (static_cast<uint32_t>(M >> 4) << 24);  // M / 16
}

__device__ __forceinline__ void tc_mma_e4m3(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on `bar` once every tcgen05 operation this thread issued so far is done.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// Whole-warp forms: every lane of the (converged) warp executes the call with the
// same operands and one elected lane issues.  Keeping the issuing warp converged
// lets the compiler hold the warp-uniform descriptors in uniform registers, so an
// MMA costs a few instructions; a single-lane loop needs per-MMA register moves
// and loses issue slots to busy warps on the same scheduler.
__device__ __forceinline__ void tc_mma_e4m3_warp(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                                 uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p, e;\nelect.sync _|e, 0xffffffff;\nsetp.ne.b32 p, %4, 0;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// MT MMAs sharing one B operand and accumulate flag, one election for the group.
__device__ __forceinline__ void tc_mma2_e4m3_warp(uint32_t d0, uint32_t d1, uint64_t a0, uint64_t a1, uint64_t b_desc,
                                                  uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p, e;\nelect.sync _|e, 0xffffffff;\nsetp.ne.b32 p, %6, 0;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %2, %4, %5, p;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%1], %3, %4, %5, p;\n}" ::"r"(d0),
      "r"(d1), "l"(a0), "l"(a1), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tc_mma3_e4m3_warp(uint32_t d0, uint32_t d1, uint32_t d2, uint64_t a0, uint64_t a1,
                                                  uint64_t a2, uint64_t b_desc, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p, e;\nelect.sync _|e, 0xffffffff;\nsetp.ne.b32 p, %8, 0;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %3, %6, %7, p;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%1], %4, %6, %7, p;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%2], %5, %6, %7, p;\n}" ::"r"(d0),
      "r"(d1), "r"(d2), "l"(a0), "l"(a1), "l"(a2), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tc_mma4_e4m3_warp(uint32_t d0, uint32_t d1, uint32_t d2, uint32_t d3, uint64_t a0,
                                                  uint64_t a1, uint64_t a2, uint64_t a3, uint64_t b_desc,
                                                  uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p, e;\nelect.sync _|e, 0xffffffff;\nsetp.ne.b32 p, %10, 0;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %4, %8, %9, p;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%1], %5, %8, %9, p;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%2], %6, %8, %9, p;\n"
      "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%3], %7, %8, %9, p;\n}" ::"r"(d0),
      "r"(d1), "r"(d2), "r"(d3), "l"(a0), "l"(a1), "l"(a2), "l"(a3), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Instruction descriptor of kind::mxf4 (block-scaled, packed E2M1 A and B, two
// per byte), UE8M0 scale factors (scale-factor IDs 0), fp32 accumulator, both
// operands K-major, dense K = 64.
__host__ __device__ constexpr uint32_t idesc_mxf4_f32(int M, int N) {
  return (1u << 7) | (1u << 10)                    // A, B: E2M1
         | (static_cast<uint32_t>(N >> 3) << 17)   // N / 8
         | (1u << 23)                              // scale factors UE8M0
         | (static_cast<uint32_t>(M >> 4) << 24);  // M / 16
}

// Block-scaled FP4 forms of the whole-warp MMAs: `sfa`, `sfb` are the tensor-
// memory addresses of the A and B scale factors (one per 32 K elements).
__device__ __forceinline__ void tc_mma_f4_warp(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                               uint32_t sfa, uint32_t sfb, uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p, e;\nelect.sync _|e, 0xffffffff;\nsetp.ne.b32 p, %6, 0;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%0], %1, %2, %3, [%4], [%5], p;\n}" ::"r"(
          d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(sfa), "r"(sfb), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tc_mma2_f4_warp(uint32_t d0, uint32_t d1, uint64_t a0, uint64_t a1, uint64_t b_desc,
                                                uint32_t idesc, uint32_t sfa, uint32_t sfb, uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p, e;\nelect.sync _|e, 0xffffffff;\nsetp.ne.b32 p, %8, 0;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%0], %2, %4, %5, [%6], [%7], p;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%1], %3, %4, %5, [%6], [%7], p;\n}" ::"r"(d0),
      "r"(d1), "l"(a0), "l"(a1), "l"(b_desc), "r"(idesc), "r"(sfa), "r"(sfb), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tc_mma3_f4_warp(uint32_t d0, uint32_t d1, uint32_t d2, uint64_t a0, uint64_t a1,
                                                uint64_t a2, uint64_t b_desc, uint32_t idesc, uint32_t sfa, uint32_t sfb,
                                                uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p, e;\nelect.sync _|e, 0xffffffff;\nsetp.ne.b32 p, %10, 0;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%0], %3, %6, %7, [%8], [%9], p;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%1], %4, %6, %7, [%8], [%9], p;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%2], %5, %6, %7, [%8], [%9], p;\n}" ::"r"(d0),
      "r"(d1), "r"(d2), "l"(a0), "l"(a1), "l"(a2), "l"(b_desc), "r"(idesc), "r"(sfa), "r"(sfb), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tc_mma4_f4_warp(uint32_t d0, uint32_t d1, uint32_t d2, uint32_t d3, uint64_t a0,
                                                uint64_t a1, uint64_t a2, uint64_t a3, uint64_t b_desc, uint32_t idesc,
                                                uint32_t sfa, uint32_t sfb, uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p, e;\nelect.sync _|e, 0xffffffff;\nsetp.ne.b32 p, %12, 0;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%0], %4, %8, %9, [%10], [%11], p;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%1], %5, %8, %9, [%10], [%11], p;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%2], %6, %8, %9, [%10], [%11], p;\n"
      "@e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%3], %7, %8, %9, [%10], [%11], p;\n}" ::"r"(d0),
      "r"(d1), "r"(d2), "r"(d3), "l"(a0), "l"(a1), "l"(a2), "l"(a3), "l"(b_desc), "r"(idesc), "r"(sfa), "r"(sfb),
      "r"(accumulate)
      : "memory");
}

// Eight 32-bit columns of this warp's 32 tensor-memory lanes set to `v`.
__device__ __forceinline__ void tmem_st8_fill(uint32_t taddr, uint32_t v) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %1, %1, %1, %1, %1, %1, %1};" ::"r"(taddr), "r"(v)
               : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Sixteen 4-bit codes (one per byte of w, each <= 15) packed two to a byte, code
// k in the low nibble of byte k / 2 when k is even and the high nibble when odd.
__device__ __forceinline__ uint32_t pack4_pair(uint32_t a, uint32_t b) {
  const uint32_t ta = (a | (a >> 4)) & 0x00FF00FFu, tb = (b | (b >> 4)) & 0x00FF00FFu;
  return __byte_perm(ta, tb, 0x6420);
}
__device__ __forceinline__ uint2 pack4_word(uint4 w) { return make_uint2(pack4_pair(w.x, w.y), pack4_pair(w.z, w.w)); }

__device__ __forceinline__ void tc_commit_warp(uint32_t bar) {
  asm volatile(
      "{\n.reg .pred e;\nelect.sync _|e, 0xffffffff;\n"
      "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n}" ::"r"(bar)
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Whole-warp tensor-memory allocation; the base address is written to smem.
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// Each lane of the warp reads 16 consecutive 32-bit columns of its own TMEM lane.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
}

// Each lane of the warp reads 32 consecutive 32-bit columns of its own TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

}  // namespace pq
