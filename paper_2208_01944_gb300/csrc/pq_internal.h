// Internal structures shared by the host code and the kernels of libpalquant.so.
// Not part of the public ABI (see include/palquant.h).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

// Bits of the device error word.
#define PQ_ERR_TIMEOUT 1u     // a bounded wait ran out
#define PQ_ERR_PRODUCER 2u    // ... in the copy (TMA) role
#define PQ_ERR_MMA 4u         // ... in the tensor-core issue role
#define PQ_ERR_EPILOGUE 8u    // ... in the epilogue role
#define PQ_ERR_TEARDOWN 16u   // ... while draining in-flight copies / MMAs
#define PQ_ERR_SELFTEST 32u   // ... in the watchdog self-test kernel

namespace pq {

constexpr int kMaxG = 64;
constexpr int kMaxTaps = 49;
constexpr int kMaxPhases = 4;
constexpr int kMaxAccStages = 4;                   // TMEM accumulator ring depth at most
constexpr int kEpiGroups = 2;                      // epilogue warpgroups, splitting the output columns
constexpr int kEpiWarps = 4 * kEpiGroups;
constexpr int kLoadWarps = 4;                      // activation-operand copy warps
constexpr int kFirstLoadWarp = 2;
constexpr int kFirstEpiWarp = kFirstLoadWarp + kLoadWarps;
constexpr int kConvThreads = 32 * (kFirstEpiWarp + kEpiWarps);  // warp 0 weights, 1 MMA, 2-5 loads, 6-13 epilogue
constexpr int kMaxSmem = 227 * 1024;

enum ConvMode : int { kModeFlat = 0, kModeRows = 1 };

// Everything the tensor-core conv kernel needs; filled by the host planner.
struct ConvParams {
  // ---- geometry
  int mode;               // kModeFlat or kModeRows
  int N, Ho, Wo;          // output batch / spatial size
  int64_t P_out;          // N * Ho * Wo
  int G, Cin_g, Cout_g;
  int Ht;                 // output rows per tile (rows mode)
  int Wh;                 // positions per tile row in the operand planes
  int Hd, Wd;             // plane rows / columns loaded per phase
  int h_off;              // first plane row = phase row oh0 + h_off
  int w_coord;            // first plane column = phase column w_coord
  int H, W, stride;       // input geometry
  int C_in_total;         // G * Cin_g (bytes per input pixel)
  int img_pix;            // H * W (flat mode tiles stay inside one image)
  int codes_c16;          // 1: input and output codes in the channel-blocked layout [N][C/16][H][W][16]
  int codes_p2;           // 1: channel-blocked 2-bit codes packed four to a byte ([N][C/16][H][W][4 B])
  // 1: 2-bit codes as packed FP4 (E2M1) nibbles, [N][C/32][H][W][16 B], read by the
  // block-scaled FP4 MMA; one 16-byte chunk then holds 32 channels.
  int codes_f4;
  int chunk_shift;        // log2(channels per 16-byte chunk): 4, or 5 for FP4 codes
  uint32_t sf_col;        // FP4: first TMEM column of the (uniform) block scale factors
  // Packed activations come by TMA into a staging ring and the copy warps unpack
  // them into the operand stages (a_unpack = 1): staged rows of pk_box_w 32-bit
  // words starting pk_off words left of the tile's first position.
  int a_unpack;
  // Stride 2 (a_split = 1): TMA stages the input window of the tile (2 Hd rows x
  // 2 Wd positions x nch chunks, every stride phase interleaved) into the staging
  // ring and the copy warps split it into the phase planes of the operand stage.
  int a_split;
  // Quantise-on-load (a_quant = 1): the input is fp32 NHWC; TMA stages boxes of 32
  // channels x all positions of a stage (128-byte rows, 128-byte swizzle) into the
  // staging ring and the copy warps quantise them into the operand stage:
  // code = min(rint(sat(x * q_inv_sat[g]) * 2^b), Qp), q_inv_sat = fl(1/s) / 2^b.
  int a_quant;
  float q_inv_sat[kMaxG];
  float q_two_b;
  uint32_t q_qmax2;  // Qp in both 16-bit halves
  // q_lu = 1: learned bounds l < u per group instead (Eq. 2 as trained):
  // code = rint(sat((x - l) * q_inv_r[g]) * Qp), q_inv_r = fl(1 / fl(u - l)),
  // q_neg_l = -l, q_qp = Qp; out-of-image positions are NaN-filled (code 0).
  // pdl = 1: launched as a programmatic dependent of the previous kernel on the
  // stream: a CTA's set-up (barriers, tensor memory) may run while that kernel's
  // last CTAs still run; every global access waits for it to complete (stream
  // order holds), and every CTA lets the next such launch start early.
  int pdl;
  // pdl_early_loads = 1 (the caller's PQ_LAYER_INPUTS_READY): only the epilogue
  // warps (every global store) wait for the previous kernel; loads, quantisation
  // and MMAs may start before it completes.
  int pdl_early_loads;
  int q_lu;
  float q_neg_l[kMaxG];
  float q_inv_r[kMaxG];
  float q_qp;
  uint32_t q_box_bytes;  // staging bytes per 32-channel box (a multiple of 1024: the 128B swizzle atom)
  int pk_box_w, pk_off;
  uint32_t pk_stage_bytes, smem_pk_off;
  int a_tma;              // 1: warp 0 loads the A operand with one TMA per stage (channel-blocked codes, stride 1)
  uint32_t a_tx_bytes;    // bytes one A stage receives (TMA mode)
  // Activation copy addressing (cp.async mode), in bytes: code (n, ih, iw, c0 + 16 j) of the
  // K block starting at channel c0 sits at n*ld_img + ih*ld_row + iw*ld_pix + ld_c0(c0) + j*ld_chunk,
  // with ld_c0(c0) = c0 * ld_c0_mul / 16.
  int64_t ld_img, ld_row, ld_pix, ld_chunk, ld_c0_mul;
  int phase_a[kMaxPhases], phase_b[kMaxPhases];  // stride phase (row, column) of each plane set
  uint32_t nch_magic;     // ceil(2^32 / nch): e / nch = umulhi(e, nch_magic) for small e
  uint32_t wh_magic;      // ceil(2^32 / Wh) (rows mode): m / Wh = umulhi(m, wh_magic) for m < 2^24
  int tiles_per_img;      // rows mode
  int64_t tiles;          // tiles per (group, n-block) unit
  int64_t items;          // tiles * G * NB
  int NB, Nblk, Npow2;    // output-channel blocks, MMA N, TMEM column stride per accumulator
  int MT;                 // 128-row accumulators per tile
  int KC, n_kb, nch;      // channels per K block, K blocks, 16-byte chunks per K block
  int taps, nph;          // kh*kw, stride phases
  int flat_box;           // pixels per flat-mode tile (= MT * 128)
  int tap_phase[kMaxTaps];
  int tap_off[kMaxTaps];  // position offset of each tap in the plane
  uint32_t tap_a16[kMaxTaps];  // stage-relative start of each tap's A operand, in 16-byte units
  uint32_t lbo_a;         // byte stride between 16-byte K chunks of the A planes
  uint32_t a_mt16;        // 16-byte units between the A operands of consecutive accumulators:
                          // 128 (one plane of positions), or nch * 128 (flat TMA: a box region each)
  uint32_t a_phase_bytes, a_stage_bytes;
  int a_stages;
  int b_resident;         // 1: the whole unit's weights stay in shared memory
  uint32_t b_slice_bytes; // one (K block, tap) slice: KC * Nblk bytes
  uint32_t b_unit_bytes;  // taps * Cin_g * Nblk
  uint32_t lbo_b;         // Nblk * 16
  int b_stages;           // ring stages when streamed
  int acc_stages;         // TMEM accumulator buffers (ring of 1..kMaxAccStages)
  uint32_t tmem_cols;
  uint32_t smem_b_off, smem_stage_off, smem_bar_off, smem_bytes;
  uint32_t stage_q_pitch, stage_f_pitch, stage_warp_bytes;
  // ---- operands
  const uint8_t* q_in;    // activation codes, NHWC
  const uint8_t* w_packed;
  // ---- epilogue
  int C_out_total;        // G * Cout_g
  float m_out[kMaxG];     // as given: y = (float)acc * m_out
  float m_req[kMaxG];     // as given: applied to the shortcut sum
  float m_out512[kMaxG];  // m_out * 2^9 (exact): applied to the raw accumulator, which holds acc * 2^-9
  float m_req512[kMaxG];  // m_req * 2^9 (exact)
  int dst_group[kMaxG];
  int src_group[kMaxG];  // input group read by conv group g (identity, or the module's Eq. 8 permutation)
  int channel_shuffle;    // 1: destination channel co*G + g (per-channel scatter)
  int relu;
  int qmax_out;
  const float* shortcut;
  int32_t* acc_out;
  float* y_out;
  uint8_t* q_out;
  // ---- failure detection
  unsigned int* err;
  uint64_t wait_limit_ns;
};

// The pointwise kernel (1x1, stride 1, pad 0 layers, channel-blocked codes in
// and codes only out); filled by the host planner.  A work item is (image,
// pixel tile, group), the group fastest.
constexpr int kPwEpiGroups = 2;                             // epilogue warpgroups, taking accumulators in turn
constexpr int kPwFirstEpiWarp = 2;                          // warp 0 loads, warp 1 issues the MMAs
constexpr int kPwThreads = 32 * (kPwFirstEpiWarp + 4 * kPwEpiGroups);
constexpr int kPwMaxStages = 8;
constexpr int kPwHalfSmem = 113 * 1024;                     // dynamic shared memory of one of two CTAs on an SM

struct PwParams {
  int N, HW, G, Cin_g, Cout_g;
  int T;                  // pixels per tile (at most 256; the last tile of an image may be shorter)
  int MT;                 // 128-row accumulators per tile (1 or 2)
  int tiles_per_img;
  int items;              // N * tiles_per_img * G
  int nch;                // Cin_g / 16: 16-channel planes of an item's input
  int ksteps;             // Cin_g / 32: MMAs per accumulator
  int Npow2;              // tensor-memory columns per accumulator
  int a_stages, acc_stages;
  int ctas_per_sm;        // 2: two CTAs share an SM (each at most half its shared memory and tensor memory)
  uint32_t a_stage_bytes; // MT * nch * 2048: per accumulator one TMA box of nch planes x 128 positions
  uint32_t a_tx_bytes;    // bytes a stage receives (whole boxes, out-of-image rows zero-filled)
  uint32_t w_bytes;       // every group's packed weights, G * Cout_g * Cin_g
  uint32_t smem_w_off, smem_bar_off, smem_bytes, tmem_cols;
  int C16_out;            // 16-channel planes of an output image: G * Cout_g / 16
  uint32_t qmax2;         // Qp_out in both 16-bit halves
  float m_req15[kMaxG];   // m_req * 2^-15, applied to the raw accumulator acc * 2^-9 (fl(acc m_req) * 2^-24)
  int dst_group[kMaxG];
  const uint8_t* w_packed;
  uint8_t* q_out;
  unsigned int* err;
  uint64_t wait_limit_ns;
  int pdl, pdl_early_loads;
};

// Host-side launch helpers implemented in the .cu files.
int launch_conv_tc(const ConvParams& p, const CUtensorMap& tma_a, int grid, cudaStream_t stream);
int launch_pointwise_tc(const PwParams& p, const CUtensorMap& tma_a, int grid, cudaStream_t stream);
int launch_bitsplit_act(const uint8_t* q, uint8_t* xs, int64_t N, int64_t HW, int C, int Ga, int B, int c16,
                        cudaStream_t stream);
// pack: 0 one code per byte [N][C/16][HW][16]; 1 four 2-bit codes per byte
// [N][C/16][HW][4 B]; 2 two 4-bit codes per byte [N][C/32][HW][16 B].
int launch_quantize_c16(const float* x, uint8_t* q, int64_t N, int64_t HW, int G, int Cg, int bits, const float* inv_s,
                        int pack, cudaStream_t stream, const float* l = nullptr, const float* u = nullptr);
// l non-NULL: learned bounds l, u per group instead of inv_s (see quantize.cu).
int launch_quantize(const float* x, uint8_t* q, int64_t P, int G, int Cg, int bits, const float* inv_s,
                    cudaStream_t stream, const float* l = nullptr, const float* u = nullptr);
int launch_act_sum(const float* x, int64_t P, int G, int Cg, double* partial, int nblocks, cudaStream_t stream);
int launch_act_sum_finish(const double* partial, int nblocks, int G, double* sums, cudaStream_t stream);
int launch_watchdog_selftest(unsigned int* err, uint64_t limit_ns, cudaStream_t stream);
unsigned int* device_error_word();  // device address of the current device's error word

}  // namespace pq
