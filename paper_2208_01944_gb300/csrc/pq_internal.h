// Internal structures shared by the host code and the kernels of libpalquant.so.
// Not part of the public ABI (see include/palquant.h).
#pragma once

#include <cuda.h>
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
constexpr int kConvThreads = 192;  // warp 0: copies, warp 1: MMA issue + TMEM, warps 2-5: epilogue
constexpr int kEpiWarps = 4;
constexpr int kMaxSmem = 227 * 1024;

enum ConvMode : int { kModeFlat = 0, kModeRows = 1 };

// Tensor maps of the activation operand, one per stride phase.
struct TensorMaps {
  CUtensorMap a[kMaxPhases];
};

// Everything the tensor-core conv kernel needs; filled by the host planner.
struct ConvParams {
  // ---- geometry
  int mode;               // kModeFlat or kModeRows
  int N, Ho, Wo;          // output batch / spatial size
  int64_t P_out;          // N * Ho * Wo
  int G, Cin_g, Cout_g;
  int Ht;                 // output rows per tile (rows mode)
  int Wh;                 // positions per tile row in the operand planes
  int Hd, Wd;             // box rows / columns loaded per phase
  int h_off;              // TMA row coordinate = oh0 + h_off (phase rows)
  int w_coord;            // TMA column coordinate (phase columns)
  int tiles_per_img;      // rows mode
  int64_t tiles;          // tiles per (group, n-block) unit
  int64_t items;          // tiles * G * NB
  int NB, Nblk, Npow2;    // output-channel blocks, MMA N, TMEM column stride per accumulator
  int MT;                 // 128-row accumulators per tile
  int KC, n_kb, nch;      // channels per K block, K blocks, 16-byte chunks per K block
  int taps, nph;          // kh*kw, stride phases
  int flat_box;           // pixels per flat-mode box (= MT * 128)
  int tap_phase[kMaxTaps];
  int tap_off[kMaxTaps];  // position offset of each tap in the plane
  uint32_t lbo_a;         // byte stride between 16-byte K chunks of the A planes
  uint32_t a_phase_bytes, a_stage_bytes, a_tx_bytes;
  int a_stages;
  int b_resident;         // 1: the whole unit's weights stay in shared memory
  uint32_t b_slice_bytes; // one (K block, tap) slice: KC * Nblk bytes
  uint32_t b_unit_bytes;  // taps * Cin_g * Nblk
  uint32_t lbo_b;         // Nblk * 16
  int b_stages;           // ring stages when streamed
  int acc_stages;         // TMEM accumulator buffers
  uint32_t tmem_cols;
  uint32_t smem_b_off, smem_stage_off, smem_bar_off, smem_bytes;
  uint32_t stage_q_pitch, stage_f_pitch, stage_warp_bytes;
  // ---- operands
  const uint8_t* w_packed;
  // ---- epilogue
  int C_out_total;        // G * Cout_g
  float m_out[kMaxG];
  float m_req[kMaxG];
  int dst_group[kMaxG];
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

// Host-side launch helpers implemented in the .cu files.
int launch_conv_tc(const ConvParams& p, const TensorMaps& tm, int grid, cudaStream_t stream);
int launch_quantize(const float* x, uint8_t* q, int64_t P, int G, int Cg, int bits, const float* inv_s,
                    cudaStream_t stream);
int launch_act_sum(const float* x, int64_t P, int G, int Cg, double* partial, int nblocks, cudaStream_t stream);
int launch_act_sum_finish(const double* partial, int nblocks, int G, double* sums, cudaStream_t stream);
int launch_watchdog_selftest(unsigned int* err, uint64_t limit_ns, cudaStream_t stream);
unsigned int* device_error_word();  // device address of the current device's error word

}  // namespace pq
