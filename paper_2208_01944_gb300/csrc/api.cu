// Host side of libpalquant.so: argument validation, the tiling planner of the
// tensor-core convolution, weight quantisation and packing, tensor-map encoding,
// launches and error reporting.  Every entry point of include/palquant.h is
// defined here.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <vector>

#include "palquant.h"
#include "pq_internal.h"

using pq::ConvParams;

namespace {

constexpr uint64_t kDefaultWaitLimitNs = 2000000000ull;
std::atomic<uint64_t> g_wait_limit_ns{kDefaultWaitLimitNs};

constexpr int kActSumBlocks = 256;

int64_t out_dim(int64_t in, int k, int s, int p) { return (in + 2 * p - k) / s + 1; }

int floor_div(int a, int b) { return (a >= 0) ? a / b : -((-a + b - 1) / b); }

int pos_mod(int a, int b) { return ((a % b) + b) % b; }

uint32_t round_up(uint64_t v, uint64_t a) { return static_cast<uint32_t>((v + a - 1) / a * a); }

int next_pow2(int v) {
  int p = 1;
  while (p < v) p <<= 1;
  return p;
}

// FP8 E4M3 encoding (1 sign bit, 4 exponent bits with bias 7, 3 mantissa bits)
// of an integer |v| <= 15: |v| in [2^e, 2^(e+1)) has exponent field e + 7 and
// mantissa (|v| / 2^e - 1) * 8, exact for |v| < 16.
uint8_t e4m3_of_int(int v) {
  if (v == 0) return 0;
  const uint8_t sign = v < 0 ? 0x80 : 0x00;
  const int a = v < 0 ? -v : v;
  int e = 0;
  while ((2 << e) <= a) ++e;
  const int mant = ((a << 3) >> e) & 7;
  return static_cast<uint8_t>(sign | ((e + 7) << 3) | mant);
}

// Inverse of e4m3_of_int for bytes it produces (normal numbers >= 1 in magnitude).
int int_of_e4m3(uint8_t b) {
  if ((b & 0x7F) == 0) return 0;
  const int e = ((b >> 3) & 15) - 7;
  const int mant = b & 7;
  const int a = ((8 + mant) << e) >> 3;
  return (b & 0x80) ? -a : a;
}

bool valid_shuffle(int G, const pq_shuffle& s, int* dst_group) {
  if (s.kind == 0 || s.kind == 2) {
    for (int g = 0; g < G; ++g) dst_group[g] = g;
  } else if (s.kind == 1) {
    for (int g = 0; g < G; ++g) dst_group[g] = pos_mod(g + s.shift, G);
  } else if (s.kind == 3) {
    if (s.perm == nullptr) return false;
    for (int g = 0; g < G; ++g) dst_group[g] = s.perm[g];
  } else {
    return false;
  }
  std::vector<int> seen(G, 0);
  for (int g = 0; g < G; ++g) {
    if (dst_group[g] < 0 || dst_group[g] >= G || seen[dst_group[g]]) return false;
    seen[dst_group[g]] = 1;
  }
  return true;
}

pq_status validate_desc(const pq_layer_desc* d) {
  if (d == nullptr) return PQ_EINVAL;
  if (d->N < 0 || d->H < 1 || d->W < 1 || d->G < 1 || d->Cin_g < 1 || d->Cout_g < 1) return PQ_EINVAL;
  if (d->kh < 1 || d->kw < 1 || d->stride < 1 || d->pad < 0) return PQ_EINVAL;
  if (d->bits_a < 1 || d->bits_a > 8 || d->bits_w < 2 || d->bits_w > 8 || d->bits_out < 1 || d->bits_out > 8)
    return PQ_EINVAL;
  if (d->relu != 0 && d->relu != 1) return PQ_EINVAL;
  if ((d->flags & ~PQ_LAYER_INPUTS_READY) != 0) return PQ_EINVAL;
  if (d->wslices < 0 || d->wslices > 8) return PQ_EINVAL;
  if (d->code_format != PQ_CODES_INT8 && d->code_format != PQ_CODES_E4M3 && d->code_format != PQ_CODES_C16 &&
      d->code_format != PQ_CODES_C16P2 && d->code_format != PQ_CODES_C32F4)
    return PQ_EINVAL;
  if (out_dim(d->H, d->kh, d->stride, d->pad) < 1 || out_dim(d->W, d->kw, d->stride, d->pad) < 1) return PQ_EINVAL;
  if (d->G > pq::kMaxG) return PQ_EUNSUPPORTED;
  return PQ_OK;
}

// Weight slices per input channel and tap (pq_layer_desc.wslices; 0 means 1).
int wslices_of(const pq_layer_desc* d) { return d->wslices > 1 ? d->wslices : 1; }

// Taps of the weight operand: kh kw positions, each with R weight slices.
int weight_taps(const pq_layer_desc* d) { return d->kh * d->kw * wslices_of(d); }

int device_sm_count() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return sms;
}

// ---------------------------------------------------------------------------
// Planner: how the tensor-core kernel tiles a layer.  Pure host arithmetic.
// ---------------------------------------------------------------------------
struct Phase {
  int a, b;
};

// quant_in: the layer's input is fp32 NHWC activations, quantised on load (the
// copy warps quantise TMA-staged 32-channel fp32 boxes into the operand stages).
// direct_out: the call reads no shortcut and writes channel-blocked codes only
// (no int32 or fp32 outputs), which the epilogue stores straight from registers,
// so the plan reserves no per-warp staging for it.  shortcut: the call reads a
// shortcut (two staging buffers per warp).
pq_status plan_conv(const pq_layer_desc* d, ConvParams* P, pq_conv_plan* pub, std::vector<Phase>* phases_out,
                    bool quant_in = false, bool direct_out = false, bool shortcut = false) {
  // Epilogue staging per warp: 32 rows of up to 32 fp32/int32 values (128 bytes,
  // chunk-swizzled), twice with a shortcut (the next unit's rows are fetched into
  // the second buffer), or 32 rows of 16 code bytes at a pitch of 80 bytes (an odd
  // number of 16-byte bank groups).
  const uint32_t warp_stage = direct_out ? 0u : (shortcut ? 2u : 1u) * 32u * 128u;
  pq_status st = validate_desc(d);
  if (st != PQ_OK) return st;
  pq_conv_plan plan;
  std::memset(&plan, 0, sizeof(plan));
  ConvParams p;
  std::memset(&p, 0, sizeof(p));
  const int Ho = static_cast<int>(out_dim(d->H, d->kh, d->stride, d->pad));
  const int Wo = static_cast<int>(out_dim(d->W, d->kw, d->stride, d->pad));
  // R weight slices per kernel position: R consecutive taps with the same
  // activation offset (the operand's tap t = position * R + slice)
  const int R = wslices_of(d);
  const int taps = d->kh * d->kw * R;
  const int qa = (1 << d->bits_a) - 1;
  const int qw = 1 << (d->bits_w - 1);
  // Coverage of the tensor-core kernel.
  const bool p2 = d->code_format == PQ_CODES_C16P2;
  const bool f4 = d->code_format == PQ_CODES_C32F4;
  const bool c16 = d->code_format == PQ_CODES_C16 || p2 || f4;  // channel-blocked (bytes or packed)
  // FP4 nibbles: 16-byte chunks of 32 channels and 64 channels per MMA K step;
  // E2M1 holds the codes v / 2 for v <= 3 and the weights -4..4.
  const int cpb = f4 ? 2 : 1;  // channels per byte of the operands
  const bool f4_ok = !f4 || (d->bits_a <= 2 && d->bits_out <= 2 && d->bits_w <= 3 && d->Cin_g % 64 == 0 &&
                             d->Cout_g % 32 == 0);
  // Packed 2-bit codes: 2-bit input and output codes, stride 1, and 16-byte aligned
  // rows (1x1: image planes) for the TMA loads of the packed tile.
  const bool flat_shape = d->kh == 1 && d->kw == 1 && d->stride == 1 && d->pad == 0;
  const bool p2_ok = !p2 || (d->bits_a <= 2 && d->bits_out <= 2 && d->stride == 1 &&
                             (flat_shape ? (static_cast<int64_t>(d->H) * d->W) % 4 == 0 : d->W % 4 == 0));
  // Quantise-on-load: stride 1, codes out one per byte (NHWC or channel-blocked) or
  // as FP4 nibbles, K blocks of one MMA K step (32 channels, 64 for FP4: two 32-channel
  // fp32 boxes), fp32 rows of 16-byte multiples for the TMA.
  const bool quant_ok = !quant_in || (d->stride == 1 && !p2 && (d->G * d->Cin_g) % 4 == 0);
  bool ok = (d->code_format == PQ_CODES_INT8 || c16) && p2_ok && f4_ok && quant_ok && d->bits_a <= 4 && d->bits_w <= 4 && d->stride <= 2 &&
            d->pad < std::max(d->kh, d->kw) && d->Cin_g % 32 == 0 && d->Cout_g % 16 == 0 && taps <= pq::kMaxTaps &&
            static_cast<int64_t>(taps) * d->Cin_g * qa * qw < (1LL << 24);
  if (!ok) {
    if (pub) *pub = plan;
    return PQ_EUNSUPPORTED;
  }
  p.N = d->N;
  p.Ho = Ho;
  p.Wo = Wo;
  p.P_out = static_cast<int64_t>(d->N) * Ho * Wo;
  p.G = d->G;
  p.Cin_g = d->Cin_g;
  p.Cout_g = d->Cout_g;
  p.taps = taps;
  // Output-channel blocks: N of one MMA is at most 256 and a multiple of 16.
  // FP4 keeps N <= 128 so that two accumulators and the 32 scale-factor columns
  // fit the 512 TMEM columns.
  const int n_max = f4 ? 128 : 256;
  int NB = (d->Cout_g + n_max - 1) / n_max;
  while (d->Cout_g % NB != 0 || (d->Cout_g / NB) % 16 != 0) ++NB;
  p.NB = NB;
  p.Nblk = d->Cout_g / NB;
  p.Npow2 = next_pow2(p.Nblk);
  const bool flat = d->kh == 1 && d->kw == 1 && d->stride == 1 && d->pad == 0;
  p.mode = flat ? pq::kModeFlat : pq::kModeRows;
  const int s = d->stride;
  // Rows-mode geometry in phase coordinates.
  const int rmin = floor_div(-d->pad, s), rmax = floor_div(d->kh - 1 - d->pad, s);
  const int cmin = floor_div(-d->pad, s), cmax = floor_div(d->kw - 1 - d->pad, s);
  const int Wh = flat ? 0 : Wo + cmax - cmin;
  // Stride phases used by the taps, and each tap's (phase, offset).
  std::vector<Phase> phases;
  int off_max = 0;
  if (!flat) {
    for (int i = 0; i < d->kh; ++i) {
      for (int j = 0; j < d->kw; ++j) {
        const int a = pos_mod(i - d->pad, s), b = pos_mod(j - d->pad, s);
        int idx = -1;
        for (size_t q = 0; q < phases.size(); ++q)
          if (phases[q].a == a && phases[q].b == b) idx = static_cast<int>(q);
        if (idx < 0) {
          phases.push_back({a, b});
          idx = static_cast<int>(phases.size()) - 1;
        }
        for (int r = 0; r < R; ++r) {
          const int t = (i * d->kw + j) * R + r;
          p.tap_phase[t] = idx;
          p.tap_off[t] = (floor_div(i - d->pad, s) - rmin) * Wh + (floor_div(j - d->pad, s) - cmin);
          off_max = std::max(off_max, p.tap_off[t]);
        }
      }
    }
  } else {
    phases.push_back({0, 0});
    for (int r = 0; r < R; ++r) {
      p.tap_phase[r] = 0;
      p.tap_off[r] = 0;
    }
  }
  p.nph = static_cast<int>(phases.size());
  // Tile shape: MT accumulators of 128 rows; rows mode packs Ht whole output
  // rows of pitch Wh into them.
  //
  // Choice of MT: a work item costs a fixed overhead (waits, commits, the
  // epilogue's per-item set-up) plus the larger of its MMA time and its
  // epilogue time, so few large items beat many small ones even at some cost in
  // padded rows.  Model (per SM, measured): an M=128, K=32 FP8 MMA (or K=64 FP4
  // MMA, the same 32 bytes of K) takes max(32 + N/4, N/2) cycles (shared-memory
  // operand reads at 128 B per cycle, tensor rate); the epilogue splits a tile
  // into units of 16 accumulator columns (32 for FP4 codes) x 128 rows, each
  // taking one warpgroup about 430 ns (550 ns for a 32-column FP4 unit), and its
  // warpgroups (three when TMA loads the operand, else two) take the units in
  // turn, so an uneven split costs a whole unit; an item costs 500 ns of
  // overhead; a unit's weights stay in shared memory up to 160 KB (beside two
  // operand stages: a 3x3 layer of 128x28x28 with 4 groups of 128 ran 63 -> 45 us
  // once its 147 KB stayed),
  // larger ones are streamed again for every item, from L2 at about 40 B/ns per SM
  // when all SMs stream.  Double-buffered accumulators come first.
  const double ns_per_clk = 1.0 / 1.9;
  const double mma_ns = std::max(32.0 + p.Npow2 / 4.0, p.Npow2 / 2.0) * ns_per_clk;
  const double mma_acc_ns = static_cast<double>(p.taps) * (d->Cin_g / (32 * cpb)) * mma_ns;  // one accumulator
  // (quantise-on-load keeps the copy warps busy converting: two epilogue groups)
  const bool tma_operand = !quant_in && c16 && d->stride == 1 && (flat || Wh <= 128);
  const int epi_groups = tma_operand ? pq::kEpiGroups + 1 : pq::kEpiGroups;
  const int unit_cols = (f4 && p.Nblk % 32 == 0) ? 32 : 16;
  const int units_per_acc = p.Nblk / unit_cols;
  const double unit_ns = unit_cols == 32 ? 550.0 : 430.0;
  const double w_unit_bytes = static_cast<double>(p.taps) * d->Cin_g * p.Nblk / cpb;
  const double w_stream_ns = w_unit_bytes > 160.0 * 1024.0 ? w_unit_bytes / 40.0 : 0.0;  // per item
  const int tmem_avail = f4 ? 512 - 32 : 512;  // FP4: 32 columns hold the scale factors
  int best_mt = 0, best_ht = 0, best_tpi = 0, best_acc = 0;
  double best_cost = 0.0;
  for (int MT : {1, 2, 3, 4}) {
    // flat tiles: up to two accumulators (by TMA, one 128-position box each); the
    // packed 2-bit path stages one box
    if (flat && (MT > 2 || ((p2 || quant_in) && MT > 1))) continue;
    int acc_stages = (2 * MT * p.Npow2 <= tmem_avail) ? 2 : ((MT * p.Npow2 <= tmem_avail) ? 1 : 0);
    if (acc_stages == 0) continue;
    int ht = 0, tpi = 0;
    if (flat) {
      tpi = static_cast<int>((static_cast<int64_t>(Ho) * Wo + MT * 128 - 1) / (MT * 128));
    } else {
      const int ht_max = (MT * 128) / Wh;
      if (ht_max < 1) continue;
      tpi = (Ho + ht_max - 1) / ht_max;
      ht = (Ho + tpi - 1) / tpi;
    }
    if (quant_in) {
      // two fp32 staging stages (128 bytes per position) and two operand stages
      // (32 bytes per position) must fit beside the weights (resident, or a
      // two-slice ring) and the epilogue staging
      const uint64_t npos = flat ? 128u : static_cast<uint64_t>(ht + rmax - rmin) * Wh;
      const uint64_t w_unit = static_cast<uint64_t>(taps) * d->Cin_g * p.Nblk / cpb;
      const uint64_t w_min = 2ull * round_up(32ull * p.Nblk, 1024);  // a streamed ring at least (resident when it fits)
      const uint64_t need = 2ull * (cpb * round_up(npos * 128, 1024) + round_up(npos * 32, 1024)) + w_min +
                            static_cast<uint64_t>(pq::kEpiWarps) * warp_stage + 1024;
      if (need > pq::kMaxSmem - 1024) continue;
    }
    const int units = MT * units_per_acc;
    const double epi_ns = ((units + epi_groups - 1) / epi_groups) * unit_ns;
    const double mma_side = std::max(MT * mma_acc_ns, w_stream_ns);
    const double cost = static_cast<double>(tpi) * (500.0 + std::max(mma_side, epi_ns));
    const bool better = best_mt == 0 || acc_stages > best_acc || (acc_stages == best_acc && cost < best_cost * 0.98);
    if (better) {
      best_mt = MT;
      best_ht = ht;
      best_tpi = tpi;
      best_acc = acc_stages;
      best_cost = cost;
    }
  }
  if (best_mt == 0) {
    if (pub) *pub = plan;
    return PQ_EUNSUPPORTED;
  }
  p.MT = best_mt;
  p.acc_stages = best_acc;
  if (flat) {
    // Flat tiles are runs of flat_box pixels inside one image.
    p.flat_box = p.MT * 128;
    p.tiles_per_img = static_cast<int>((static_cast<int64_t>(Ho) * Wo + p.flat_box - 1) / p.flat_box);
    p.tiles = static_cast<int64_t>(d->N) * p.tiles_per_img;
    p.Ht = 0;
    p.Wh = 0;
    p.Hd = 0;
    p.Wd = 0;
  } else {
    p.Ht = best_ht;
    p.tiles_per_img = best_tpi;
    p.tiles = static_cast<int64_t>(d->N) * best_tpi;
    p.Wh = Wh;
    p.Wd = Wh;
    p.Hd = p.Ht + rmax - rmin;
    p.h_off = rmin;
    p.w_coord = cmin;
    if (p.Wd > 256 || p.Hd > 256) {
      if (pub) *pub = plan;
      return PQ_EUNSUPPORTED;
    }
    for (size_t i = 0; i < phases.size(); ++i) {
      p.phase_a[i] = phases[i].a;
      p.phase_b[i] = phases[i].b;
    }
  }
  p.items = p.tiles * d->G * NB;
  // K blocks, weights residency and pipeline depth under the shared-memory budget.
  const uint32_t budget = pq::kMaxSmem - 1024;
  auto a_stage_bytes = [&](int KC, uint32_t* phase_bytes, uint32_t* lbo) -> uint32_t {
    const int nch = KC / (16 * cpb);
    if (flat && c16 && !p2) {
      // TMA: per accumulator a region of nch planes of 128 positions (one box)
      *lbo = 128u * 16u;
      *phase_bytes = static_cast<uint32_t>(p.MT) * nch * 2048u;
      return round_up(*phase_bytes, 1024);
    }
    if (flat) {
      const uint32_t plane = static_cast<uint32_t>(p.flat_box) * 16u;
      *phase_bytes = round_up(static_cast<uint64_t>(nch) * plane, 128);
      *lbo = plane;
      return round_up(*phase_bytes, 1024);
    }
    const uint32_t plane = static_cast<uint32_t>(p.Hd) * p.Wd * 16u;
    *phase_bytes = round_up(static_cast<uint64_t>(nch) * plane, 128);
    *lbo = plane;
    const uint64_t overrun = static_cast<uint64_t>(p.nph - 1) * (*phase_bytes) + static_cast<uint64_t>(nch - 1) * plane +
                             16ull * (p.MT * 128 + off_max);
    return round_up(std::max<uint64_t>(static_cast<uint64_t>(p.nph) * (*phase_bytes), overrun), 1024);
  };
  const uint32_t q_pitch = 80;
  const uint32_t f_pitch = 128;
  // Staging for every warp that runs the epilogue: the copy warps join it only when
  // TMA loads the activation operand as it is (not unpacked, not quantised).
  const bool third_group =
      !quant_in && !p2 && c16 && d->stride == 1 && (flat ? p.flat_box <= 256 : p.Wd <= 128);
  const uint32_t stage_total =
      direct_out ? 0u : warp_stage * (third_group ? pq::kEpiWarps + pq::kLoadWarps : pq::kEpiWarps);
  const uint32_t bar_bytes = 1024;  // barriers, abort flag, TMEM slot (generous)
  const uint64_t unit_bytes = static_cast<uint64_t>(taps) * d->Cin_g * p.Nblk / cpb;
  // Packed codes: a staging stage per operand stage holding the TMA box of 32-bit
  // words (rows start at the tile's first position rounded down to a multiple of
  // 4, the TMA's 16-byte alignment of the innermost coordinate).
  const int pk_x0 = flat ? 0 : static_cast<int>(std::floor(p.w_coord / 4.0)) * 4;
  const int pk_off = flat ? 0 : p.w_coord - pk_x0;
  const int pk_box_w = flat ? p.flat_box : static_cast<int>(round_up(static_cast<uint64_t>(p.Wd + pk_off), 4));
  if (p2 && pk_box_w > 256) {
    if (pub) *pub = plan;
    return PQ_EUNSUPPORTED;
  }
  // Stride 2 with channel-blocked codes: TMA stages the tile's input window (2 Hd
  // rows x 2 Wd positions, both stride phases) and the copy warps split it into
  // the phase planes; the window's row of 2 Wd positions is one box row of
  // 4 Wd 8-byte elements (at most 256).
  const bool split = c16 && !p2 && !quant_in && d->stride == 2 && !flat && 4 * p.Wd <= 256 && 2 * p.Hd <= 256;
  auto pk_stage_bytes = [&](int KC) -> uint32_t {
    if (split) return round_up(static_cast<uint64_t>(KC / (16 * cpb)) * (2 * p.Hd) * (2 * p.Wd) * 16, 1024);
    if (quant_in) {
      // KC/32 fp32 boxes of 32 channels x all positions of the stage (128-byte rows),
      // each starting on a 1024-byte swizzle atom
      const uint64_t npos = flat ? static_cast<uint64_t>(p.flat_box) : static_cast<uint64_t>(p.Hd) * p.Wd;
      return static_cast<uint32_t>(KC / 32) * round_up(npos * 128, 1024);
    }
    if (!p2) return 0;
    const uint64_t rows = flat ? 1 : p.Hd;
    return round_up(static_cast<uint64_t>(pk_box_w) * rows * (KC / 16) * 4, 1024);
  };
  // Largest K block (input channels per pipeline stage) that fits with the whole
  // unit's weights resident, else the largest with a ring of (K block, tap)
  // slices (the stage-4 conv1 of the network: 84 -> 72 us with conv1 + down once
  // its 147 KB of weights stayed at half the K block).
  bool found = false, resident = false;
  int KC = d->Cin_g, a_stages = 0, b_stages = 0;
  uint32_t stage_bytes = 0, phase_bytes = 0, lbo = 0;
  // K blocks of {8, 4, 3, 2, 1} MMA K steps (32 channels each, 64 for FP4): the
  // MMA issue loop is compiled for these K-step counts.
  for (int pass = 1; pass >= 0 && !found; --pass)
  for (int kc1 : {256, 128, 96, 64, 32}) {
    if (found) break;
    // at most four 32-channel fp32 boxes per stage, a power-of-two chunk count
    if (quant_in && (kc1 > 128 || kc1 == 96)) continue;
    const int kc = kc1 * cpb;
    if (d->Cin_g % kc != 0) continue;
    uint32_t sb, pb, l;
    sb = a_stage_bytes(kc, &pb, &l);
    if (sb > 64u * 1024u) continue;
    for (int res = pass; res >= pass && !found; --res) {
      if (res && unit_bytes > 160u * 1024u) continue;
      const uint64_t slice = static_cast<uint64_t>(kc) * p.Nblk / cpb;
      if (!res && slice > 32u * 1024u) continue;
      for (int na = 4; na >= 2 && !found; --na) {
        for (int nb = (res ? 1 : 4); nb >= (res ? 1 : 2) && !found; --nb) {
          const uint64_t bb = res ? round_up(unit_bytes, 1024) : round_up(nb * slice, 1024);
          if (bb + stage_total + bar_bytes + static_cast<uint64_t>(na) * (sb + pk_stage_bytes(kc)) <= budget) {
            found = true;
            resident = res != 0;
            KC = kc;
            a_stages = na;
            b_stages = nb;
            stage_bytes = sb;
            phase_bytes = pb;
            lbo = l;
          }
        }
      }
    }
  }
  if (!found) {
    if (pub) *pub = plan;
    return PQ_EUNSUPPORTED;
  }
  const uint32_t b_bytes =
      resident ? round_up(unit_bytes, 1024) : round_up(static_cast<uint64_t>(b_stages) * KC * p.Nblk / cpb, 1024);
  p.KC = KC;
  p.nch = KC / (16 * cpb);
  p.nch_magic = static_cast<uint32_t>(((1ull << 32) + p.nch - 1) / p.nch);
  p.wh_magic = p.Wh > 0 ? static_cast<uint32_t>(((1ull << 32) + p.Wh - 1) / p.Wh) : 0u;
  p.H = d->H;
  p.W = d->W;
  p.stride = d->stride;
  p.C_in_total = d->G * d->Cin_g;
  p.img_pix = d->H * d->W;
  p.codes_c16 = c16 ? 1 : 0;
  p.codes_p2 = p2 ? 1 : 0;
  p.codes_f4 = f4 ? 1 : 0;
  p.chunk_shift = f4 ? 5 : 4;
  p.a_unpack = p2 ? 1 : 0;
  p.a_split = split ? 1 : 0;
  p.a_quant = quant_in ? 1 : 0;
  p.q_box_bytes = quant_in ? round_up(static_cast<uint64_t>(flat ? p.flat_box : p.Hd * p.Wd) * 128, 1024) : 0;
  p.pk_box_w = pk_box_w;
  p.pk_off = pk_off;
  p.pk_stage_bytes = pk_stage_bytes(KC);
  // The A operand comes by TMA when every plane row is one contiguous run in
  // global memory (channel-blocked codes, stride 1, rows of at most 128
  // positions), or through the staging ring (packed codes, quantise-on-load,
  // stride-2 windows).
  p.a_tma = (quant_in || p2 || split || (c16 && d->stride == 1 && (flat ? p.flat_box <= 256 : p.Wd <= 128))) ? 1 : 0;
  p.a_mt16 = (flat && c16 && !p2 && !quant_in) ? static_cast<uint32_t>(p.nch) * 128u : 128u;
  p.a_tx_bytes = quant_in ? static_cast<uint32_t>(KC) * 4u * (flat ? p.flat_box : p.Hd * p.Wd)
                 : p2 ? static_cast<uint32_t>(p.nch) * pk_box_w * (flat ? 1 : p.Hd) * 4u
                 : split ? static_cast<uint32_t>(p.nch) * (2 * p.Hd) * (2 * p.Wd) * 16u
                 : flat ? static_cast<uint32_t>(p.nch) * p.flat_box * 16u
                        : static_cast<uint32_t>(p.nph) * p.nch * p.Hd * p.Wd * 16u;
  {
    const int64_t C = p.C_in_total, H = d->H, W = d->W;
    if (c16) {
      // 16-byte chunks of 16 channels (32 for FP4 nibbles)
      p.ld_pix = 16;
      p.ld_row = W * 16;
      p.ld_chunk = H * W * 16;
      p.ld_img = (C / (16 * cpb)) * H * W * 16;
      p.ld_c0_mul = H * W * 16 / cpb;  // channel block c0/16 (c0/32) starts that many chunks in
    } else {
      p.ld_pix = C;
      p.ld_row = W * C;
      p.ld_chunk = 16;
      p.ld_img = H * W * C;
      p.ld_c0_mul = 16;  // channel c0 is c0 bytes in
    }
  }
  p.n_kb = d->Cin_g / KC;
  p.lbo_a = lbo;
  p.a_phase_bytes = phase_bytes;
  for (int t = 0; t < taps; ++t)
    p.tap_a16[t] = (static_cast<uint32_t>(p.tap_phase[t]) * phase_bytes + static_cast<uint32_t>(p.tap_off[t]) * 16u) >> 4;
  p.a_stage_bytes = stage_bytes;
  p.a_stages = a_stages;
  p.b_resident = resident ? 1 : 0;
  p.b_slice_bytes = static_cast<uint32_t>(KC) * p.Nblk / cpb;
  p.b_unit_bytes = static_cast<uint32_t>(unit_bytes);
  p.lbo_b = static_cast<uint32_t>(p.Nblk) * 16u;
  p.b_stages = resident ? 1 : b_stages;
  {
    const int acc_cols = std::max(32, p.acc_stages * p.MT * p.Npow2);
    p.sf_col = static_cast<uint32_t>(round_up(acc_cols, 32));  // FP4 scale factors after the accumulators
    p.tmem_cols = static_cast<uint32_t>(next_pow2(f4 ? static_cast<int>(p.sf_col) + 32 : acc_cols));
  }
  p.smem_b_off = static_cast<uint32_t>(a_stages) * stage_bytes;
  p.smem_stage_off = p.smem_b_off + b_bytes;
  p.smem_pk_off = p.smem_stage_off + stage_total;  // packed staging ring (a_stages x pk_stage_bytes)
  p.smem_bar_off = p.smem_pk_off + static_cast<uint32_t>(a_stages) * p.pk_stage_bytes;
  p.smem_bytes = p.smem_bar_off + bar_bytes;
  p.stage_q_pitch = q_pitch;
  p.stage_f_pitch = f_pitch;
  p.stage_warp_bytes = warp_stage;
  p.C_out_total = d->G * d->Cout_g;
  p.relu = d->relu;
  p.qmax_out = (1 << d->bits_out) - 1;
  for (int g = 0; g < d->G; ++g) p.dst_group[g] = g;
  for (int g = 0; g < d->G; ++g) p.src_group[g] = g;

  plan.supported = 1;
  plan.mode = p.mode;
  plan.rows_per_tile = p.Ht;
  plan.m_tiles = p.MT;
  plan.tile_pitch = p.Wh;
  plan.n_block = p.Nblk;
  plan.n_blocks = p.NB;
  plan.k_chunk = p.KC;
  plan.k_blocks = p.n_kb;
  plan.taps = taps;
  plan.weights_resident = p.b_resident;
  plan.acc_stages = p.acc_stages;
  plan.smem_bytes = static_cast<int32_t>(p.smem_bytes);
  plan.tiles = p.tiles;
  plan.work_items = p.items;
  if (pub) *pub = plan;
  if (P) *P = p;
  if (phases_out) *phases_out = phases;
  return PQ_OK;
}

// ---------------------------------------------------------------------------
// Planner of the pointwise kernel: 1x1, stride 1, pad 0 layers with
// channel-blocked byte codes in and codes only out.  Pure host arithmetic; false
// when the kernel does not cover the layer (the general kernel then runs it).
//   tiles: up to 256 pixels of one image (two 128-row accumulators) when they
//   fit the CTA's tensor memory, else up to 128; every group's weights resident
//   in shared memory (at most 96 KB); as many stages of input codes as the rest
//   of the CTA's shared memory holds (up to kPwMaxStages); two CTAs per SM when
//   each fits half the SM.  The weights use the general
//   kernel's packing with one output block per group (Cout_g <= 256).
// ---------------------------------------------------------------------------
bool plan_pointwise(const pq_layer_desc* d, pq::PwParams* out) {
  if (!(d->kh == 1 && d->kw == 1 && d->stride == 1 && d->pad == 0) || wslices_of(d) != 1) return false;
  if (d->code_format != PQ_CODES_C16) return false;
  if (d->G < 1 || d->G > pq::kMaxG || d->Cin_g % 32 != 0 || d->Cout_g % 16 != 0 || d->Cout_g > 256) return false;
  if (d->bits_a > 4 || d->bits_w > 4) return false;
  const int64_t qa = (1 << d->bits_a) - 1, qw = 1 << (d->bits_w - 1);
  if (static_cast<int64_t>(d->Cin_g) * qa * qw >= (1LL << 24)) return false;  // exact fp32 sums
  const int64_t HW = static_cast<int64_t>(d->H) * d->W;
  if (HW < 1 || HW > (1LL << 22)) return false;  // 32-bit plane offsets in the epilogue
  pq::PwParams p;
  std::memset(&p, 0, sizeof(p));
  p.Npow2 = std::max(32, next_pow2(d->Cout_g));  // the epilogue reads 32 columns at a time
  p.w_bytes = static_cast<uint32_t>(d->G) * d->Cin_g * d->Cout_g;
  if (p.w_bytes > 96u * 1024u) return false;
  p.nch = d->Cin_g / 16;
  if (p.nch > 256) return false;  // TMA box extent
  p.ksteps = d->Cin_g / 32;
  const uint32_t w_round = round_up(p.w_bytes, 1024);
  const uint32_t bar_bytes = 1024;
  // Two CTAs per SM where each fits half of the SM's shared memory (three or more
  // stages) and half of its tensor memory: a CTA of the next launch then starts
  // loading as soon as one of this launch's two CTAs on the SM finishes, and the
  // two CTAs' pipelines overlap.  Else one CTA with the whole SM.
  int stages = 0;
  for (int pair = 1; pair >= 0 && stages < 2; --pair) {
    const int tmem = pair ? 256 : 512;
    p.ctas_per_sm = pair ? 2 : 1;
    p.MT = (HW > 128 && 2 * p.Npow2 <= tmem / (pair ? 1 : 2)) ? 2 : 1;
    p.acc_stages = std::max(1, std::min(4, tmem / (p.MT * p.Npow2)));
    if (p.acc_stages == 3) p.acc_stages = 2;
    p.a_stage_bytes = static_cast<uint32_t>(p.MT) * p.nch * 2048u;
    const int64_t room = static_cast<int64_t>(pair ? pq::kPwHalfSmem : pq::kMaxSmem) - 1024 - w_round - bar_bytes;
    stages = static_cast<int>(std::min<int64_t>(pq::kPwMaxStages, room / p.a_stage_bytes));
    if (pair && stages < 3) stages = 0;
  }
  if (stages < 2) return false;
  p.tmem_cols = static_cast<uint32_t>(std::max(32, next_pow2(p.acc_stages * p.MT * p.Npow2)));
  p.T = static_cast<int>(std::min<int64_t>(HW, 128 * p.MT));
  p.tiles_per_img = static_cast<int>((HW + p.T - 1) / p.T);
  const int64_t items = static_cast<int64_t>(d->N) * p.tiles_per_img * d->G;
  if (items >= (1LL << 31)) return false;
  p.a_tx_bytes = p.a_stage_bytes;
  p.a_stages = stages;
  p.N = d->N;
  p.HW = static_cast<int>(HW);
  p.G = d->G;
  p.Cin_g = d->Cin_g;
  p.Cout_g = d->Cout_g;
  p.items = static_cast<int>(items);
  p.smem_w_off = static_cast<uint32_t>(stages) * p.a_stage_bytes;
  p.smem_bar_off = p.smem_w_off + w_round;
  p.smem_bytes = p.smem_bar_off + bar_bytes;
  p.C16_out = d->G * d->Cout_g / 16;
  p.qmax2 = static_cast<uint32_t>((1 << d->bits_out) - 1) * 0x00010001u;
  if (out) *out = p;
  return true;
}

// Tensor map of the pointwise kernel's input codes, channel-blocked: 8-byte
// elements, dims (2 HW, C/16, N); box (2 * 128, nch, 1), one accumulator's 128
// positions of the group's planes.  Positions past the image are zero-filled.
bool encode_pw_map(const pq_layer_desc* d, const pq::PwParams& p, const void* q_dev, CUtensorMap* map);

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

// Learned bounds usable by the quantisers: finite, l < u, and fl(1 / fl(u - l)) finite.
bool valid_bounds(int G, const float* l, const float* u) {
  for (int g = 0; g < G; ++g) {
    if (!std::isfinite(l[g]) || !std::isfinite(u[g]) || !(u[g] > l[g])) return false;
    const float r = u[g] - l[g];
    if (!std::isfinite(r) || !(r > 0.0f) || !std::isfinite(1.0f / r)) return false;
  }
  return true;
}

pq_status quantize_act_impl(const float* x_dev, void* q_dev, int64_t N, int32_t H, int32_t W, int32_t G, int32_t Cg,
                            int32_t bits, int32_t code_format, const float* inv_s_host, const float* l_host,
                            const float* u_host, pq_stream_t stream);

// ---------------------------------------------------------------------------
// Tensor map of channel-blocked activation codes for the TMA operand loads.
// Element = 8 bytes, so one 16-byte position is 2 elements and a plane row of
// Wd positions is one box row of 2 Wd elements (a contiguous run).
// Rows mode (stride 1): dims (2W, H, C/16, N); box (2 Wd, Hd, nch, 1).
// Flat mode: dims (2 HW, C/16, N); box (2 * 128, nch, 1).
// Out-of-range elements are zero-filled: the zero padding.
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static std::once_flag once;
  static EncodeTiledFn fn = nullptr;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult qres;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &qres) ==
            cudaSuccess &&
        qres == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

bool encode_c16_map(const pq_layer_desc* d, const ConvParams& p, const void* q_dev, CUtensorMap* map) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return false;
  std::memset(map, 0, sizeof(*map));
  // 16-byte chunks per position: C/16, or C/32 for FP4 nibbles
  const uint64_t C16 = static_cast<uint64_t>(d->G) * d->Cin_g / (p.codes_f4 ? 32 : 16), H = d->H, W = d->W;
  cuuint32_t es[4] = {1, 1, 1, 1};
  if (p.codes_p2) {
    // Packed codes: one 32-bit word per (position, 16-channel block).
    if (p.mode == pq::kModeFlat) {
      cuuint64_t dims[3] = {H * W, C16, static_cast<cuuint64_t>(d->N)};
      cuuint64_t strides[2] = {H * W * 4, C16 * H * W * 4};
      cuuint32_t box[3] = {static_cast<cuuint32_t>(p.pk_box_w), static_cast<cuuint32_t>(p.nch), 1};
      return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT32, 3, const_cast<void*>(q_dev), dims, strides, box, es,
                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
    }
    cuuint64_t dims[4] = {W, H, C16, static_cast<cuuint64_t>(d->N)};
    cuuint64_t strides[3] = {W * 4, H * W * 4, C16 * H * W * 4};
    cuuint32_t box[4] = {static_cast<cuuint32_t>(p.pk_box_w), static_cast<cuuint32_t>(p.Hd),
                         static_cast<cuuint32_t>(p.nch), 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT32, 4, const_cast<void*>(q_dev), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  }
  if (p.mode == pq::kModeFlat) {
    cuuint64_t dims[3] = {2 * H * W, C16, static_cast<cuuint64_t>(d->N)};
    cuuint64_t strides[2] = {H * W * 16, C16 * H * W * 16};
    cuuint32_t box[3] = {2u * 128u, static_cast<cuuint32_t>(p.nch), 1};  // one accumulator's 128 positions
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT64, 3, const_cast<void*>(q_dev), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  }
  cuuint64_t dims[4] = {2 * W, H, C16, static_cast<cuuint64_t>(d->N)};
  cuuint64_t strides[3] = {W * 16, H * W * 16, C16 * H * W * 16};
  // stride 2 (a_split): the window of 2 Hd rows x 2 Wd positions
  const cuuint32_t sw = p.a_split ? 2u : 1u;
  cuuint32_t box[4] = {2u * sw * static_cast<cuuint32_t>(p.Wd), sw * static_cast<cuuint32_t>(p.Hd),
                       static_cast<cuuint32_t>(p.nch), 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT64, 4, const_cast<void*>(q_dev), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tensor map of fp32 NHWC activations for quantise-on-load: boxes of 32 channels
// (128 bytes, swizzled 128B so the copy warps read them without bank conflicts)
// x Wd positions x Hd rows (rows mode), or x 128 positions (flat mode, HW as one
// dimension).  Out-of-range positions are zero-filled (code 0, the zero padding),
// or with learned bounds NaN-filled, which that quantiser maps to code 0 whatever
// the lower bound is.
bool encode_f32_map(const pq_layer_desc* d, const ConvParams& p, const void* x_dev, CUtensorMap* map) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return false;
  std::memset(map, 0, sizeof(*map));
  // learned bounds: NaN padding (code 0 for any lower bound); else zeros (code 0)
  const CUtensorMapFloatOOBfill fill =
      p.q_lu ? CU_TENSOR_MAP_FLOAT_OOB_FILL_NAN_REQUEST_ZERO_FMA : CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE;
  const uint64_t C = static_cast<uint64_t>(d->G) * d->Cin_g, H = d->H, W = d->W;
  cuuint32_t es[4] = {1, 1, 1, 1};
  if (p.mode == pq::kModeFlat) {
    cuuint64_t dims[3] = {C, H * W, static_cast<cuuint64_t>(d->N)};
    cuuint64_t strides[2] = {C * 4, H * W * C * 4};
    cuuint32_t box[3] = {32u, static_cast<cuuint32_t>(p.flat_box), 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void*>(x_dev), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               fill) == CUDA_SUCCESS;
  }
  cuuint64_t dims[4] = {C, W, H, static_cast<cuuint64_t>(d->N)};
  cuuint64_t strides[3] = {C * 4, W * C * 4, H * W * C * 4};
  cuuint32_t box[4] = {32u, static_cast<cuuint32_t>(p.Wd), static_cast<cuuint32_t>(p.Hd), 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<void*>(x_dev), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             fill) == CUDA_SUCCESS;
}

bool encode_pw_map(const pq_layer_desc* d, const pq::PwParams& p, const void* q_dev, CUtensorMap* map) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return false;
  std::memset(map, 0, sizeof(*map));
  const uint64_t C16 = static_cast<uint64_t>(d->G) * d->Cin_g / 16, HW = static_cast<uint64_t>(p.HW);
  cuuint32_t es[3] = {1, 1, 1};
  cuuint64_t dims[3] = {2 * HW, C16, static_cast<cuuint64_t>(d->N)};
  cuuint64_t strides[2] = {HW * 16, C16 * HW * 16};
  cuuint32_t box[3] = {256u, static_cast<cuuint32_t>(p.nch), 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT64, 3, const_cast<void*>(q_dev), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ---------------------------------------------------------------------------
// Weight packing (tensor-core operand layout of the planner's tiling).
//   unit u = g * NB + nb; for each tap t, 16-byte chunk J of the input channels
//   (J = kb * nch + j for K block kb), output channel c (of the block) and
//   channel e of the chunk (E = 16 channels per chunk, 32 for FP4):
//   element[(((u * taps + t) * NCH + J) * Nblk + c) * E + e]
//     = w_q[g, nb*Nblk + c, tap t, J*E + e],   NCH = Cin_g / E
//   so a (K block, tap) slice is one contiguous run whatever the K blocking
//   (the same packing serves every tiling of the layer).
//   as an E4M3 byte, or (FP4) an E2M1 nibble, element 2i in the low nibble of
//   byte i and element 2i+1 in the high one.
// ---------------------------------------------------------------------------
template <typename F>
void for_each_packed(const ConvParams& p, int kw, F&& f) {
  const int E = 16 << (p.chunk_shift - 4);
  for (int g = 0; g < p.G; ++g)
    for (int nb = 0; nb < p.NB; ++nb)
      for (int kb = 0; kb < p.n_kb; ++kb)
        for (int t = 0; t < p.taps; ++t)
          for (int j = 0; j < p.nch; ++j)
            for (int c = 0; c < p.Nblk; ++c)
              for (int e = 0; e < E; ++e) {
                const int u = g * p.NB + nb;
                const size_t dst =
                    ((((static_cast<size_t>(u) * p.taps + t) * p.n_kb + kb) * p.nch + j) * p.Nblk + c) * E + e;
                const int co = nb * p.Nblk + c;
                const int ci = kb * p.KC + j * E + e;
                const int i = t / kw, jj = t % kw;
                const size_t src = (((static_cast<size_t>(g) * p.Cout_g + co) * (p.taps / kw) + i) * kw + jj) * p.Cin_g + ci;
                f(dst, src);
              }
}

// E2M1 nibble of an integer weight code in [-4, 4]: the magnitudes 0..4 are the
// E2M1 values 0, 1.0, 2.0, 3.0, 4.0 (nibbles 0, 2, 4, 5, 6), bit 3 the sign.
uint8_t e2m1_of_int(int v) {
  static const uint8_t mag[5] = {0, 2, 4, 5, 6};
  const int a = v < 0 ? -v : v;
  return static_cast<uint8_t>(mag[a] | (v < 0 ? 8 : 0));
}

// Inverse of e2m1_of_int (nibbles it does not produce read as -128).
int int_of_e2m1(uint8_t b) {
  static const int val[8] = {0, -128, 1, -128, 2, 3, 4, -128};
  const int m = val[b & 7];
  return (b & 8) && m != -128 ? -m : m;
}

// Bytes of the packed weight operand: one per code, or one per two (FP4).
size_t packed_weight_bytes_of(const pq_layer_desc* d, const ConvParams& p) {
  const size_t elems = static_cast<size_t>(d->G) * d->Cout_g * weight_taps(d) * d->Cin_g;
  return p.codes_f4 ? elems / 2 : elems;
}

// Write the signed codes wq [G][Cout_g][kh][kw][R][Cin_g] in the operand layout
// (a tap of the operand is a kernel position and weight slice: kw R per row).
void pack_codes(const ConvParams& p, const pq_layer_desc* d, const int8_t* wq, uint8_t* out) {
  const int kwr = d->kw * wslices_of(d);
  if (p.codes_f4) {
    std::memset(out, 0, packed_weight_bytes_of(d, p));
    for_each_packed(p, kwr, [&](size_t dst, size_t src) {
      out[dst >> 1] = static_cast<uint8_t>(out[dst >> 1] | (e2m1_of_int(wq[src]) << (4 * (dst & 1))));
    });
  } else {
    for_each_packed(p, kwr, [&](size_t dst, size_t src) { out[dst] = e4m3_of_int(wq[src]); });
  }
}

// inv_s_in (host, G floats, or NULL): q_dev is fp32 NHWC activations quantised on
// load with these reciprocal steps instead of codes.
pq_status layer_fused_impl(const void* q_dev, const void* w_packed_dev, const pq_layer_desc* d,
                           const float* m_out_host, const float* m_req_host, pq_shuffle shuf,
                           const float* shortcut_dev, int32_t* acc_out_dev, float* y_out_dev, void* q_out_dev,
                           const int* src_group, pq_stream_t stream, const float* inv_s_in = nullptr,
                           const float* l_in = nullptr, const float* u_in = nullptr) {
  pq_status st = validate_desc(d);
  if (st != PQ_OK) return st;
  if (q_dev == nullptr || w_packed_dev == nullptr) return PQ_EINVAL;
  if (acc_out_dev == nullptr && y_out_dev == nullptr && q_out_dev == nullptr) return PQ_EINVAL;
  if ((y_out_dev != nullptr || q_out_dev != nullptr) && m_out_host == nullptr) return PQ_EINVAL;
  if (q_out_dev != nullptr && m_req_host == nullptr) return PQ_EINVAL;
  if (!aligned16(q_dev) || !aligned16(w_packed_dev) || !aligned16(acc_out_dev) || !aligned16(y_out_dev) ||
      !aligned16(q_out_dev) || !aligned16(shortcut_dev))
    return PQ_EINVAL;
  ConvParams p;
  std::vector<Phase> phases;
  // Channel-blocked codes as the only output are stored from registers (the
  // per-channel scatter of the channel shuffle is unstaged too).
  const bool direct_out =
      acc_out_dev == nullptr && y_out_dev == nullptr && shortcut_dev == nullptr && d->code_format != PQ_CODES_INT8;
  const bool quant_in = inv_s_in != nullptr || l_in != nullptr;
  st = plan_conv(d, &p, nullptr, &phases, quant_in, direct_out, shortcut_dev != nullptr);
  if (st != PQ_OK) return st;
  if (l_in != nullptr) {
    // learned bounds: the training forward's codes (sat((x - l) * fl(1/fl(u - l))) * Qp, rounded)
    if (u_in == nullptr || !valid_bounds(d->G, l_in, u_in)) return PQ_EINVAL;
    p.q_lu = 1;
    for (int g = 0; g < d->G; ++g) {
      p.q_neg_l[g] = -l_in[g];
      p.q_inv_r[g] = 1.0f / (u_in[g] - l_in[g]);
    }
    p.q_qp = static_cast<float>((1 << d->bits_a) - 1);
    p.q_qmax2 = static_cast<uint32_t>((1 << d->bits_a) - 1) * 0x00010001u;
  } else if (inv_s_in != nullptr) {
    // reciprocal steps scaled by 2^-b (exact: a power of two) for the saturating form
    const float inv_two_b = 1.0f / static_cast<float>(1 << d->bits_a);
    for (int g = 0; g < d->G; ++g) {
      if (!std::isfinite(inv_s_in[g]) || !(inv_s_in[g] >= 0.0f) || (inv_s_in[g] != 0.0f && inv_s_in[g] < 1e-30f) ||
          inv_s_in[g] > 1e30f)
        return PQ_EINVAL;
      p.q_inv_sat[g] = inv_s_in[g] * inv_two_b;
    }
    p.q_two_b = static_cast<float>(1 << d->bits_a);
    p.q_qmax2 = static_cast<uint32_t>((1 << d->bits_a) - 1) * 0x00010001u;
  }
  int dst[pq::kMaxG];
  if (!valid_shuffle(d->G, shuf, dst)) return PQ_EINVAL;
  if (d->N == 0) return PQ_OK;
  // Multipliers are scaled by 2^9 inside the kernel; keep them in the range where
  // that scaling and every product with an accumulator stay exact normal floats.
  auto usable = [](float m) { return std::isfinite(m) && (m == 0.0f || (std::fabs(m) > 1e-30f && std::fabs(m) < 1e30f)); };
  for (int g = 0; g < d->G; ++g) {
    p.dst_group[g] = dst[g];
    p.src_group[g] = src_group ? src_group[g] : g;
    p.m_out[g] = m_out_host ? m_out_host[g] : 0.0f;
    p.m_req[g] = m_req_host ? m_req_host[g] : 0.0f;
    if (!usable(p.m_out[g]) || !usable(p.m_req[g])) return PQ_EINVAL;
    p.m_out512[g] = p.m_out[g] * 512.0f;
    p.m_req512[g] = p.m_req[g] * 512.0f;
  }
  p.channel_shuffle = shuf.kind == 2 ? 1 : 0;
  // A per-channel scatter cannot write single 2-bit codes into packed bytes.
  if (p.channel_shuffle && (p.codes_p2 || p.codes_f4) && q_out_dev != nullptr) return PQ_EUNSUPPORTED;
  p.w_packed = static_cast<const uint8_t*>(w_packed_dev);
  p.shortcut = shortcut_dev;
  p.acc_out = acc_out_dev;
  p.y_out = y_out_dev;
  p.q_out = static_cast<uint8_t*>(q_out_dev);
  p.err = pq::device_error_word();
  if (p.err == nullptr) return PQ_ECUDA;
  p.wait_limit_ns = g_wait_limit_ns.load();
  p.q_in = static_cast<const uint8_t*>(q_dev);
  const int sms = device_sm_count();
  if (sms <= 0) return PQ_ECUDA;
  // 1x1 layers with codes only out run on the pointwise kernel where it covers them.
  pq::PwParams pw;
  if (!quant_in && direct_out && q_out_dev != nullptr && shortcut_dev == nullptr && src_group == nullptr &&
      !p.channel_shuffle && plan_pointwise(d, &pw)) {
    for (int g = 0; g < d->G; ++g) {
      pw.m_req15[g] = p.m_req[g] * (1.0f / 32768.0f);  // exact: m_req is 0 or above 1e-30 in magnitude
      pw.dst_group[g] = dst[g];
    }
    pw.w_packed = p.w_packed;
    pw.q_out = p.q_out;
    pw.err = p.err;
    pw.wait_limit_ns = p.wait_limit_ns;
    pw.pdl = 1;
    pw.pdl_early_loads = (d->flags & PQ_LAYER_INPUTS_READY) ? 1 : 0;
    const int pw_grid = std::min(sms * pw.ctas_per_sm, pw.items);
    if (pw_grid <= 0) return PQ_OK;
    CUtensorMap pw_map;
    if (!encode_pw_map(d, pw, q_dev, &pw_map)) return PQ_ECUDA;
    if (pq::launch_pointwise_tc(pw, pw_map, pw_grid, static_cast<cudaStream_t>(stream)) != 0) return PQ_ECUDA;
    return PQ_OK;
  }
  const int grid = static_cast<int>(std::min<int64_t>(sms, p.items));
  if (grid <= 0) return PQ_OK;
  CUtensorMap map;
  std::memset(&map, 0, sizeof(map));
  p.pdl = 1;  // programmatic dependent launch: the set-up overlaps the previous grid's last CTAs
  p.pdl_early_loads = (d->flags & PQ_LAYER_INPUTS_READY) ? 1 : 0;
  if (p.a_quant) {
    if (!encode_f32_map(d, p, q_dev, &map)) return PQ_ECUDA;
  } else if (p.a_tma && !encode_c16_map(d, p, q_dev, &map)) {
    return PQ_ECUDA;
  }
  if (pq::launch_conv_tc(p, map, grid, static_cast<cudaStream_t>(stream)) != 0) return PQ_ECUDA;
  return PQ_OK;
}

}  // namespace

// ===========================================================================
// Public ABI
// ===========================================================================
extern "C" {

const char* palquant_strerror(pq_status s) {
  switch (s) {
    case PQ_OK: return "ok";
    case PQ_EINVAL: return "invalid argument";
    case PQ_EUNSUPPORTED: return "unsupported layer shape or format";
    case PQ_ECUDA: return "CUDA error";
    case PQ_ETIMEOUT: return "in-kernel wait timed out";
  }
  return "unknown status";
}

int palquant_version(void) { return 100; }

size_t palquant_act_steps_scratch_bytes(int64_t P, int32_t G) {
  (void)P;
  if (G < 1) return 0;
  return sizeof(double) * (static_cast<size_t>(kActSumBlocks) * G + G);
}

pq_status palquant_act_steps(const float* x_dev, int64_t N, int32_t H, int32_t W, int32_t G, int32_t Cg, int32_t bits,
                             void* scratch_dev, size_t scratch_bytes, float* s_out_host, pq_stream_t stream) {
  if (x_dev == nullptr || scratch_dev == nullptr || s_out_host == nullptr) return PQ_EINVAL;
  if (N < 1 || H < 1 || W < 1 || G < 1 || Cg < 1 || bits < 1 || bits > 8) return PQ_EINVAL;
  const int64_t P = N * H * W;
  if (scratch_bytes < palquant_act_steps_scratch_bytes(P, G) || (reinterpret_cast<uintptr_t>(scratch_dev) & 7u))
    return PQ_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  double* partial = static_cast<double*>(scratch_dev);
  double* sums = partial + static_cast<size_t>(kActSumBlocks) * G;
  if (pq::launch_act_sum(x_dev, P, G, Cg, partial, kActSumBlocks, s) != 0) return PQ_ECUDA;
  if (pq::launch_act_sum_finish(partial, kActSumBlocks, G, sums, s) != 0) return PQ_ECUDA;
  std::vector<double> h(G);
  if (cudaMemcpyAsync(h.data(), sums, sizeof(double) * G, cudaMemcpyDeviceToHost, s) != cudaSuccess) return PQ_ECUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return PQ_ECUDA;
  const double qp = static_cast<double>((1 << bits) - 1);
  for (int g = 0; g < G; ++g) {
    const double mean = h[g] / static_cast<double>(P * Cg);
    s_out_host[g] = static_cast<float>(2.0 * mean / std::sqrt(qp));
  }
  return PQ_OK;
}

pq_status palquant_weight_steps(const float* w_host, const pq_layer_desc* d, float* s_w_out_host) {
  if (w_host == nullptr || s_w_out_host == nullptr) return PQ_EINVAL;
  pq_status st = validate_desc(d);
  if (st != PQ_OK) return st;
  if (wslices_of(d) != 1) return PQ_EINVAL;  // float weights belong to plain layers
  const int64_t per_group = static_cast<int64_t>(d->Cout_g) * d->kh * d->kw * d->Cin_g;
  const double qp = static_cast<double>((1 << (d->bits_w - 1)) - 1);
  for (int g = 0; g < d->G; ++g) {
    double sum = 0.0;
    for (int64_t i = 0; i < per_group; ++i) sum += std::fabs(static_cast<double>(w_host[g * per_group + i]));
    s_w_out_host[g] = static_cast<float>(2.0 * (sum / static_cast<double>(per_group)) / std::sqrt(qp));
  }
  return PQ_OK;
}

pq_status palquant_epilogue_scales(int32_t G, const float* s_w_host, const float* s_a_host, double alpha,
                                   const float* s_next_host, pq_shuffle shuf, float* m_out_host, float* m_req_host) {
  if (G < 1 || G > pq::kMaxG || s_w_host == nullptr || s_a_host == nullptr || m_out_host == nullptr) return PQ_EINVAL;
  if (s_next_host != nullptr && m_req_host == nullptr) return PQ_EINVAL;
  int dst[pq::kMaxG];
  if (!valid_shuffle(G, shuf, dst)) return PQ_EINVAL;
  for (int g = 0; g < G; ++g) {
    const double m = static_cast<double>(s_w_host[g]) * static_cast<double>(s_a_host[g]) * alpha;
    m_out_host[g] = static_cast<float>(m);
    if (s_next_host != nullptr) m_req_host[g] = static_cast<float>(m / static_cast<double>(s_next_host[dst[g]]));
  }
  return PQ_OK;
}

size_t palquant_packed_weight_bytes(const pq_layer_desc* d) {
  ConvParams p;
  if (plan_conv(d, &p, nullptr, nullptr) != PQ_OK) return 0;
  return packed_weight_bytes_of(d, p);
}

pq_status palquant_pack_weight_codes_host(const int8_t* wq_host, const pq_layer_desc* d, void* packed_host,
                                          size_t packed_bytes) {
  if (wq_host == nullptr || packed_host == nullptr) return PQ_EINVAL;
  ConvParams p;
  pq_status st = plan_conv(d, &p, nullptr, nullptr);
  if (st != PQ_OK) return st;
  const size_t elems = static_cast<size_t>(d->G) * d->Cout_g * weight_taps(d) * d->Cin_g;
  if (packed_bytes < packed_weight_bytes_of(d, p)) return PQ_EINVAL;
  const int lo = -(1 << (d->bits_w - 1)), hi = (1 << (d->bits_w - 1)) - 1;
  for (size_t i = 0; i < elems; ++i)
    if (wq_host[i] < lo || wq_host[i] > hi) return PQ_EINVAL;
  pack_codes(p, d, wq_host, static_cast<uint8_t*>(packed_host));
  return PQ_OK;
}

pq_status palquant_unpack_weight_codes_host(const void* packed_host, const pq_layer_desc* d, int8_t* wq_host) {
  if (packed_host == nullptr || wq_host == nullptr) return PQ_EINVAL;
  ConvParams p;
  pq_status st = plan_conv(d, &p, nullptr, nullptr);
  if (st != PQ_OK) return st;
  const uint8_t* in = static_cast<const uint8_t*>(packed_host);
  const int kwr = d->kw * wslices_of(d);
  if (p.codes_f4)
    for_each_packed(p, kwr, [&](size_t dst, size_t src) {
      wq_host[src] = static_cast<int8_t>(int_of_e2m1(static_cast<uint8_t>(in[dst >> 1] >> (4 * (dst & 1)))));
    });
  else
    for_each_packed(p, kwr, [&](size_t dst, size_t src) { wq_host[src] = static_cast<int8_t>(int_of_e4m3(in[dst])); });
  return PQ_OK;
}

pq_status palquant_pack_weights_host(const float* w_host, const pq_layer_desc* d, const float* inv_sw_host,
                                     void* packed_host, size_t packed_bytes) {
  if (w_host == nullptr || inv_sw_host == nullptr || packed_host == nullptr) return PQ_EINVAL;
  pq_status st = validate_desc(d);
  if (st != PQ_OK) return st;
  if (wslices_of(d) != 1) return PQ_EINVAL;  // float weights belong to plain layers
  const size_t per_group = static_cast<size_t>(d->Cout_g) * d->kh * d->kw * d->Cin_g;
  std::vector<int8_t> wq(per_group * d->G);
  const float lo = static_cast<float>(-(1 << (d->bits_w - 1))), hi = static_cast<float>((1 << (d->bits_w - 1)) - 1);
  for (int g = 0; g < d->G; ++g)
    for (size_t i = 0; i < per_group; ++i) {
      // one fp32 multiply, round half to even, clamp (volatile keeps it a single
      // IEEE fp32 product, never fused or widened)
      volatile float t = w_host[g * per_group + i] * inv_sw_host[g];
      float r = std::nearbyint(static_cast<float>(t));
      r = std::fmax(r, lo);
      r = std::fmin(r, hi);
      wq[g * per_group + i] = static_cast<int8_t>(static_cast<int>(r));
    }
  return palquant_pack_weight_codes_host(wq.data(), d, packed_host, packed_bytes);
}

pq_status palquant_pack_weights_odd_host(const float* w_host, const pq_layer_desc* d, const float* u_host,
                                        void* packed_host, size_t packed_bytes) {
  if (w_host == nullptr || u_host == nullptr || packed_host == nullptr) return PQ_EINVAL;
  ConvParams p;
  pq_status st = plan_conv(d, &p, nullptr, nullptr);
  if (st != PQ_OK) return st;
  if (wslices_of(d) != 1) return PQ_EINVAL;  // float weights belong to plain layers
  const size_t per_group = static_cast<size_t>(d->Cout_g) * d->kh * d->kw * d->Cin_g;
  const size_t need = per_group * d->G;
  if (packed_bytes < packed_weight_bytes_of(d, p)) return PQ_EINVAL;
  const int qp = (1 << d->bits_w) - 1;
  // the odd levels reach 2^b - 1 in magnitude: keep every sum exact in fp32 (and,
  // for FP4 operands, every level an E2M1 value: b <= 2)
  const int64_t taps = static_cast<int64_t>(d->kh) * d->kw;
  if (qp > 15 || taps * d->Cin_g * ((1LL << d->bits_a) - 1) * qp >= (1LL << 24)) return PQ_EUNSUPPORTED;
  if (p.codes_f4 && qp > 3) return PQ_EUNSUPPORTED;
  std::vector<int8_t> wq(need);
  for (int g = 0; g < d->G; ++g) {
    if (!(u_host[g] > 0.0f) || !std::isfinite(u_host[g])) return PQ_EINVAL;
    const float k = static_cast<float>(static_cast<double>(qp) / (2.0 * static_cast<double>(u_host[g])));
    for (size_t i = 0; i < per_group; ++i) {
      // one fp32 add and one fp32 multiply (volatile: never fused or widened)
      volatile float a = w_host[g * per_group + i] + u_host[g];
      volatile float t = a * k;
      float r = std::nearbyint(static_cast<float>(t));
      r = std::fmax(r, 0.0f);
      r = std::fmin(r, static_cast<float>(qp));
      wq[g * per_group + i] = static_cast<int8_t>(2 * static_cast<int>(r) - qp);
    }
  }
  pack_codes(p, d, wq.data(), static_cast<uint8_t*>(packed_host));
  return PQ_OK;
}

pq_status palquant_pack_weights(const float* w_host, const pq_layer_desc* d, const float* inv_sw_host,
                                void* packed_dev, size_t packed_bytes, pq_stream_t stream) {
  if (packed_dev == nullptr) return PQ_EINVAL;
  const size_t need = palquant_packed_weight_bytes(d);
  if (need == 0) {
    pq_status st = validate_desc(d);
    return st != PQ_OK ? st : PQ_EUNSUPPORTED;
  }
  if (packed_bytes < need) return PQ_EINVAL;
  std::vector<uint8_t> host(need);
  pq_status st = palquant_pack_weights_host(w_host, d, inv_sw_host, host.data(), need);
  if (st != PQ_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(packed_dev, host.data(), need, cudaMemcpyHostToDevice, s) != cudaSuccess) return PQ_ECUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return PQ_ECUDA;
  return PQ_OK;
}

pq_status palquant_quantize_act(const float* x_dev, void* q_dev, int64_t N, int32_t H, int32_t W, int32_t G, int32_t Cg,
                                int32_t bits, int32_t code_format, const float* inv_s_host, pq_stream_t stream) {
  if (inv_s_host == nullptr) return PQ_EINVAL;
  return quantize_act_impl(x_dev, q_dev, N, H, W, G, Cg, bits, code_format, inv_s_host, nullptr, nullptr, stream);
}

pq_status palquant_quantize_act_lu(const float* x_dev, void* q_dev, int64_t N, int32_t H, int32_t W, int32_t G,
                                   int32_t Cg, int32_t bits, int32_t code_format, const float* l_host,
                                   const float* u_host, pq_stream_t stream) {
  if (l_host == nullptr || u_host == nullptr) return PQ_EINVAL;
  if (G >= 1 && G <= pq::kMaxG && !valid_bounds(G, l_host, u_host)) return PQ_EINVAL;
  return quantize_act_impl(x_dev, q_dev, N, H, W, G, Cg, bits, code_format, nullptr, l_host, u_host, stream);
}

}  // extern "C"

namespace {

pq_status quantize_act_impl(const float* x_dev, void* q_dev, int64_t N, int32_t H, int32_t W, int32_t G, int32_t Cg,
                            int32_t bits, int32_t code_format, const float* inv_s_host, const float* l_host,
                            const float* u_host, pq_stream_t stream) {
  if (x_dev == nullptr || q_dev == nullptr) return PQ_EINVAL;
  if (N < 0 || H < 1 || W < 1 || G < 1 || Cg < 1 || bits < 1 || bits > 8) return PQ_EINVAL;
  if (G > pq::kMaxG) return PQ_EUNSUPPORTED;
  if (code_format == PQ_CODES_E4M3) return PQ_EUNSUPPORTED;
  if (code_format != PQ_CODES_INT8 && code_format != PQ_CODES_C16 && code_format != PQ_CODES_C16P2 &&
      code_format != PQ_CODES_C32F4)
    return PQ_EINVAL;
  const int64_t P = N * H * W;
  if (code_format != PQ_CODES_INT8) {
    if (Cg % 16 != 0) return PQ_EINVAL;
    if ((code_format == PQ_CODES_C16P2 || code_format == PQ_CODES_C32F4) && bits > 2) return PQ_EINVAL;
    if (code_format == PQ_CODES_C32F4 && (static_cast<int64_t>(G) * Cg) % 32 != 0) return PQ_EINVAL;
    if (!aligned16(x_dev) || !aligned16(q_dev)) return PQ_EINVAL;
    const int pack = code_format == PQ_CODES_C16P2 ? 1 : (code_format == PQ_CODES_C32F4 ? 2 : 0);
    if (pq::launch_quantize_c16(x_dev, static_cast<uint8_t*>(q_dev), N, static_cast<int64_t>(H) * W, G, Cg, bits,
                                inv_s_host, pack, static_cast<cudaStream_t>(stream), l_host, u_host) != 0)
      return PQ_ECUDA;
    return PQ_OK;
  }
  if (pq::launch_quantize(x_dev, static_cast<uint8_t*>(q_dev), P, G, Cg, bits, inv_s_host,
                          static_cast<cudaStream_t>(stream), l_host, u_host) != 0)
    return PQ_ECUDA;
  return PQ_OK;
}

}  // namespace

extern "C" {

pq_status palquant_layer_fused(const void* q_dev, const void* w_packed_dev, const pq_layer_desc* d,
                               const float* m_out_host, const float* m_req_host, pq_shuffle shuf,
                               const float* shortcut_dev, int32_t* acc_out_dev, float* y_out_dev, void* q_out_dev,
                               pq_stream_t stream) {
  return layer_fused_impl(q_dev, w_packed_dev, d, m_out_host, m_req_host, shuf, shortcut_dev, acc_out_dev, y_out_dev,
                          q_out_dev, nullptr, stream);
}

pq_status palquant_quantize_layer_fused(const float* x_dev, const float* inv_s_host, const void* w_packed_dev,
                                        const pq_layer_desc* d, const float* m_out_host, const float* m_req_host,
                                        pq_shuffle shuf, const float* shortcut_dev, int32_t* acc_out_dev,
                                        float* y_out_dev, void* q_out_dev, pq_stream_t stream) {
  if (inv_s_host == nullptr) return PQ_EINVAL;
  return layer_fused_impl(x_dev, w_packed_dev, d, m_out_host, m_req_host, shuf, shortcut_dev, acc_out_dev, y_out_dev,
                          q_out_dev, nullptr, stream, inv_s_host);
}

pq_status palquant_quantize_layer_fused_lu(const float* x_dev, const float* l_host, const float* u_host,
                                           const void* w_packed_dev, const pq_layer_desc* d, const float* m_out_host,
                                           const float* m_req_host, pq_shuffle shuf, const float* shortcut_dev,
                                           int32_t* acc_out_dev, float* y_out_dev, void* q_out_dev,
                                           pq_stream_t stream) {
  if (l_host == nullptr || u_host == nullptr) return PQ_EINVAL;
  return layer_fused_impl(x_dev, w_packed_dev, d, m_out_host, m_req_host, shuf, shortcut_dev, acc_out_dev, y_out_dev,
                          q_out_dev, nullptr, stream, nullptr, l_host, u_host);
}

pq_status palquant_cyclic_shuffle_module(const void* q_dev, const void* w_packed_dev, const pq_layer_desc* d,
                                         const float* m_out_host, const float* m_req_host, int32_t shift,
                                         const float* x_dev, float* z_out_dev, void* q_out_dev, pq_stream_t stream) {
  pq_status st = validate_desc(d);
  if (st != PQ_OK) return st;
  if (d->kh != 1 || d->kw != 1 || d->stride != 1 || d->pad != 0 || d->Cin_g != d->Cout_g) return PQ_EINVAL;
  if (x_dev == nullptr || (z_out_dev == nullptr && q_out_dev == nullptr)) return PQ_EINVAL;
  // Eq. 8: Y[:, pi(i)] = X[:, i] with pi(i) = (i + shift) mod G, so conv group g reads
  // input group pi^-1(g) = (g - shift) mod G.
  int src[pq::kMaxG];
  if (d->G > pq::kMaxG) return PQ_EUNSUPPORTED;
  for (int g = 0; g < d->G; ++g) src[g] = pos_mod(g - shift, d->G);
  pq_shuffle none = {0, 0, nullptr};
  return layer_fused_impl(q_dev, w_packed_dev, d, m_out_host, m_req_host, none, x_dev, nullptr, z_out_dev, q_out_dev,
                          src, stream);
}

pq_status palquant_group_conv(const void* q_dev, const void* w_packed_dev, int32_t* acc_dev, const pq_layer_desc* d,
                              pq_stream_t stream) {
  if (acc_dev == nullptr) return PQ_EINVAL;
  pq_shuffle none = {0, 0, nullptr};
  return palquant_layer_fused(q_dev, w_packed_dev, d, nullptr, nullptr, none, nullptr, acc_dev, nullptr, nullptr,
                              stream);
}

// ---------------------------------------------------------------------------
// Bit-level decomposition (Sec. 3.3, Eq. 4).
// ---------------------------------------------------------------------------
namespace {
int ceil_div(int a, int b) { return (a + b - 1) / b; }

// The decomposed layer: K blocks (i, j) for i < Ga activation slices, j < Gw
// weight slices; PQ_OK only when every shifted weight slice value is an exact
// E4M3 number and the M-bit products stay exact in fp32.
pq_status bitsplit_layer(const pq_layer_desc* d, int bits_b, pq_layer_desc* out, int* ga, int* gw) {
  pq_status st = validate_desc(d);
  if (st != PQ_OK) return st;
  if (bits_b < 1 || bits_b > 4) return PQ_EINVAL;
  // the M-bit input codes and the shifted weight slices are one per byte
  if (d->code_format == PQ_CODES_C16P2 || d->code_format == PQ_CODES_C32F4) return PQ_EUNSUPPORTED;
  const int Ga = ceil_div(d->bits_a, bits_b), Gw = ceil_div(d->bits_w, bits_b);
  // (i+1) B <= 8 keeps the byte-wise slicing exact; the largest shifted weight
  // slice is (2^B - 1) 2^((Ga-1 + Gw-1) B) (E4M3 holds integers m 2^k with
  // m < 16 up to 448).
  if (Ga * bits_b > 8) return PQ_EUNSUPPORTED;
  const int64_t wmax = ((1LL << bits_b) - 1) << ((Ga - 1 + Gw - 1) * bits_b);
  if (wmax > 448) return PQ_EUNSUPPORTED;
  const int64_t taps = static_cast<int64_t>(d->kh) * d->kw;
  if (taps * d->Cin_g * ((1LL << d->bits_a) - 1) * (1LL << (d->bits_w - 1)) >= (1LL << 24)) return PQ_EUNSUPPORTED;
  if (wslices_of(d) != 1) return PQ_EINVAL;  // an M-bit plain layer
  *out = *d;
  // the derived layer reads the split codes the kernel before it writes
  out->flags = d->flags & ~PQ_LAYER_INPUTS_READY;
  // input channel block i holds activation slice X_i (stored once); each of its
  // codes meets the Gw weight slices of its tap
  out->Cin_g = d->Cin_g * Ga;
  out->wslices = Gw;
  out->bits_a = bits_b;
  out->bits_w = bits_b < 2 ? 2 : bits_b;
  *ga = Ga;
  *gw = Gw;
  return PQ_OK;
}
}  // namespace

pq_status palquant_bitsplit_desc(const pq_layer_desc* d, int32_t bits_b, pq_layer_desc* out) {
  if (out == nullptr) return PQ_EINVAL;
  int Ga, Gw;
  pq_layer_desc t;
  pq_status st = bitsplit_layer(d, bits_b, &t, &Ga, &Gw);
  if (st != PQ_OK) return st;
  ConvParams p;
  st = plan_conv(&t, &p, nullptr, nullptr);
  if (st != PQ_OK) return st;
  *out = t;
  return PQ_OK;
}

size_t palquant_bitsplit_scratch_bytes(const pq_layer_desc* d, int32_t bits_b) {
  pq_layer_desc t;
  if (palquant_bitsplit_desc(d, bits_b, &t) != PQ_OK) return 0;
  return static_cast<size_t>(t.N) * t.H * t.W * t.G * t.Cin_g;
}

pq_status palquant_bitsplit_pack_weight_codes_host(const int8_t* wq_host, const pq_layer_desc* d, int32_t bits_b,
                                                   void* packed_host, size_t packed_bytes) {
  if (wq_host == nullptr || packed_host == nullptr) return PQ_EINVAL;
  int Ga, Gw;
  pq_layer_desc t;
  pq_status st = bitsplit_layer(d, bits_b, &t, &Ga, &Gw);
  if (st != PQ_OK) return st;
  ConvParams p;
  st = plan_conv(&t, &p, nullptr, nullptr);
  if (st != PQ_OK) return st;
  const size_t need = static_cast<size_t>(t.G) * t.Cout_g * t.kh * t.kw * t.Cin_g;
  if (packed_bytes < need) return PQ_EINVAL;
  const int lo = -(1 << (d->bits_w - 1)), hi = (1 << (d->bits_w - 1)) - 1;
  const size_t n_codes = static_cast<size_t>(d->G) * d->Cout_g * d->kh * d->kw * d->Cin_g;
  for (size_t i = 0; i < n_codes; ++i)
    if (wq_host[i] < lo || wq_host[i] > hi) return PQ_EINVAL;
  // Weight slice j of input channel block i (activation slice X_i) holds
  // 2^((i+j)B) w_j (w_j: slice j of w, the lower slices unsigned B-bit, the top
  // one the signed rest), encoded as E4M3 (exact: bitsplit_layer bounded the
  // magnitude).  The derived weights are [Cout][kh][kw][Gw][Ga Cin_g].
  uint8_t* out = static_cast<uint8_t*>(packed_host);
  const int Cin_t = t.Cin_g;
  for_each_packed(p, t.kw * Gw, [&](size_t dst, size_t src) {
    const size_t r = src / Cin_t;                  // (co, kernel position, weight slice)
    const int k = static_cast<int>(src - r * Cin_t);
    const int i = k / d->Cin_g, c = k - i * d->Cin_g;
    const size_t pos = r / Gw;                     // (co, kernel position)
    const int j = static_cast<int>(r - pos * Gw);
    const int w = wq_host[pos * d->Cin_g + c];
    const int wj = (j < Gw - 1) ? ((w >> (j * bits_b)) & ((1 << bits_b) - 1)) : (w >> (j * bits_b));
    out[dst] = e4m3_of_int(wj * (1 << ((i + j) * bits_b)));
  });
  return PQ_OK;
}

pq_status palquant_bitsplit_act(const void* q_dev, void* xs_dev, size_t xs_bytes, const pq_layer_desc* d,
                                int32_t bits_b, pq_stream_t stream) {
  if (q_dev == nullptr || xs_dev == nullptr || !aligned16(q_dev) || !aligned16(xs_dev)) return PQ_EINVAL;
  int Ga, Gw;
  pq_layer_desc t;
  pq_status st = bitsplit_layer(d, bits_b, &t, &Ga, &Gw);
  if (st != PQ_OK) return st;
  const int C = d->G * d->Cin_g;
  if (C % 16 != 0) return PQ_EUNSUPPORTED;
  if (xs_bytes < palquant_bitsplit_scratch_bytes(d, bits_b)) return PQ_EINVAL;
  if (d->code_format == PQ_CODES_C16P2) return PQ_EUNSUPPORTED;  // M-bit codes are one per byte
  if (d->N == 0) return PQ_OK;
  if (d->G != 1) return PQ_EUNSUPPORTED;  // one group: the M-bit layer of Eq. 4
  return pq::launch_bitsplit_act(static_cast<const uint8_t*>(q_dev), static_cast<uint8_t*>(xs_dev), d->N,
                                 static_cast<int64_t>(d->H) * d->W, C, Ga, bits_b,
                                 d->code_format == PQ_CODES_C16 ? 1 : 0, static_cast<cudaStream_t>(stream)) == 0
             ? PQ_OK
             : PQ_ECUDA;
}

pq_status palquant_bitsplit_conv(const void* q_dev, void* xs_dev, size_t xs_bytes, const void* w_packed_dev,
                                 int32_t* acc_dev, const pq_layer_desc* d, int32_t bits_b, pq_stream_t stream) {
  pq_layer_desc t;
  pq_status st = palquant_bitsplit_desc(d, bits_b, &t);
  if (st != PQ_OK) return st;
  st = palquant_bitsplit_act(q_dev, xs_dev, xs_bytes, d, bits_b, stream);
  if (st != PQ_OK) return st;
  return palquant_group_conv(xs_dev, w_packed_dev, acc_dev, &t, stream);
}

pq_status palquant_sync_check(pq_stream_t stream) {
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return PQ_ECUDA;
  unsigned int* word = pq::device_error_word();
  if (word == nullptr) return PQ_ECUDA;
  unsigned int h = 0;
  if (cudaMemcpy(&h, word, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess) return PQ_ECUDA;
  if (h != 0) {
    if (cudaMemset(word, 0, sizeof(h)) != cudaSuccess) return PQ_ECUDA;
    if (cudaDeviceSynchronize() != cudaSuccess) return PQ_ECUDA;
  }
  if (h & PQ_ERR_TIMEOUT) return PQ_ETIMEOUT;
  return PQ_OK;
}

pq_status palquant_set_wait_limit_ns(uint64_t ns) {
  g_wait_limit_ns.store(ns == 0 ? kDefaultWaitLimitNs : ns);
  return PQ_OK;
}

pq_status palquant_watchdog_selftest(uint64_t limit_ns, pq_stream_t stream) {
  if (limit_ns == 0 || limit_ns > 10000000000ull) return PQ_EINVAL;
  unsigned int* word = pq::device_error_word();
  if (word == nullptr) return PQ_ECUDA;
  if (pq::launch_watchdog_selftest(word, limit_ns, static_cast<cudaStream_t>(stream)) != 0) return PQ_ECUDA;
  return palquant_sync_check(stream);
}

pq_status palquant_conv_plan(const pq_layer_desc* d, pq_conv_plan* plan) {
  if (plan == nullptr) return PQ_EINVAL;
  const pq_status st = plan_conv(d, nullptr, plan, nullptr);
  if (st == PQ_OK) plan->pointwise = plan_pointwise(d, nullptr) ? 1 : 0;
  return st;
}

}  // extern "C"
