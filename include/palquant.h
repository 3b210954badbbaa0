/*
 * palquant.h -- C ABI of the GB300 (sm_103a) PalQuant layer library, libpalquant.so.
 *
 * PalQuant (Hu et al., "PalQuant: Accelerating High-precision Networks on
 * Low-precision Accelerators", arXiv 2208.01944) expands a convolution's channels
 * G times, splits them into G groups, quantises every group's activations and
 * weights to B bits and runs a B-bit group convolution (Sec. 4.1).  A cyclic
 * permutation pi(g) = (g + 1) mod G moves each group's output to the next group
 * (Sec. 4.2, Eq. 6-8).  This library runs the inference hot path of one such
 * layer on one GPU:
 *
 *   palquant_quantize_act   activations -> per-group B-bit codes     (Eq. 2)
 *   palquant_group_conv     codes (x) weight codes -> int32 sums      (Sec. 4.1)
 *   palquant_layer_fused    group conv + rescale + shortcut + ReLU + output
 *                           permutation + requantisation, one kernel  (Sec. 3.2,
 *                                                                      4.1, 4.2)
 * plus the set-up calls that produce its inputs (step initialisation, weight
 * quantisation and packing).
 *
 * Conventions that hold for every call:
 *  - Layouts.  Activations, codes and outputs are NHWC, channel c = g*C_g + j
 *    (Sec. 4.2 views [N, C, H, W] as [N, G, C/G, H, W]).  Float weights are
 *    [G][Cout_g][kh][kw][Cin_g].
 *  - Codes.  One code per byte.  Activation codes are unsigned integers in
 *    [0, 2^bits - 1]; weight codes are signed in [-2^(bits-1), 2^(bits-1) - 1].
 *    An activation code tensor is NHWC (PQ_CODES_INT8), channel-blocked
 *    (PQ_CODES_C16) or channel-blocked with 2-bit codes packed four to a byte
 *    (PQ_CODES_C16P2), see pq_code_format; all hold the same integer values.
 *  - Memory.  The caller owns every buffer.  Pointers named *_dev are device
 *    pointers, *_host are host pointers.  The compute calls allocate nothing;
 *    small host arrays (per-group scalars, permutations) are copied into the
 *    launch at call time and may be freed on return.
 *  - Streams.  pq_stream_t is a cudaStream_t (NULL = legacy default stream).
 *    Compute calls are asynchronous on that stream.
 *  - Errors.  Invalid arguments return PQ_EINVAL before anything is launched;
 *    shapes the fast path does not cover return PQ_EUNSUPPORTED; CUDA launch or
 *    runtime failures return PQ_ECUDA.  Every wait inside a kernel is bounded:
 *    a wait that runs out records PQ_ETIMEOUT in a device error word, the kernel
 *    returns, and palquant_sync_check() reports it.
 *  - Devices.  Kernels are built for sm_103a (GB300) only.  Calls act on the
 *    current CUDA device.
 */
#ifndef PALQUANT_H
#define PALQUANT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef void* pq_stream_t; /* a cudaStream_t */

typedef enum {
    PQ_OK = 0,
    PQ_EINVAL = -1,        /* bad argument; nothing launched */
    PQ_EUNSUPPORTED = -2,  /* valid but outside the implemented shapes */
    PQ_ECUDA = -3,         /* a CUDA call failed */
    PQ_ETIMEOUT = -4       /* a bounded in-kernel wait ran out */
} pq_status;

typedef enum {
    PQ_CODES_INT8 = 0, /* code v stored as the byte v, NHWC: byte (((n*H + h)*W + w)*C + c) */
    PQ_CODES_E4M3 = 1, /* reserved (PQ_EUNSUPPORTED) */
    PQ_CODES_C16 = 2,  /* code v stored as the byte v, channel-blocked in 16-channel blocks:
                          byte ((((n*(C/16) + c/16)*H + h)*W + w)*16 + c%16).  C % 16 == 0.
                          The tensor cores' operand layout: every run of positions of one
                          16-channel block is contiguous. */
    PQ_CODES_C16P2 = 3, /* 2-bit codes packed four to a byte, channel-blocked: the 16 codes of
                          a position and 16-channel block form one little-endian 32-bit word
                          at byte ((((n*(C/16) + c/16)*H + h)*W + w)*4), code of channel c at
                          bits 2 (c % 16).  bits <= 2, C % 16 == 0; as a layer input it needs
                          stride 1 and W % 4 == 0 (H W % 4 == 0 for 1x1 layers).  A quarter
                          of the bytes of PQ_CODES_C16. */
    PQ_CODES_C32F4 = 4  /* 2-bit codes as packed FP4: two to a byte, channel-blocked in
                          32-channel blocks of 16 bytes per position; code of channel c in the
                          4 bits at byte ((((n*(C/32) + c/32)*H + h)*W + w)*16 + (c%32)/2),
                          low nibble for even c, high nibble for odd c.  A code v <= 3 is the
                          FP4 E2M1 encoding of v/2, so the layer's block-scaled FP4 tensor-core
                          path reads it in place.  bits <= 2, C % 32 == 0; as a layer format it
                          also needs Cin_g % 64 == 0, Cout_g % 32 == 0, bits_w <= 3, and no
                          channel shuffle.  Half the bytes of PQ_CODES_C16. */
} pq_code_format;

/* Output channel permutation (Sec. 4.2).  kind:
 *   0  none
 *   1  cyclic: source group g goes to group (g + shift) mod G; Eq. 6 is shift = 1
 *   2  channel shuffle (ShuffleNet, used at block ends in Sec. 4.3): source channel
 *      g*Cout_g + j goes to channel j*G + g
 *   3  explicit group permutation: group g goes to group perm[g] (host array of G)
 * Kinds 0, 1 and 3 must describe a permutation of the G groups, else PQ_EINVAL. */
typedef struct {
    int32_t kind;
    int32_t shift;
    const int32_t* perm;
} pq_shuffle;

/* One PalQuant layer.  Input [N, H, W, G*Cin_g] codes, weights
 * [G][Cout_g][kh][kw][Cin_g], output [N, Ho, Wo, G*Cout_g] with
 * Ho = (H + 2 pad - kh) / stride + 1 and Wo likewise.  Zero padding is code 0
 * (exact because the activation quantiser's lower bound l is 0, Eq. 2). */
typedef struct {
    int32_t N, H, W;
    int32_t G;
    int32_t Cin_g, Cout_g;
    int32_t kh, kw;
    int32_t stride, pad;
    int32_t bits_a;      /* activation code bits, 1..4 */
    int32_t bits_w;      /* weight code bits, 2..4 */
    int32_t bits_out;    /* requantised output code bits, 1..4 */
    int32_t relu;        /* 1: ReLU after the rescale (and the shortcut add) */
    int32_t code_format; /* pq_code_format of the input codes and the output codes */
    int32_t flags;       /* PQ_LAYER_* bits; 0 for none */
    int32_t wslices;     /* weight slices per input channel and tap: 0 or 1 for a plain
                            layer.  R > 1 (set by palquant_bitsplit_desc, 2..8) makes
                            every input code meet R weight codes, the sum running over
                            them: acc = sum_{tap, r, ci} q[...] w[g, co, tap, r, ci],
                            weights [G][Cout_g][kh][kw][R][Cin_g] (Eq. 4's G^2 products
                            with each activation slice stored once) */
} pq_layer_desc;

/* pq_layer_desc.flags bit: the kernel launched on the stream immediately before this
 * call writes neither this layer's input (codes or fp32 activations) nor its packed
 * weights, e.g. consecutive layers over independent batches.  The layer kernel then
 * starts loading them and computing on them while that kernel's last blocks still
 * run; its stores (and its reads of the shortcut) still wait for that kernel to
 * complete.  The caller answers for the promise: a layer
 * that consumes the previous kernel's output (the next layer of a network) must
 * leave the bit clear, and then every access waits.  Kernels launched earlier
 * than that one have completed before the loads start (each layer kernel lets its
 * dependent launch start only after its own wait for the kernel before it), so a
 * layer may read what a layer two launches back wrote.  Under the bit, the time
 * the previous kernel still runs counts against the in-kernel wait limit
 * (palquant_set_wait_limit_ns) of the waits that depend on it.  Other bits:
 * PQ_EINVAL. */
#define PQ_LAYER_INPUTS_READY 1

/* Human-readable name of a status. */
const char* palquant_strerror(pq_status s);

/* Library version, major*10000 + minor*100 + patch. */
int palquant_version(void);

/* ------------------------------------------------------------------------ */
/* Set-up: step initialisation and epilogue multipliers (untimed).          */
/* ------------------------------------------------------------------------ */

/* Bytes of device scratch palquant_act_steps needs for a tensor of P = N*H*W
 * pixels and G groups. */
size_t palquant_act_steps_scratch_bytes(int64_t P, int32_t G);

/* Per-group activation step s[g] = 2 mean(x_g) / sqrt(2^bits - 1): the LSQ step
 * initialisation the paper's training follows (Sec. 5, "Training Details";
 * Eq. 2 with l = 0, u = s (2^bits - 1)).  x_dev is NHWC fp32 [N,H,W,G*Cg]; the
 * mean runs over every element of the group, summed in double in a fixed order
 * (deterministic), and the step is rounded to float once.  scratch_dev must hold
 * palquant_act_steps_scratch_bytes(N*H*W, G) bytes.  s_out_host receives G
 * floats.  Synchronises the stream. */
pq_status palquant_act_steps(const float* x_dev, int64_t N, int32_t H, int32_t W, int32_t G, int32_t Cg,
                             int32_t bits, void* scratch_dev, size_t scratch_bytes, float* s_out_host,
                             pq_stream_t stream);

/* The same per-group activation steps as palquant_act_steps, for callers that
 * cannot allocate device memory (for example code whose device memory is owned
 * by a host framework, or a path whose memory budget is fixed in advance).  The
 * paper has no counterpart: this is a deployment convenience.
 *
 * It allocates nothing.  Its scratch is a fixed array of 131,584 bytes in the
 * library's own device memory (held by every GPU that loads the library until
 * the process exits), which bounds the group count: G <= 64, else
 * PQ_EUNSUPPORTED.  The first call on a device looks up that array's device
 * address and caches it for the process (make that call before any stream
 * capture); the cached address does not survive cudaDeviceReset, so do not call
 * this entry point on a device after resetting it.  All calls share the array and
 * overwrite what they read, so calls that run on the GPU at the same time race
 * and must be serialised by the caller.  Results are identical to
 * palquant_act_steps for the same input.  Synchronises the stream. */
pq_status palquant_act_steps_noalloc(const float* x_dev, int64_t N, int32_t H, int32_t W, int32_t G, int32_t Cg,
                                     int32_t bits, float* s_out_host, pq_stream_t stream);

/* Per-group weight step s_w[g] = 2 mean|w_g| / sqrt(2^(bits-1) - 1) (LSQ), mean
 * in double over the group's weights; w_host is [G][Cout_g][kh][kw][Cin_g].
 * Host only.  s_w_out_host receives G floats. */
pq_status palquant_weight_steps(const float* w_host, const pq_layer_desc* d, float* s_w_out_host);

/* Epilogue multipliers (Sec. 3.2: the output scale alpha multiplies the layer's
 * output; the requantised code of source group g lands in group dst(g) of the
 * next layer and uses that group's step):
 *   m_out[g] = fl(s_w[g] s_a[g] alpha)
 *   m_req[g] = fl(s_w[g] s_a[g] alpha / s_next[dst(g)])       (s_next may be NULL)
 * computed in double and rounded once.  Host only. */
pq_status palquant_epilogue_scales(int32_t G, const float* s_w_host, const float* s_a_host, double alpha,
                                   const float* s_next_host, pq_shuffle shuf, float* m_out_host,
                                   float* m_req_host);

/* ------------------------------------------------------------------------ */
/* Set-up: weight quantisation and packing (untimed).                       */
/* ------------------------------------------------------------------------ */

/* Size of the packed weight operand of a layer (opaque, tensor-core layout). */
size_t palquant_packed_weight_bytes(const pq_layer_desc* d);

/* Quantise float weights to signed codes per group,
 *   w_q = clamp(rint(w * inv_sw[g]), -2^(bits_w-1), 2^(bits_w-1) - 1)
 * (one fp32 multiply, round half to even; Eq. 2 in LSQ's signed form), and
 * write the packed operand to packed_host (palquant_packed_weight_bytes bytes).
 * Host only. */
pq_status palquant_pack_weights_host(const float* w_host, const pq_layer_desc* d, const float* inv_sw_host,
                                     void* packed_host, size_t packed_bytes);

/* The paper's own weight quantiser (Sec. 3.2: Eq. 2 with the clip range
 * [-u[g], u[g]] and Eq. 3's de-quantised weight 2 (x_q / (2^b - 1) - 0.5)):
 *   x_q = clamp(rint((w + u[g]) * k[g]), 0, 2^b - 1), k[g] = fl((2^b - 1) / (2 u[g])),
 *   code = 2 x_q - (2^b - 1)
 * (one fp32 add and one fp32 multiply), i.e. the odd levels -3, -1, 1, 3 at
 * b = 2 instead of the LSQ range [-2^(b-1), 2^(b-1) - 1]; the de-quantised
 * weight is code * u[g] / (2^b - 1), so its epilogue scale uses
 * s_w = u / (2^b - 1).  Packed like palquant_pack_weights_host (same size).
 * u_host: G positive floats.  PQ_EUNSUPPORTED when the larger codes could
 * make a sum reach 2^24.  Host only. */
pq_status palquant_pack_weights_odd_host(const float* w_host, const pq_layer_desc* d, const float* u_host,
                                        void* packed_host, size_t packed_bytes);

/* The same, with the packed operand copied to device memory on `stream`
 * (synchronises the stream before returning so w_host may be freed). */
pq_status palquant_pack_weights(const float* w_host, const pq_layer_desc* d, const float* inv_sw_host,
                                void* packed_dev, size_t packed_bytes, pq_stream_t stream);

/* Pack already-quantised signed weight codes wq_host [G][Cout_g][kh][kw][Cin_g]
 * (each in the bits_w range, else PQ_EINVAL).  Host only. */
pq_status palquant_pack_weight_codes_host(const int8_t* wq_host, const pq_layer_desc* d, void* packed_host,
                                          size_t packed_bytes);

/* Inverse of the packing: recover the signed codes from a packed operand. */
pq_status palquant_unpack_weight_codes_host(const void* packed_host, const pq_layer_desc* d, int8_t* wq_host);

/* ------------------------------------------------------------------------ */
/* Hot path.                                                                */
/* ------------------------------------------------------------------------ */

/* Group-wise activation quantisation (Eq. 2 with l = 0, u = s (2^bits - 1); one
 * fp32 multiply, round half to even, clamp):
 *   q[p, g*Cg + j] = clamp(rint(x[p, g*Cg + j] * inv_s[g]), 0, 2^bits - 1)
 * x_dev is NHWC fp32 [N,H,W,G*Cg]; q_dev receives one byte per element in
 * code_format (PQ_CODES_INT8: NHWC; PQ_CODES_C16: channel-blocked, needs
 * Cg % 16 == 0; PQ_CODES_C16P2: channel-blocked 2-bit codes four to a byte,
 * needs Cg % 16 == 0 and bits <= 2; PQ_CODES_C32F4: 2-bit codes two to a byte
 * in 32-channel blocks, needs Cg % 16 == 0, G*Cg % 32 == 0 and bits <= 2).  inv_s_host holds G floats (fl(1/s) of the steps), copied at
 * call time.  NaN maps to 0 and +inf to 2^bits - 1.  bits in 1..8. */
pq_status palquant_quantize_act(const float* x_dev, void* q_dev, int64_t N, int32_t H, int32_t W, int32_t G,
                                int32_t Cg, int32_t bits, int32_t code_format, const float* inv_s_host,
                                pq_stream_t stream);

/* B-bit group convolution (Sec. 3.1 Eq. 1 lowered per group; Sec. 4.1):
 *   acc[n,oh,ow,g*Cout_g+co] = sum_{kh,kw,ci} q[n, oh*s-p+kh, ow*s-p+kw, g*Cin_g+ci]
 *                                             * w_q[g,co,kh,kw,ci]
 * exact in int32 (every product and partial sum is an integer below 2^24).
 * q_dev holds codes in d->code_format; w_packed_dev comes from
 * palquant_pack_weights for the same d; acc_dev is int32 NHWC.  No permutation. */
pq_status palquant_group_conv(const void* q_dev, const void* w_packed_dev, int32_t* acc_dev,
                              const pq_layer_desc* d, pq_stream_t stream);

/* The whole layer in one kernel (Sec. 3.2, 4.1, 4.2).  For every output pixel
 * and source channel (g, co) with acc the group-conv sum above:
 *   y = (float)acc * m_out[g]
 *   y = y + shortcut[pixel, g*Cout_g + co]        if shortcut_dev != NULL
 *   y = max(y, 0)                                  if d->relu
 *   t = shortcut_dev ? y : (float)acc
 *   q = clamp(rint(t * m_req[g]), 0, 2^bits_out - 1)
 * and acc, y, q are written at the destination channel of (g, co) under shuf.
 * m_out_host, m_req_host: G floats each (m_req may be NULL only when
 * q_out_dev is NULL).  Any of acc_out_dev (int32), y_out_dev (fp32) and
 * q_out_dev (codes in d->code_format) may be NULL, but not all three.
 * shortcut_dev is fp32 NHWC with the output's shape.  Float products and sums
 * are single IEEE fp32 operations in the order written. */
pq_status palquant_layer_fused(const void* q_dev, const void* w_packed_dev, const pq_layer_desc* d,
                               const float* m_out_host, const float* m_req_host, pq_shuffle shuf,
                               const float* shortcut_dev, int32_t* acc_out_dev, float* y_out_dev,
                               void* q_out_dev, pq_stream_t stream);

/* The activation quantiser and the whole layer in one kernel (Sec. 3.2 Eq. 2,
 * then as palquant_layer_fused): the layer's input is the fp32 NHWC activation
 * tensor x_dev [N, H, W, G*Cin_g] instead of codes, quantised as it is loaded,
 *   q[p, g*Cin_g + j] = clamp(rint(x[p, g*Cin_g + j] * inv_s[g]), 0, 2^bits_a - 1)
 * (one fp32 multiply, round half to even, NaN -> 0; the codes palquant_quantize_act
 * produces), so the codes never pass through memory.  inv_s_host: G floats
 * (fl(1/s) of the input steps, >= 0), copied at call time.  Everything else as
 * palquant_layer_fused: w_packed_dev comes from palquant_pack_weights for the same
 * d, whose code_format (PQ_CODES_INT8, PQ_CODES_C16, or PQ_CODES_C32F4 with its
 * constraints) is the output codes'.  Needs stride 1 and 16-byte aligned x_dev;
 * other shapes return PQ_EUNSUPPORTED. */
pq_status palquant_quantize_layer_fused(const float* x_dev, const float* inv_s_host, const void* w_packed_dev,
                                        const pq_layer_desc* d, const float* m_out_host, const float* m_req_host,
                                        pq_shuffle shuf, const float* shortcut_dev, int32_t* acc_out_dev,
                                        float* y_out_dev, void* q_out_dev, pq_stream_t stream);

/* Inference quantisers with learned per-group bounds l[g] < u[g] (Eq. 2 as the
 * paper trains it, Sec. 5): the codes of palquant_fake_quant_forward,
 *   code = rint(min(max((x - l) * fl(1 / fl(u - l)), 0), 1) * (2^bits - 1))
 * (one fp32 rounding per operation, NaN -> 0), so a layer trained with those
 * kernels runs on exactly the codes its training forward used.  l_host and u_host
 * hold G finite floats each (PQ_EINVAL otherwise).  Otherwise as
 * palquant_quantize_act (all code formats) and palquant_quantize_layer_fused; in
 * the fused form the out-of-image positions of the zero padding are code 0 for any
 * l (the fp32 tiles are NaN-filled there). */
pq_status palquant_quantize_act_lu(const float* x_dev, void* q_dev, int64_t N, int32_t H, int32_t W, int32_t G,
                                   int32_t Cg, int32_t bits, int32_t code_format, const float* l_host,
                                   const float* u_host, pq_stream_t stream);
pq_status palquant_quantize_layer_fused_lu(const float* x_dev, const float* l_host, const float* u_host,
                                           const void* w_packed_dev, const pq_layer_desc* d, const float* m_out_host,
                                           const float* m_req_host, pq_shuffle shuf, const float* shortcut_dev,
                                           int32_t* acc_out_dev, float* y_out_dev, void* q_out_dev,
                                           pq_stream_t stream);

/* Cyclic shuffle module (Sec. 4.2, Eq. 9-10), fused into one kernel:
 *   Y = CyclicPermute(X):  Y[:, pi(i)] = X[:, i] with pi(i) = (i + shift) mod G (Eq. 8,
 *                          group-level; Eq. 6 for shift = 1)
 *   Z = X + Conv1x1(Y)     the 1x1 B-bit group convolution of the permuted codes,
 *                          rescaled (m_out), plus the fp32 X, then ReLU if d->relu.
 * The permutation is not a data movement: conv group g reads input group
 * pi^-1(g) = (g - shift) mod G.  q_dev holds X's codes in d->code_format;
 * x_dev is X in fp32 NHWC (the short-cut); z_out_dev (fp32 NHWC, nullable)
 * receives Z and q_out_dev (nullable, d->code_format) Z's codes for the next
 * layer, clamp(rint(z * m_req[g]), 0, 2^bits_out - 1) (m_req is then the next
 * layer's fl(1/s) of group g, no permutation after the module).  d must be a
 * 1x1, stride-1, pad-0 layer with Cin_g == Cout_g (PQ_EINVAL otherwise); at
 * least one output.  Other conventions as palquant_layer_fused. */
pq_status palquant_cyclic_shuffle_module(const void* q_dev, const void* w_packed_dev, const pq_layer_desc* d,
                                         const float* m_out_host, const float* m_req_host, int32_t shift,
                                         const float* x_dev, float* z_out_dev, void* q_out_dev, pq_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Failure detection.                                                       */
/* ------------------------------------------------------------------------ */

/* Synchronise `stream`, then read and clear the device error word of the
 * current device.  Returns PQ_ETIMEOUT if any kernel's bounded wait ran out
 * since the last check, PQ_ECUDA on a CUDA error, else PQ_OK. */
pq_status palquant_sync_check(pq_stream_t stream);

/* Limit, in nanoseconds, of every in-kernel wait of kernels launched after this
 * call (default 2e9).  0 restores the default. */
pq_status palquant_set_wait_limit_ns(uint64_t ns);

/* Launch a one-CTA kernel whose barrier wait nobody completes, with the given
 * wait limit, and return palquant_sync_check()'s verdict (PQ_ETIMEOUT when the
 * watchdog works).  The kernel ends by itself; the context stays usable. */
pq_status palquant_watchdog_selftest(uint64_t limit_ns, pq_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Bit-level decomposition (Sec. 3.3, Eq. 4): the baseline PalQuant is        */
/* compared with.  An M-bit layer on B-bit hardware runs as the G^2 products  */
/* of B-bit slices, G = ceil(M / B), each shifted by 2^((i + j) B):           */
/*   Y = sum_i sum_j X_i W_j^T 2^((i + j) B)                                 */
/* with x = sum_i X_i 2^(iB), X_i in [0, 2^B - 1], and w = sum_j W_j 2^(jB),   */
/* the lower weight slices unsigned B-bit and the top one the signed rest.     */
/* Here the G^2 products form the K dimension of one tensor-core pass: the    */
/* input channels are the slice pairs (i, j), block (i Gw + j) carrying X_i,   */
/* and the packed weight block (i, j) holds 2^((i+j)B) W_j.  The result equals */
/* palquant_group_conv of the M-bit layer exactly.                             */
/*                                                                            */
/* d describes the M-bit layer (bits_a = M_a, bits_w = M_w, one group:        */
/* d->G == 1, codes one per byte, G * Cin_g % 16 == 0).  bits_b in 1..4.      */
/* Shapes whose shifted weight slices are not exact E4M3 values (beyond      */
/* (2^B - 1) 2^((Ga - 1 + Gw - 1) B) = 448, e.g. 6-bit on 2-bit hardware) or   */
/* whose M-bit sums could reach 2^24 return PQ_EUNSUPPORTED.                   */
/* ------------------------------------------------------------------------ */

/* The decomposed layer's descriptor: Cin_g multiplied by Ga (the activation
 * slices, each stored once), wslices = Gw (every slice meets the Gw shifted
 * weight slices), bits_a = B, PQ_LAYER_INPUTS_READY cleared (the decomposed layer
 * reads the slices that the kernel launched just before it writes). */
pq_status palquant_bitsplit_desc(const pq_layer_desc* d, int32_t bits_b, pq_layer_desc* out);

/* Bytes of the slice buffer (N H W Ga Cin_g); 0 if unsupported. */
size_t palquant_bitsplit_scratch_bytes(const pq_layer_desc* d, int32_t bits_b);

/* Pack the decomposed weights from the M-bit signed codes wq_host
 * ([G][Cout_g][kh][kw][Cin_g], in [-2^(M_w-1), 2^(M_w-1) - 1], else PQ_EINVAL)
 * into packed_host (palquant_packed_weight_bytes of the decomposed
 * descriptor).  Host only. */
pq_status palquant_bitsplit_pack_weight_codes_host(const int8_t* wq_host, const pq_layer_desc* d, int32_t bits_b,
                                                   void* packed_host, size_t packed_bytes);

/* Slice the M-bit activation codes q_dev (d->code_format) into xs_dev (same
 * format, the decomposed layer's input; xs_bytes >= the scratch size). */
pq_status palquant_bitsplit_act(const void* q_dev, void* xs_dev, size_t xs_bytes, const pq_layer_desc* d,
                                int32_t bits_b, pq_stream_t stream);

/* Eq. 4 end to end: palquant_bitsplit_act into xs_dev, then the decomposed
 * convolution into acc_dev (int32 NHWC, as palquant_group_conv of d). */
pq_status palquant_bitsplit_conv(const void* q_dev, void* xs_dev, size_t xs_bytes, const void* w_packed_dev,
                                 int32_t* acc_dev, const pq_layer_desc* d, int32_t bits_b, pq_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Full-precision layers around the PalQuant body of a network.  The paper   */
/* keeps the first and the last layer in full precision (Sec. 5); these are  */
/* not part of the PalQuant method itself.  Each output is summed in one     */
/* fixed order, with one fused multiply-add (a single IEEE rounding) per     */
/* term, so values do not depend on the launch shape.  All tensors are fp32  */
/* device buffers owned by the caller; calls are asynchronous on `stream`.   */
/* ------------------------------------------------------------------------ */

/* Direct convolution: x NHWC [N,H,W,Cin], w [Cout][k][k][Cin], y NHWC
 * [N,Ho,Wo,Cout] (16-byte aligned) with Ho = (H + 2 pad - k) / stride + 1.
 * y[n,oh,ow,co] = fma-sum over (kh, kw, ci) in that order, starting from 0, of
 * x[n, oh*stride - pad + kh, ow*stride - pad + kw, ci] * w[co,kh,kw,ci], taps
 * outside the image skipped (zero padding); then max(y, 0) if relu.  Cout must
 * be a multiple of 16; pad < k.  PQ_EINVAL otherwise. */
pq_status palquant_conv2d_f32(const float* x_dev, const float* w_dev, float* y_dev, int64_t N, int32_t H, int32_t W,
                              int32_t Cin, int32_t Cout, int32_t k, int32_t stride, int32_t pad, int32_t relu,
                              pq_stream_t stream);

/* The network's first layer and the pooling after it in one pass (Sec. 5 keeps
 * the first layer in full precision): stem = max(conv2d_f32(x, w, stride 2,
 * pad 3, 7 x 7), 0) exactly as palquant_conv2d_f32 with relu computes it, and
 * pool = palquant_maxpool2d_f32(stem, 3 x 3, stride 2, pad 1).  x NHWC
 * [N,H,W,3], w [Cout][7][7][3], pool NHWC [N,Hp,Wp,Cout] with Ho = (H - 1) / 2 + 1,
 * Hp = (Ho - 1) / 2 + 1 (likewise W); stem_dev, NHWC [N,Ho,Wo,Cout], may be NULL
 * (the stem output is then never written to memory).  Outputs 16-byte aligned.
 * The call zeroes pool on the stream first (windows that span two tiles of the
 * kernel are combined by atomic maxima); the result is exact, so it equals the
 * two separate calls bit for bit.  Cout must be 128 (PQ_EUNSUPPORTED otherwise:
 * use the two calls); PQ_EINVAL on bad sizes or pointers. */
pq_status palquant_stem_pool_f32(const float* x_dev, const float* w_dev, float* stem_dev, float* pool_dev, int64_t N,
                                 int32_t H, int32_t W, int32_t Cout, pq_stream_t stream);

/* Max pooling, NHWC: y[n,oh,ow,c] = max over the in-image taps of the k x k
 * window at (oh*stride - pad, ow*stride - pad) (padding taps are ignored);
 * pad < k. */
pq_status palquant_maxpool2d_f32(const float* x_dev, float* y_dev, int64_t N, int32_t H, int32_t W, int32_t C,
                                 int32_t k, int32_t stride, int32_t pad, pq_stream_t stream);

/* Global average pooling: y[n,c] = (sum over h, w in storage order of
 * x[n,h,w,c]) / (H W), x NHWC, y [N,C]. */
pq_status palquant_avgpool_f32(const float* x_dev, float* y_dev, int64_t N, int32_t H, int32_t W, int32_t C,
                               pq_stream_t stream);

/* Fully connected layer without bias: y[n,o] = fma-sum over i in order of
 * x[n,i] w[o,i]; x [N,Cin], w [Cout][Cin], y [N,Cout]. */
pq_status palquant_linear_f32(const float* x_dev, const float* w_dev, float* y_dev, int64_t N, int32_t Cin,
                              int32_t Cout, pq_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Quantisation-aware training of the quantiser (Sec. 3.2 Eq. 2-3, Sec. 5).  */
/* ------------------------------------------------------------------------ */

/* Fake quantisation with learned per-group bounds (the training-time form of
 * Eq. 2-3; Sec. 5 learns l and u through back-propagation).  x_dev is
 * [P][G*Cg] fp32 (group g = channel / Cg: NHWC activations with P = N*H*W, or
 * weights with P = 1 and Cg = the group's weight count); l_host, u_host hold G
 * floats with l[g] < u[g] (finite).  Per element, in fp32 with one rounding per
 * operation and the divisions taken as multiplies by fp32 reciprocals:
 *   t   = (x - l) * fl(1 / fl(u - l)),   x_n = min(max(t, 0), 1)   (NaN -> 0)
 *   x_q = rint(x_n * (2^bits - 1))                                 (half to even)
 *   kind 0 (activations): xhat = x_q * fl(1 / (2^bits - 1))              in [0, 1]
 *   kind 1 (weights):     xhat = 2 * (x_q * fl(1 / (2^bits - 1)) - 0.5)  in [-1, 1]
 * (Eq. 3 is printed with its two cases swapped; the activations are the
 * non-negative ones.)  Requires Cg % 4 == 0, 16-byte aligned pointers,
 * 1 <= bits <= 8, G <= 64 and P * Cg / 4 < 2^32 (else PQ_EUNSUPPORTED); P = 0
 * does nothing.  Bound by HBM: 8 bytes per element.  Asynchronous on the
 * stream. */
pq_status palquant_fake_quant_forward(const float* x_dev, float* xhat_dev, int64_t P, int32_t G, int32_t Cg,
                                      int32_t bits, int32_t kind, const float* l_host, const float* u_host,
                                      pq_stream_t stream);

/* Bytes of device scratch palquant_fake_quant_backward needs (16-byte aligned). */
size_t palquant_fake_quant_scratch_bytes(int64_t P, int32_t G, int32_t Cg);

/* Its backward with the straight-through estimator: the rounding passes the
 * gradient unchanged, the clip does not.  With c = 1 (kind 0) or 2 (kind 1),
 * r = u - l and t as in the forward:
 *   dx[i] = dy[i] * (c * fl(1 / fl(r)))     if 0 < t < 1, else 0    (fp32)
 *   dl[g] =  c / r^2 * sum over group g's elements with 0 < t < 1 of dy * (x - u)
 *   du[g] = -c / r^2 * sum over the same elements of dy * (x - l)
 * dl_dev and du_dev receive G doubles each (device).  The sums take each product
 * in fp32, add four in fp32, accumulate a thread's share in a compensated fp32
 * sum and the threads in double, over a partition fixed by the problem size, so
 * they are deterministic; their error is below 1e-6 of
 * c / r^2 * sum |dy (x - u)| (resp. |dy (x - l)|).  Bound by HBM: 12 bytes per
 * element.  Same requirements as the forward; scratch_dev holds
 * palquant_fake_quant_scratch_bytes(P, G, Cg) bytes.  P = 0 gives zero
 * gradients (the element pointers and the scratch may then be NULL).
 * Asynchronous. */
pq_status palquant_fake_quant_backward(const float* x_dev, const float* dy_dev, float* dx_dev, double* dl_dev,
                                       double* du_dev, int64_t P, int32_t G, int32_t Cg, int32_t bits, int32_t kind,
                                       const float* l_host, const float* u_host, void* scratch_dev,
                                       size_t scratch_bytes, pq_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Introspection (host only; no GPU needed).                                */
/* ------------------------------------------------------------------------ */

/* How the tensor-core kernel tiles a layer.  Filled by palquant_conv_plan. */
typedef struct {
    int32_t supported;     /* 1 if the tensor-core kernel runs this layer */
    int32_t mode;          /* 0 flat pixels (1x1, stride 1, pad 0), 1 rows of whole image rows */
    int32_t rows_per_tile; /* output rows per tile (mode 1) */
    int32_t m_tiles;       /* 128-row accumulators per tile */
    int32_t tile_pitch;    /* positions per tile row in shared memory */
    int32_t n_block;       /* output channels per accumulator (MMA N) */
    int32_t n_blocks;      /* output-channel blocks per group */
    int32_t k_chunk;       /* input channels per K block */
    int32_t k_blocks;      /* K blocks per tap */
    int32_t taps;          /* kh*kw */
    int32_t weights_resident; /* 1 if a group's weights stay in shared memory */
    int32_t acc_stages;    /* tensor-memory accumulator buffers */
    int32_t smem_bytes;    /* dynamic shared memory per CTA of a call that stages its
                              outputs; a call writing channel-blocked codes only (no
                              int32 or fp32 outputs, no shortcut) reserves no per-warp
                              staging and launches with less */
    int64_t tiles;         /* tiles per (group, n-block) unit */
    int64_t work_items;    /* tiles * G * n_blocks */
    int32_t pointwise;     /* 1 if a call writing channel-blocked codes only (no int32 or
                              fp32 outputs, no shortcut, no channel shuffle, codes in)
                              runs on the pointwise kernel (1x1 layers); the fields above
                              describe the general kernel */
} pq_conv_plan;

pq_status palquant_conv_plan(const pq_layer_desc* d, pq_conv_plan* plan);

#ifdef __cplusplus
}
#endif

#endif /* PALQUANT_H */
