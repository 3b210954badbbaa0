/*
 * PalQuant CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously correct CPU statement of what one PalQuant
 * parallel low-precision convolution layer computes at inference time.
 * Only the test suite, the package smoke check and the benchmark's CPU
 * baseline leg may load this file.  It shares no code, header, table or
 * constant with the GPU library; the GPU library never loads it.
 *
 * Every function names the passage of the paper (Hu et al., "PalQuant:
 * Accelerating High-precision Networks on Low-precision Accelerators",
 * arXiv 2208.01944) it follows.  Notation: activations are NHWC, channel
 * c = g*Cg + j for group g in [0,G) and j in [0,Cg) (Sec. 4.2 reshapes
 * [N,C,H,W] into [N,G,C/G,H,W]); weights are [G][Cout_g][kh][kw][Cin_g].
 *
 * Readings of the paper that this file takes (each one is listed with its
 * reason in the design notes):
 *   - Eq. 2 with l = 0 and u = s*Qp for activations (LSQ step form, Sec. 5
 *     training details): x_q = round(clip(x/s, 0, Qp)).  Because the clip
 *     bounds are integers, rounding first and clipping second gives the same
 *     code, and the division is replaced by one fp32 multiply with
 *     inv_s = fl(1/s) so both implementations make the same fp32 decision.
 *   - round-to-nearest of Eq. 2 is taken as round-half-to-even (rintf).
 *   - signed weight codes in [-2^(b-1), 2^(b-1)-1] (LSQ convention).
 *   - the cyclic permutation of Eq. 6-8 is applied to the output of the
 *     group convolution: output group g is written to group pi(g) with
 *     pi(g) = (g + 1) mod G (Eq. 6, Eq. 8: Y[:, pi(i)] = X[:, i]).
 *
 * Parity status of each function (what pins it, see tests/test_oracle_*.py):
 *   oracle_quantize_act      pinned (hand rounding cases, code range, closed
 *                            forms)
 *   oracle_quantize_weights  pinned (hand cases, code range)
 *   oracle_quantize_weights_odd  pinned (hand cases, odd levels, monotone,
 *                            the clip bounds)
 *   oracle_quantize_act_lu   pinned (hand cases; equal to the codes of the
 *                            training forward)
 *   oracle_fake_quant_fwd /
 *   oracle_fake_quant_bwd    pinned (hand cases, levels, monotone; the
 *                            straight-through gradients against central
 *                            differences of the unrounded quantiser in
 *                            float64; shift and scale invariance of Eq. 2's
 *                            normalisation)
 *   oracle_group_conv        pinned (float64 library convolution on codes,
 *                            brute-force dequantised conv, 1x1 = matmul,
 *                            all-max closed form, G = 1 case)
 *   oracle_epilogue          pinned (hand cases, Eq. 8 = torch.roll on the
 *                            group axis, inverse permutation round trip)
 *   oracle_act_step /
 *   oracle_weight_step       pinned (half-normal / Gaussian closed forms,
 *                            statistical)
 *   oracle_epilogue_scales   pinned (hand cases)
 *   oracle_conv2d_f32,
 *   oracle_maxpool_f32,
 *   oracle_avgpool_f32,
 *   oracle_linear_f32        pinned (float64 library convolution / pooling /
 *                            matmul within the fp32 error bound; hand cases;
 *                            max pooling exactly)
 *
 * The full-precision functions serve the ResNet-18-shaped network around the
 * PalQuant layers (the paper keeps the first and the last layer in full
 * precision, Sec. 5).  Each sums in one fixed order with one fused
 * multiply-add per term (fmaf, a single IEEE rounding), so that the values
 * feeding the next quantiser are defined to the bit.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* Number of OpenMP threads the oracle uses (1 when built without OpenMP). */
int oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_num_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* ---------------------------------------------------------------------- */
/* Sec. 3.2, Eq. 2: uniform quantizer for activations.                     */
/* x_n = clip((x - l)/(u - l), 0, 1), x_q = round((2^b - 1) x_n) with      */
/* l = 0, u = s (2^b - 1):  x_q = clamp(rint(x * inv_s), 0, 2^b - 1).       */
/* ---------------------------------------------------------------------- */
static uint8_t quantize_unsigned(float x, float inv_s, int qmax) {
    float t = x * inv_s;              /* one fp32 multiply */
    float r = rintf(t);               /* round half to even */
    r = fmaxf(r, 0.0f);               /* NaN -> 0 */
    r = fminf(r, (float)qmax);
    return (uint8_t)(int)r;
}

/* Quantize an NHWC fp32 activation tensor per group (Sec. 4.1: "quantize
 * the activations ... to B-bit in each group").  inv_s has G entries. */
void oracle_quantize_act(const float* x, uint8_t* q, int64_t N, int64_t H, int64_t W,
                         int G, int Cg, int bits, const float* inv_s) {
    const int64_t C = (int64_t)G * Cg;
    const int64_t P = N * H * W;
    const int qmax = (1 << bits) - 1;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < P; ++p) {
        for (int64_t c = 0; c < C; ++c) {
            int g = (int)(c / Cg);
            q[p * C + c] = quantize_unsigned(x[p * C + c], inv_s[g], qmax);
        }
    }
}

/* Signed weight codes in [-2^(b-1), 2^(b-1) - 1], one fp32 multiply by
 * inv_sw[g], round half to even, clamp (Eq. 2 in LSQ's signed form). */
void oracle_quantize_weights(const float* w, int8_t* wq, int G, int Cout_g, int kh, int kw,
                             int Cin_g, int bits, const float* inv_sw) {
    const int64_t per_group = (int64_t)Cout_g * kh * kw * Cin_g;
    const int qmax = (1 << (bits - 1)) - 1;
    const int qmin = -(1 << (bits - 1));
    for (int g = 0; g < G; ++g) {
        for (int64_t i = 0; i < per_group; ++i) {
            float t = w[g * per_group + i] * inv_sw[g];
            float r = rintf(t);
            r = fmaxf(r, (float)qmin);
            r = fminf(r, (float)qmax);
            wq[g * per_group + i] = (int8_t)(int)r;
        }
    }
}

/* The paper's own weight quantiser (Sec. 3.2, Eq. 2 with the de-quantised form
 * 2 (x_q / (2^b - 1) - 0.5) of Eq. 3 for weights): with the clip range
 * [l, u] = [-u, u], x_n = clip((w + u) / (2 u), 0, 1), x_q = round((2^b - 1) x_n),
 * and the weight enters the convolution as the odd integer 2 x_q - (2^b - 1)
 * (levels -3, -1, 1, 3 at b = 2; the de-quantised weight is that integer times
 * u / (2^b - 1)).  In fp32: one add, one multiply by k[g] = fl((2^b - 1) / (2 u[g]))
 * (computed in double), round half to even, clamp. */
/* Quantisation-aware training forward (Sec. 3.2 Eq. 2-3; Sec. 5: the bounds l,
 * u are learned, the rounding is passed by the straight-through estimator).
 * x is [P][G*Cg], group g = channel / Cg, bounds l[g] < u[g].  Per element, in
 * fp32 with one IEEE rounding per operation, the divisions taken as multiplies
 * by fp32 reciprocals (as the inference quantiser takes x / s as x * fl(1/s)):
 *   t = (x - l) * fl(1 / fl(u - l)),  x_n = min(max(t, 0), 1)  (NaN -> 0),
 *   x_q = rint(x_n * (2^b - 1))                                (half to even),
 *   kind 0 (activations): x_hat = x_q * fl(1 / (2^b - 1))            in [0, 1]
 *   kind 1 (weights):     x_hat = 2 * (x_q * fl(1 / (2^b - 1)) - 0.5) in [-1, 1]
 * (Eq. 3 printed with its two cases swapped; activations are the non-negative
 * ones.) */
static float fq_t(float x, float l, float inv_r) { return (x - l) * inv_r; }

void oracle_fake_quant_fwd(const float* x, float* xhat, int64_t P, int G, int64_t Cg, int bits, int kind,
                           const float* l, const float* u) {
    const float qp = (float)((1 << bits) - 1);
    const float inv_qp = 1.0f / qp;
    const int64_t C = (int64_t)G * Cg;
    for (int64_t p = 0; p < P; ++p) {
        for (int g = 0; g < G; ++g) {
            const float inv_r = 1.0f / (u[g] - l[g]);
            for (int64_t j = 0; j < Cg; ++j) {
                const int64_t i = p * C + (int64_t)g * Cg + j;
                float xn = fminf(fmaxf(fq_t(x[i], l[g], inv_r), 0.0f), 1.0f);
                float xq = rintf(xn * qp);
                float v = xq * inv_qp;
                xhat[i] = kind ? 2.0f * (v - 0.5f) : v;
            }
        }
    }
}

/* Inference codes with learned bounds (Sec. 3.2 Eq. 2 with l, u per group, the
 * training forward's x_q above): x_q = rint(min(max((x - l) * fl(1/fl(u - l)),
 * 0), 1) * (2^b - 1)), NaN -> 0, one code per byte, x and q [P][G*Cg]. */
void oracle_quantize_act_lu(const float* x, uint8_t* q, int64_t P, int G, int64_t Cg, int bits, const float* l,
                            const float* u) {
    const float qp = (float)((1 << bits) - 1);
    const int64_t C = (int64_t)G * Cg;
    for (int64_t p = 0; p < P; ++p) {
        for (int g = 0; g < G; ++g) {
            const float inv_r = 1.0f / (u[g] - l[g]);
            for (int64_t j = 0; j < Cg; ++j) {
                const int64_t i = p * C + (int64_t)g * Cg + j;
                float xn = fminf(fmaxf(fq_t(x[i], l[g], inv_r), 0.0f), 1.0f);
                q[i] = (uint8_t)(int)rintf(xn * qp);
            }
        }
    }
}

/* Its backward with the straight-through estimator: the rounding passes the
 * gradient unchanged, the clip does not (zero outside 0 < t < 1).  With the
 * de-quantisation factor c = 1 (activations) or 2 (weights) and r = u - l:
 *   dx     = dy * c * fl(1 / fl(r))             (fp32, elements with 0 < t < 1; else 0)
 *   dl[g]  = c / r^2 * sum over those elements of group g of dy * (x - u)
 *   du[g]  = -c / r^2 * sum over those elements of group g of dy * (x - l)
 * (d t / d l = (x - u) / r^2, d t / d u = -(x - l) / r^2), the sums and the
 * factors in double.  t is the forward's fp32 value, so both sides decide
 * "inside" in the same precision. */
void oracle_fake_quant_bwd(const float* x, const float* dy, float* dx, double* dl, double* du, int64_t P, int G,
                           int64_t Cg, int bits, int kind, const float* l, const float* u) {
    (void)bits;
    const int64_t C = (int64_t)G * Cg;
    const double c = kind ? 2.0 : 1.0;
    for (int g = 0; g < G; ++g) {
        const float inv_r = 1.0f / (u[g] - l[g]);
        const float k = (float)c * inv_r;
        const double rd = (double)u[g] - (double)l[g];
        double sa = 0.0, sb = 0.0;
        for (int64_t p = 0; p < P; ++p) {
            for (int64_t j = 0; j < Cg; ++j) {
                const int64_t i = p * C + (int64_t)g * Cg + j;
                const float t = fq_t(x[i], l[g], inv_r);
                if (t > 0.0f && t < 1.0f) {
                    dx[i] = dy[i] * k;
                    sa += (double)dy[i] * ((double)x[i] - (double)u[g]);
                    sb += (double)dy[i] * ((double)x[i] - (double)l[g]);
                } else {
                    dx[i] = 0.0f;
                }
            }
        }
        dl[g] = c / (rd * rd) * sa;
        du[g] = -c / (rd * rd) * sb;
    }
}

void oracle_quantize_weights_odd(const float* w, int8_t* wq, int G, int64_t per_group, int bits, const float* u) {
    const int qp = (1 << bits) - 1;
    for (int g = 0; g < G; ++g) {
        const float k = (float)((double)qp / (2.0 * (double)u[g]));
        for (int64_t i = 0; i < per_group; ++i) {
            float t = (w[g * per_group + i] + u[g]) * k;
            float r = rintf(t);
            r = fmaxf(r, 0.0f);
            r = fminf(r, (float)qp);
            wq[g * per_group + i] = (int8_t)(2 * (int)r - qp);
        }
    }
}

/* ---------------------------------------------------------------------- */
/* Sec. 3.1, Eq. 1 (conv as Y = X W^T) and Sec. 4.1 ("B-bit group          */
/* convolution"): for every image n, output pixel (oh, ow), group g and    */
/* output channel co of that group                                          */
/*   acc = sum_{kh,kw,ci} q[n, oh*s - p + kh, ow*s - p + kw, g*Cin_g + ci]  */
/*                        * wq[g, co, kh, kw, ci]                           */
/* with out-of-range input pixels contributing 0 (zero padding, which is   */
/* code 0 because l = 0).  int64 accumulation.                              */
/* ---------------------------------------------------------------------- */
typedef struct {
    int64_t N, H, W;
    int G, Cin_g, Cout_g, kh, kw, stride, pad;
} oracle_conv_shape;

static int64_t out_dim(int64_t in, int k, int s, int p) { return (in + 2 * p - k) / s + 1; }

static void conv_one_pixel(const uint8_t* q, const int8_t* wq, const oracle_conv_shape* sh,
                           int64_t n, int64_t oh, int64_t ow, int g, int64_t* acc /* Cout_g */) {
    const int64_t Cin = (int64_t)sh->G * sh->Cin_g;
    for (int co = 0; co < sh->Cout_g; ++co) {
        int64_t a = 0;
        for (int r = 0; r < sh->kh; ++r) {
            int64_t ih = oh * sh->stride - sh->pad + r;
            if (ih < 0 || ih >= sh->H) continue;
            for (int s = 0; s < sh->kw; ++s) {
                int64_t iw = ow * sh->stride - sh->pad + s;
                if (iw < 0 || iw >= sh->W) continue;
                const uint8_t* xp = q + ((n * sh->H + ih) * sh->W + iw) * Cin + (int64_t)g * sh->Cin_g;
                const int8_t* wp = wq + ((((int64_t)g * sh->Cout_g + co) * sh->kh + r) * sh->kw + s) * sh->Cin_g;
                for (int ci = 0; ci < sh->Cin_g; ++ci) a += (int64_t)xp[ci] * (int64_t)wp[ci];
            }
        }
        acc[co] = a;
    }
}

/* Full grouped convolution.  acc is [N, Ho, Wo, G*Cout_g] int64, group g's
 * channels at g*Cout_g (no permutation).  Returns the largest |acc|. */
int64_t oracle_group_conv(const uint8_t* q, const int8_t* wq, int64_t* acc, int64_t N, int64_t H,
                          int64_t W, int G, int Cin_g, int Cout_g, int kh, int kw, int stride, int pad) {
    oracle_conv_shape sh = {N, H, W, G, Cin_g, Cout_g, kh, kw, stride, pad};
    const int64_t Ho = out_dim(H, kh, stride, pad), Wo = out_dim(W, kw, stride, pad);
    const int64_t Cout = (int64_t)G * Cout_g;
    int64_t amax = 0;
#pragma omp parallel for collapse(2) schedule(dynamic, 1) reduction(max : amax)
    for (int64_t n = 0; n < N; ++n) {
        for (int64_t oh = 0; oh < Ho; ++oh) {
            for (int64_t ow = 0; ow < Wo; ++ow) {
                for (int g = 0; g < G; ++g) {
                    int64_t* a = acc + ((n * Ho + oh) * Wo + ow) * Cout + (int64_t)g * Cout_g;
                    conv_one_pixel(q, wq, &sh, n, oh, ow, g, a);
                    for (int co = 0; co < Cout_g; ++co) {
                        int64_t v = a[co] < 0 ? -a[co] : a[co];
                        if (v > amax) amax = v;
                    }
                }
            }
        }
    }
    return amax;
}

/* The same convolution evaluated only at a list of output pixels
 * (pix[i] = (n*Ho + oh)*Wo + ow); acc is [npix, G*Cout_g]. */
void oracle_group_conv_pixels(const uint8_t* q, const int8_t* wq, int64_t* acc, const int64_t* pix,
                              int64_t npix, int64_t N, int64_t H, int64_t W, int G, int Cin_g,
                              int Cout_g, int kh, int kw, int stride, int pad) {
    oracle_conv_shape sh = {N, H, W, G, Cin_g, Cout_g, kh, kw, stride, pad};
    const int64_t Ho = out_dim(H, kh, stride, pad), Wo = out_dim(W, kw, stride, pad);
    const int64_t Cout = (int64_t)G * Cout_g;
#pragma omp parallel for schedule(dynamic, 4)
    for (int64_t i = 0; i < npix; ++i) {
        int64_t p = pix[i];
        int64_t ow = p % Wo, oh = (p / Wo) % Ho, n = p / (Wo * Ho);
        for (int g = 0; g < G; ++g) conv_one_pixel(q, wq, &sh, n, oh, ow, g, acc + i * Cout + (int64_t)g * Cout_g);
    }
}

/* ---------------------------------------------------------------------- */
/* Output permutation of the cyclic shuffle (Sec. 4.2, Eq. 6-8).            */
/* kind 0: identity; kind 1: pi(g) = (g + shift) mod G (Eq. 6 is shift 1);  */
/* kind 3: explicit group permutation perm[g].  dst[g] receives the        */
/* destination group of source group g.  kind 2 (channel shuffle of        */
/* ShuffleNet, Sec. 4.3) is a per-channel permutation, handled by          */
/* oracle_dst_channel.  Returns 0, or -1 if the spec is not a permutation. */
/* ---------------------------------------------------------------------- */
int oracle_group_perm(int G, int kind, int shift, const int32_t* perm, int32_t* dst) {
    if (kind == 0 || kind == 2) {
        for (int g = 0; g < G; ++g) dst[g] = g;
    } else if (kind == 1) {
        for (int g = 0; g < G; ++g) dst[g] = (int32_t)((((g + shift) % G) + G) % G);
    } else if (kind == 3) {
        for (int g = 0; g < G; ++g) dst[g] = perm[g];
    } else {
        return -1;
    }
    for (int g = 0; g < G; ++g) {
        if (dst[g] < 0 || dst[g] >= G) return -1;
        for (int h = 0; h < g; ++h)
            if (dst[h] == dst[g]) return -1;
    }
    return 0;
}

/* Destination channel of source channel (g, co).  For kind 2 the channel
 * shuffle of Sec. 4.3 (ShuffleNet's reshape [G, Cg] -> transpose ->
 * flatten) sends channel g*Cg + co to co*G + g. */
static int64_t dst_channel(int kind, const int32_t* dst_group, int G, int Cout_g, int g, int co) {
    if (kind == 2) return (int64_t)co * G + g;
    return (int64_t)dst_group[g] * Cout_g + co;
}

/* ---------------------------------------------------------------------- */
/* Epilogue of one layer (Sec. 3.2 de-quantisation and the alpha output    */
/* scale, Sec. 4.2 output permutation, Eq. 2 requantisation for the next   */
/* layer).  For every output pixel and source channel (g, co):             */
/*   y  = (float)acc * m_out[g]            (m_out = s_w s_a alpha)          */
/*   y  = y + shortcut[pixel, g*Cout_g+co]  if a shortcut is given          */
/*   y  = max(y, 0)                         if relu                        */
/*   t  = shortcut ? y : (float)acc; q = clamp(rint(t * m_req[g]), 0, Qp)  */
/* all written at the destination channel of (g, co).  acc must satisfy    */
/* |acc| < 2^24 so that (float)acc is exact; returns -1 otherwise.         */
/* Any of acc_out / y_out / q_out may be NULL.                             */
/* ---------------------------------------------------------------------- */
int oracle_epilogue(const int64_t* acc, int64_t npix, int G, int Cout_g, const float* m_out,
                    const float* m_req, int shuffle_kind, int shuffle_shift, const int32_t* perm,
                    const float* shortcut, int relu, int bits_out, int32_t* acc_out, float* y_out,
                    uint8_t* q_out) {
    int32_t dst_group[256];
    if (G > 256) return -1;
    if (oracle_group_perm(G, shuffle_kind, shuffle_shift, perm, dst_group) != 0) return -1;
    const int64_t C = (int64_t)G * Cout_g;
    const int qmax = (1 << bits_out) - 1;
    for (int64_t i = 0; i < npix * C; ++i)
        if (acc[i] >= (1 << 24) || acc[i] <= -(1 << 24)) return -1;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < npix; ++p) {
        for (int g = 0; g < G; ++g) {
            for (int co = 0; co < Cout_g; ++co) {
                int64_t src = (int64_t)g * Cout_g + co;
                int64_t dst = dst_channel(shuffle_kind, dst_group, G, Cout_g, g, co);
                int64_t a = acc[p * C + src];
                float af = (float)a;
                float y = af * m_out[g];
                if (shortcut) y = y + shortcut[p * C + src];
                if (relu) y = fmaxf(y, 0.0f);
                if (acc_out) acc_out[p * C + dst] = (int32_t)a;
                if (y_out) y_out[p * C + dst] = y;
                if (q_out) {
                    float t = (shortcut ? y : af) * m_req[g];
                    float r = rintf(t);
                    r = fmaxf(r, 0.0f);
                    r = fminf(r, (float)qmax);
                    q_out[p * C + dst] = (uint8_t)(int)r;
                }
            }
        }
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Step-size initialisation (Sec. 5 follows LSQ for training; LSQ sets the */
/* step to 2 mean|v| / sqrt(Qp)).  Means are taken in double over every    */
/* element of the group in storage order, then the step is rounded to      */
/* float once.                                                             */
/* ---------------------------------------------------------------------- */
void oracle_act_step(const float* x, int64_t N, int64_t H, int64_t W, int G, int Cg, int bits, float* s_out) {
    const int64_t C = (int64_t)G * Cg;
    const int64_t P = N * H * W;
    const double qp = (double)((1 << bits) - 1);
    for (int g = 0; g < G; ++g) {
        double sum = 0.0;
        for (int64_t p = 0; p < P; ++p)
            for (int j = 0; j < Cg; ++j) sum += (double)x[p * C + (int64_t)g * Cg + j];
        double mean = sum / (double)(P * Cg);
        s_out[g] = (float)(2.0 * mean / sqrt(qp));
    }
}

void oracle_weight_step(const float* w, int G, int64_t per_group, int bits, float* s_out) {
    const double qp = (double)((1 << (bits - 1)) - 1);
    for (int g = 0; g < G; ++g) {
        double sum = 0.0;
        for (int64_t i = 0; i < per_group; ++i) sum += fabs((double)w[g * per_group + i]);
        double mean = sum / (double)per_group;
        s_out[g] = (float)(2.0 * mean / sqrt(qp));
    }
}

/* Reciprocal of a step, rounded to float: the multiplier both sides use. */
float oracle_inv_step(float s) { return (float)(1.0 / (double)s); }

/* Epilogue multipliers (Sec. 3.2: alpha scales the layer output):
 *   m_out[g] = fl(s_w[g] s_a[g] alpha)
 *   m_req[g] = fl(s_w[g] s_a[g] alpha / s_next[dst(g)])
 * where dst(g) is the destination group of g, because the requantised code
 * lands in group dst(g) of the next layer and uses that group's step. */
int oracle_epilogue_scales(int G, const float* s_w, const float* s_a, double alpha, const float* s_next,
                           int shuffle_kind, int shuffle_shift, const int32_t* perm, float* m_out,
                           float* m_req) {
    int32_t dst_group[256];
    if (G > 256) return -1;
    if (oracle_group_perm(G, shuffle_kind, shuffle_shift, perm, dst_group) != 0) return -1;
    for (int g = 0; g < G; ++g) {
        double m = (double)s_w[g] * (double)s_a[g] * alpha;
        m_out[g] = (float)m;
        if (s_next) m_req[g] = (float)(m / (double)s_next[dst_group[g]]);
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Full-precision layers around the PalQuant body (Sec. 5: the first and  */
/* the last layer are not quantised).                                      */
/* ---------------------------------------------------------------------- */

/* Direct NHWC convolution, weights [Cout][k][k][Cin]: every output starts
 * from 0 and adds fmaf(x, w, acc) over (kh, kw, ci) in that order, skipping
 * taps outside the image (zero padding); optional ReLU (fmaxf, NaN -> 0). */
void oracle_conv2d_f32(const float* x, const float* w, float* y, int64_t N, int64_t H, int64_t W, int Cin,
                       int Cout, int k, int s, int p, int relu) {
    const int64_t Ho = out_dim(H, k, s, p), Wo = out_dim(W, k, s, p);
#pragma omp parallel for collapse(2) schedule(static)
    for (int64_t n = 0; n < N; ++n) {
        for (int64_t oh = 0; oh < Ho; ++oh) {
            for (int64_t ow = 0; ow < Wo; ++ow) {
                for (int co = 0; co < Cout; ++co) {
                    float acc = 0.0f;
                    for (int kh = 0; kh < k; ++kh) {
                        const int64_t ih = oh * s - p + kh;
                        if (ih < 0 || ih >= H) continue;
                        for (int kw = 0; kw < k; ++kw) {
                            const int64_t iw = ow * s - p + kw;
                            if (iw < 0 || iw >= W) continue;
                            const float* xp = x + ((n * H + ih) * W + iw) * Cin;
                            const float* wp = w + (((int64_t)co * k + kh) * k + kw) * Cin;
                            for (int ci = 0; ci < Cin; ++ci) acc = fmaf(xp[ci], wp[ci], acc);
                        }
                    }
                    if (relu) acc = fmaxf(acc, 0.0f);
                    y[((n * Ho + oh) * Wo + ow) * Cout + co] = acc;
                }
            }
        }
    }
}

/* Max pooling over the in-image taps of each k x k window (padding taps are
 * ignored), taken with fmaxf in (kh, kw) order starting from -infinity. */
void oracle_maxpool_f32(const float* x, float* y, int64_t N, int64_t H, int64_t W, int C, int k, int s, int p) {
    const int64_t Ho = out_dim(H, k, s, p), Wo = out_dim(W, k, s, p);
#pragma omp parallel for collapse(2) schedule(static)
    for (int64_t n = 0; n < N; ++n) {
        for (int64_t oh = 0; oh < Ho; ++oh) {
            for (int64_t ow = 0; ow < Wo; ++ow) {
                for (int c = 0; c < C; ++c) {
                    float m = -INFINITY;
                    for (int kh = 0; kh < k; ++kh) {
                        const int64_t ih = oh * s - p + kh;
                        if (ih < 0 || ih >= H) continue;
                        for (int kw = 0; kw < k; ++kw) {
                            const int64_t iw = ow * s - p + kw;
                            if (iw < 0 || iw >= W) continue;
                            m = fmaxf(m, x[((n * H + ih) * W + iw) * C + c]);
                        }
                    }
                    y[((n * Ho + oh) * Wo + ow) * C + c] = m;
                }
            }
        }
    }
}

/* Global average pooling: the sum over (h, w) in storage order from 0, then
 * one division by H * W. */
void oracle_avgpool_f32(const float* x, float* y, int64_t N, int64_t H, int64_t W, int C) {
#pragma omp parallel for schedule(static)
    for (int64_t n = 0; n < N; ++n) {
        for (int c = 0; c < C; ++c) {
            float acc = 0.0f;
            for (int64_t i = 0; i < H * W; ++i) acc = acc + x[(n * H * W + i) * C + c];
            y[n * C + c] = acc / (float)(H * W);
        }
    }
}

/* Fully connected layer without bias, weights [Cout][Cin]: each output is
 * fmaf(x_i, w_oi, acc) over i in order from 0. */
void oracle_linear_f32(const float* x, const float* w, float* y, int64_t N, int Cin, int Cout) {
#pragma omp parallel for collapse(2) schedule(static)
    for (int64_t n = 0; n < N; ++n) {
        for (int o = 0; o < Cout; ++o) {
            float acc = 0.0f;
            for (int i = 0; i < Cin; ++i) acc = fmaf(x[n * Cin + i], w[(int64_t)o * Cin + i], acc);
            y[n * Cout + o] = acc;
        }
    }
}
