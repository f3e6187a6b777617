/*
 * TASQ oracle: a plain, slow CPU statement of the masked-W8A8 path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
 * load this file: only tests/, __graft_entry__.smoke() and bench.py's
 * cpu_baseline / --impl reference legs use it.  It shares no header, helper,
 * table or constant with the CUDA library; its only common ground with that
 * library is the seeded input generators that feed both.
 *
 * Every function cites the passage of the paper (TASQ, arXiv 2608.03057) it
 * restates.  Floating point is fp32 where a float decides an integer (the
 * quantized codes), following one fixed operation order that is the kernel's
 * precision; the dequantized result is given twice: in the kernel's fp32
 * rounding order (oq_epilogue_f32) and by the definition in fp64
 * (oq_linear_def_f64 / oq_conv3x3_def_f64).  Compile with -ffp-contract=off so
 * that the compiler fuses nothing: every operation rounds once to nearest-even,
 * and the only fused multiply-adds are the explicit fmaf calls of the epilogue.
 *
 * Readings of the paper taken here (the paper is silent on them):
 *  - Weights are quantized per output channel, activations per token (linear)
 *    or per tensor (3x3 conv input).
 *  - "Symmetric" range: the App. A.1 formulas are applied verbatim with the
 *    range forced to [-max|v|, +max|v|].  For weights this gives alpha =
 *    max|w|/2^(n-1) and z = 2^(n-1) exactly, so the stored code Q - 2^(n-1)
 *    is a true signed integer with no weight zero point.
 *  - Rounding to nearest (Eq. act_quant) breaks ties to even.
 *  - Degenerate range (max == min): alpha = 1, z = 2^(n-1) for the symmetric
 *    range, z = -min for the asymmetric range.
 *  - Truncation (Eq. truncquant, Eq. hw_rightshift) is a floor on the
 *    unsigned code; the operating precision b keeps the top b of the 8 stored
 *    planes.  The dequantization factor 2^n/(2^n-1) of Eq. weight_dequant uses
 *    the stored precision n = 8 for every b.
 *  - 3x3 conv (stride 1, pad 1): zero padding lives in the real domain, so a
 *    padded tap contributes nothing to the dequantized sum.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OQ_SYMRANGE 0
#define OQ_ASYM 1

/* Round-to-nearest-even from fp32 to bf16 (the upper 16 bits), finite input. */
static uint16_t oq_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    uint32_t keep_even = (u >> 16) & 1u;
    u += 0x7FFFu + keep_even;
    return (uint16_t)(u >> 16);
}

void oq_f32_to_bf16(const float* in, int64_t n, uint16_t* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = oq_bf16_rne(in[i]);
}

/* Range of one group of values: [min, max] (asymmetric) or [-max|v|, max|v|]. */
static void oq_range(const float* v, int64_t n, int64_t stride, int mode, float* lo, float* hi) {
    if (mode == OQ_SYMRANGE) {
        float a = 0.0f;
        for (int64_t i = 0; i < n; ++i) {
            float m = fabsf(v[i * stride]);
            if (m > a) a = m;
        }
        *lo = -a;
        *hi = a;
    } else {
        float mn = v[0], mx = v[0];
        for (int64_t i = 1; i < n; ++i) {
            float x = v[i * stride];
            if (x < mn) mn = x;
            if (x > mx) mx = x;
        }
        *lo = mn;
        *hi = mx;
    }
}

/*
 * Weight quantizer, App. A.1.1 (Eqs. weight_quant, weight_scale,
 * weight_dequant), one output channel (row of w[N][K]) at a time:
 *   alpha = (max - min) / 2^n,  z = -min / alpha,
 *   Q = clamp(floor(w/alpha + z), 0, 2^n - 1).
 * Outputs the unsigned code Q (q_out, may be NULL), the stored signed code
 * Q - 2^(n-1) (s_out, may be NULL; n <= 8), alpha, z, and the dequantization
 * scale c = (2^n/(2^n-1)) * alpha so that w_hat = c * (Q - z).
 * fp32 order: alpha = RN(RN(hi - lo) / 2^n); z = RN(-lo / alpha);
 * u = RN(RN(w / alpha) + z); Q = floor(u); c = RN(alpha * RN(2^n / (2^n - 1))).
 */
void oq_quant_weight(const float* w, int N, int K, int n_bits, int mode, int32_t* q_out, int8_t* s_out,
                     float* alpha_out, float* z_out, float* c_out) {
    const float levels = (float)(1 << n_bits);              /* 2^n */
    const float half = (float)(1 << (n_bits - 1));          /* 2^(n-1) */
    const float deq = levels / (levels - 1.0f);              /* 2^n / (2^n - 1) */
    const int qmax = (1 << n_bits) - 1;
    for (int n = 0; n < N; ++n) {
        const float* row = w + (int64_t)n * K;
        float lo, hi;
        oq_range(row, K, 1, mode, &lo, &hi);
        float range = hi - lo;
        float alpha, z;
        if (range == 0.0f) {
            alpha = 1.0f;
            z = (mode == OQ_SYMRANGE) ? half : -lo;
        } else {
            alpha = range / levels;
            z = -lo / alpha;
        }
        for (int k = 0; k < K; ++k) {
            float t = row[k] / alpha;
            float u = t + z;
            float f = floorf(u);
            int q = (f < 0.0f) ? 0 : (f > (float)qmax ? qmax : (int)f);
            if (q_out) q_out[(int64_t)n * K + k] = q;
            if (s_out) s_out[(int64_t)n * K + k] = (int8_t)(q - (int)half);
        }
        alpha_out[n] = alpha;
        if (z_out) z_out[n] = z;
        if (c_out) c_out[n] = alpha * deq;
    }
}

/*
 * Activation quantizer, App. A.1.2 (Eqs. act_quant, act_scale):
 *   alpha = (max - min) / (2^n - 1),  z = -min / alpha,
 *   Q = clamp(round_half_even(x/alpha + z), 0, 2^n - 1).
 * gran = 0: one (alpha, z) per row of x[M][K] (per token); gran = 1: one for
 * the whole tensor.  Outputs s = Q - 2^(n-1) (int8), alpha and
 * zc = 2^(n-1) - z, so that x_hat = alpha * (Q - z) = alpha * (s + zc).
 * fp32 order: alpha = RN(RN(hi - lo) / (2^n - 1)); z = RN(-lo / alpha);
 * u = RN(RN(x / alpha) + z); Q = rint(u); zc = RN(2^(n-1) - z).
 */
void oq_quant_act(const float* x, int M, int K, int n_bits, int mode, int gran, int8_t* s_out,
                  float* alpha_out, float* zc_out) {
    const float denom = (float)((1 << n_bits) - 1);
    const float half = (float)(1 << (n_bits - 1));
    const int qmax = (1 << n_bits) - 1;
    int groups = gran ? 1 : M;
    int64_t per = gran ? (int64_t)M * K : (int64_t)K;
    for (int g = 0; g < groups; ++g) {
        const float* v = x + (int64_t)g * per;
        float lo, hi;
        oq_range(v, per, 1, mode, &lo, &hi);
        float range = hi - lo;
        float alpha, z;
        if (range == 0.0f) {
            alpha = 1.0f;
            z = (mode == OQ_SYMRANGE) ? half : -lo;
        } else {
            alpha = range / denom;
            z = -lo / alpha;
        }
        for (int64_t i = 0; i < per; ++i) {
            float t = v[i] / alpha;
            float u = t + z;
            float r = rintf(u); /* default rounding mode: nearest, ties to even */
            int q = (r < 0.0f) ? 0 : (r > (float)qmax ? qmax : (int)r);
            s_out[(int64_t)g * per + i] = (int8_t)(q - (int)half);
        }
        alpha_out[g] = alpha;
        zc_out[g] = half - z;
    }
}

/*
 * Operating-precision weight, Eq. hw_rightshift with k = 8 - b dropped planes:
 * from the stored 8-bit code Q = s + 128, Q_b = floor(Q / 2^k), whose value on
 * the stored 8-bit grid is 2^k * Q_b (Eq. hw_multi_lsb: Q - LSB^(k)).
 * Returned as the signed stored form 2^k * Q_b - 128.
 */
int oq_mask(int s, int b) {
    int q = s + 128;
    int k = 8 - b;
    int qb = q / (1 << k); /* q >= 0: integer division is the floor */
    return qb * (1 << k) - 128;
}

void oq_mask_weights(const int8_t* s_w, int64_t n, int b, int8_t* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = (int8_t)oq_mask(s_w[i], b);
}

/*
 * Integer contraction of Eq. qalora, Y = Q(X) Q_M(W), on the stored codes:
 *   acc[m][n] = sum_k s_x[m][k] * mask_b(s_w[n][k]).
 * Accumulates in int64; returns the number of results outside int32 (0 when
 * every result fits, which the caller checks).
 */
int64_t oq_gemm(const int8_t* s_x, int M, const int8_t* s_w, int N, int K, int b, int32_t* acc) {
    int64_t overflow = 0;
    int8_t* wm = (int8_t*)malloc((size_t)N * K);
    oq_mask_weights(s_w, (int64_t)N * K, b, wm);
#pragma omp parallel for reduction(+ : overflow) schedule(static)
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            int64_t sum = 0;
            const int8_t* xr = s_x + (int64_t)m * K;
            const int8_t* wr = wm + (int64_t)n * K;
            for (int k = 0; k < K; ++k) sum += (int64_t)xr[k] * (int64_t)wr[k];
            if (sum > INT32_MAX || sum < INT32_MIN) overflow++;
            acc[(int64_t)m * N + n] = (int32_t)sum;
        }
    }
    free(wm);
    return overflow;
}

/* rs_b[n] = sum_k mask_b(s_w[n][k]): the weight row sum that carries the
 * activation zero point through the integer contraction. */
void oq_row_sums(const int8_t* s_w, int N, int K, int b, int32_t* rs) {
    for (int n = 0; n < N; ++n) {
        int64_t sum = 0;
        for (int k = 0; k < K; ++k) sum += oq_mask(s_w[(int64_t)n * K + k], b);
        rs[n] = (int32_t)sum;
    }
}

/*
 * Dequantization (Eqs. act_dequant and weight_dequant) folded around the
 * integer contraction, in the kernel's fp32 rounding order (two fused
 * multiply-adds, each rounded once):
 *   u = RN(zc * float(rs) + float(acc)),  s = RN(alpha * c),  y = RN(u * s + bias),
 *   output bf16_rne(y),
 * because sum_k alpha(s_x + zc) * c * mask(s_w) = alpha * c * (acc + zc * rs).
 * alpha/zc are indexed by row_of(m) = m (per token) or 0 (per tensor);
 * rs[m*rs_stride_m + n] lets a conv pass one row sum per output pixel.
 */
void oq_epilogue_f32(const int32_t* acc, int M, int N, const float* alpha, const float* zc, int per_tensor,
                     const int32_t* rs, int64_t rs_stride_m, const float* c_w, const float* bias, float* y_f32,
                     uint16_t* y_bf16) {
    for (int m = 0; m < M; ++m) {
        int r = per_tensor ? 0 : m;
        for (int n = 0; n < N; ++n) {
            float a = (float)acc[(int64_t)m * N + n];
            float u = fmaf(zc[r], (float)rs[(int64_t)m * rs_stride_m + n], a);
            float s = alpha[r] * c_w[n];
            float y = fmaf(u, s, bias ? bias[n] : 0.0f);
            if (y_f32) y_f32[(int64_t)m * N + n] = y;
            if (y_bf16) y_bf16[(int64_t)m * N + n] = oq_bf16_rne(y);
        }
    }
}

/*
 * The linear layer by its definition, in fp64: dequantize each operand
 * element (x_hat = alpha * (s_x + zc), Eq. act_dequant; w_hat = c * mask_b(s_w),
 * Eq. weight_dequant with z = 128) and sum the products, then add the bias.
 * No factoring of the zero point; used to pin oq_epilogue_f32.
 */
void oq_linear_def_f64(const int8_t* s_x, const float* alpha, const float* zc, int M, const int8_t* s_w,
                       const float* c_w, const float* bias, int N, int K, int b, double* y) {
#pragma omp parallel for schedule(static)
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            double sum = 0.0;
            for (int k = 0; k < K; ++k) {
                double xh = (double)alpha[m] * ((double)s_x[(int64_t)m * K + k] + (double)zc[m]);
                double wh = (double)c_w[n] * (double)oq_mask(s_w[(int64_t)n * K + k], b);
                sum += xh * wh;
            }
            y[(int64_t)m * N + n] = sum + (bias ? (double)bias[n] : 0.0);
        }
    }
}

/*
 * 3x3 convolution, stride 1, padding 1, NHWC activations and weights
 * w[Cout][3][3][Cin] (K = 9*Cin ordered (kh, kw, cin)), on the stored codes:
 *   acc[p][n] = sum over in-bounds taps and cin of s_x * mask_b(s_w);
 *   rs[p][n]  = sum over the same in-bounds taps of mask_b(s_w).
 * A padded tap is left out of both sums: its real-domain value is 0, so it
 * contributes nothing after dequantization.  p = (b*H + h)*W + w.
 */
void oq_conv3x3(const int8_t* s_x, int B, int H, int W, int Cin, const int8_t* s_w, int Cout, int b,
                int32_t* acc, int32_t* rs) {
    int64_t P = (int64_t)B * H * W;
    int K = 9 * Cin;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < P; ++p) {
        int bb = (int)(p / ((int64_t)H * W));
        int h = (int)((p / W) % H);
        int w = (int)(p % W);
        for (int n = 0; n < Cout; ++n) {
            int64_t sum = 0, wsum = 0;
            for (int kh = 0; kh < 3; ++kh) {
                int ih = h + kh - 1;
                if (ih < 0 || ih >= H) continue;
                for (int kw = 0; kw < 3; ++kw) {
                    int iw = w + kw - 1;
                    if (iw < 0 || iw >= W) continue;
                    const int8_t* xr = s_x + (((int64_t)bb * H + ih) * W + iw) * Cin;
                    const int8_t* wr = s_w + (int64_t)n * K + (kh * 3 + kw) * Cin;
                    for (int c = 0; c < Cin; ++c) {
                        int wm = oq_mask(wr[c], b);
                        sum += (int64_t)xr[c] * wm;
                        wsum += wm;
                    }
                }
            }
            acc[p * Cout + n] = (int32_t)sum;
            rs[p * Cout + n] = (int32_t)wsum;
        }
    }
}

/*
 * The 3x3 convolution by its definition, in fp64: x_hat = alpha * (s_x + zc)
 * inside the image and 0 in the padding; w_hat = c * mask_b(s_w).
 */
void oq_conv3x3_def_f64(const int8_t* s_x, float alpha, float zc, int B, int H, int W, int Cin, const int8_t* s_w,
                        const float* c_w, const float* bias, int Cout, int b, double* y) {
    int64_t P = (int64_t)B * H * W;
    int K = 9 * Cin;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < P; ++p) {
        int bb = (int)(p / ((int64_t)H * W));
        int h = (int)((p / W) % H);
        int w = (int)(p % W);
        for (int n = 0; n < Cout; ++n) {
            double sum = 0.0;
            for (int kh = 0; kh < 3; ++kh) {
                for (int kw = 0; kw < 3; ++kw) {
                    int ih = h + kh - 1, iw = w + kw - 1;
                    for (int c = 0; c < Cin; ++c) {
                        double xh = 0.0;
                        if (ih >= 0 && ih < H && iw >= 0 && iw < W)
                            xh = (double)alpha *
                                 ((double)s_x[(((int64_t)bb * H + ih) * W + iw) * Cin + c] + (double)zc);
                        double wh = (double)c_w[n] * (double)oq_mask(s_w[(int64_t)n * K + (kh * 3 + kw) * Cin + c], b);
                        sum += xh * wh;
                    }
                }
            }
            y[p * Cout + n] = sum + (bias ? (double)bias[n] : 0.0);
        }
    }
}

/* ------------------------------------------------------------------------
 * Asymmetric weights: the App. A.1.1 quantizer on each channel's true
 * [min, max] (oq_quant_weight with OQ_ASYM) leaves a real-valued zero point
 * z, and Eq. weight_dequant on the masked code reads
 *   w_hat = c * (Q_b - z) = c * (mask_b(s_w) + zcw),   zcw = 2^(n-1) - z,
 * (Q_b = mask_b(s_w) + 2^(n-1) on the stored grid).  The dequantized
 * contraction then has four integer-carried terms:
 *   sum_k x_hat * w_hat = alpha * c * (acc + zc * rs_b + zcw * sx + K * zc * zcw),
 *   sx[m] = sum_k s_x[m][k].
 * ------------------------------------------------------------------------ */

/* zcw[n] = RN(2^(n-1) - z[n]). */
void oq_weight_zero_offsets(const float* z, int N, int n_bits, float* zcw) {
    const float half = (float)(1 << (n_bits - 1));
    for (int n = 0; n < N; ++n) zcw[n] = half - z[n];
}

/* sx[m] = sum_k s_x[m][k] (int32: |sx| <= 128 K). */
void oq_code_sums(const int8_t* s_x, int M, int K, int32_t* sx) {
    for (int m = 0; m < M; ++m) {
        int64_t sum = 0;
        for (int k = 0; k < K; ++k) sum += s_x[(int64_t)m * K + k];
        sx[m] = (int32_t)sum;
    }
}

/*
 * The four-term dequantization in fp32, per token (linear layers).  The two
 * zero-offset terms share the factor zcw: zcw * sx + K * zc * zcw =
 * zcw * t with t[m] = sx[m] + K * zc[m] = sum_k (s_x[m][k] + zc[m]), the
 * token's dequantized activation sum over alpha.  Each step rounded once:
 *   t  = RN(float(sx) + RN(float(K) * zc))                    (per token)
 *   u1 = RN(zc * float(rs) + float(acc)),  u2 = RN(zcw * t + u1),
 *   s  = RN(alpha * c),                    y  = RN(u2 * s + bias),  bf16_rne(y).
 * With zcw = 0 (symmetric weights) u2 = u1 and this is oq_epilogue_f32.
 */
void oq_epilogue_zp_f32(const int32_t* acc, int M, int N, int K, const float* alpha, const float* zc,
                        const int32_t* sx, const int32_t* rs, const float* c_w, const float* zcw, const float* bias,
                        float* y_f32, uint16_t* y_bf16) {
    for (int m = 0; m < M; ++m) {
        const float kz = (float)K * zc[m];
        const float t = (float)sx[m] + kz;
        for (int n = 0; n < N; ++n) {
            float a = (float)acc[(int64_t)m * N + n];
            float u1 = fmaf(zc[m], (float)rs[n], a);
            float u2 = fmaf(zcw[n], t, u1);
            float s = alpha[m] * c_w[n];
            float y = fmaf(u2, s, bias ? bias[n] : 0.0f);
            if (y_f32) y_f32[(int64_t)m * N + n] = y;
            if (y_bf16) y_bf16[(int64_t)m * N + n] = oq_bf16_rne(y);
        }
    }
}

/*
 * The linear layer with asymmetric weights by its definition, in fp64:
 * x_hat = alpha * (s_x + zc) (Eq. act_dequant), w_hat = c * (Q_b - z) with
 * Q_b = mask_b(s_w) + 128 and the quantizer's own z (Eq. weight_dequant),
 * summed product by product.  No term is factored out.
 */
void oq_linear_zp_def_f64(const int8_t* s_x, const float* alpha, const float* zc, int M, const int8_t* s_w,
                          const float* c_w, const float* z, const float* bias, int N, int K, int b, double* y) {
#pragma omp parallel for schedule(static)
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            double sum = 0.0;
            for (int k = 0; k < K; ++k) {
                double xh = (double)alpha[m] * ((double)s_x[(int64_t)m * K + k] + (double)zc[m]);
                double qb = (double)oq_mask(s_w[(int64_t)n * K + k], b) + 128.0;
                double wh = (double)c_w[n] * (qb - (double)z[n]);
                sum += xh * wh;
            }
            y[(int64_t)m * N + n] = sum + (bias ? (double)bias[n] : 0.0);
        }
    }
}

/*
 * 3x3 convolution with asymmetric weights.  The padded taps are zero in the
 * real domain, so over output pixel p only the in-bounds taps carry terms:
 *   sum x_hat * w_hat_b = alpha * c * (acc + zc * rs[p] + zcw * t[p]),
 *   t[p] = sxw[p] + Kv[p] * zc,
 * with sxw[p] the sum of the codes of the in-bounds taps' input pixels (all
 * Cin channels) and Kv[p] = Cin * (number of in-bounds taps).  Outputs sxw
 * and Kv per output pixel p = (b*H + h)*W + w.
 */
void oq_conv3x3_code_sums(const int8_t* s_x, int B, int H, int W, int Cin, int32_t* sxw, int32_t* kv) {
    int64_t P = (int64_t)B * H * W;
    for (int64_t p = 0; p < P; ++p) {
        int bb = (int)(p / ((int64_t)H * W));
        int h = (int)((p / W) % H);
        int w = (int)(p % W);
        int64_t sum = 0;
        int taps = 0;
        for (int kh = 0; kh < 3; ++kh) {
            int ih = h + kh - 1;
            if (ih < 0 || ih >= H) continue;
            for (int kw = 0; kw < 3; ++kw) {
                int iw = w + kw - 1;
                if (iw < 0 || iw >= W) continue;
                const int8_t* xr = s_x + (((int64_t)bb * H + ih) * W + iw) * Cin;
                for (int c = 0; c < Cin; ++c) sum += xr[c];
                ++taps;
            }
        }
        sxw[p] = (int32_t)sum;
        kv[p] = taps * Cin;
    }
}

/*
 * The conv four-term dequantization in fp32, one activation scale for the
 * tensor (alpha, zc), rs[p][n] the in-bounds row sums of oq_conv3x3:
 *   t  = RN(float(sxw[p]) + RN(float(Kv[p]) * zc)),
 *   u1 = RN(zc * float(rs) + float(acc)),  u2 = RN(zcw * t + u1),
 *   y  = RN(u2 * RN(alpha * c) + bias),    bf16_rne(y).
 */
void oq_conv_epilogue_zp_f32(const int32_t* acc, int64_t P, int N, float alpha, float zc, const int32_t* sxw,
                             const int32_t* kv, const int32_t* rs, const float* c_w, const float* zcw,
                             const float* bias, float* y_f32, uint16_t* y_bf16) {
    for (int64_t p = 0; p < P; ++p) {
        const float t = (float)sxw[p] + (float)kv[p] * zc;
        for (int n = 0; n < N; ++n) {
            float a = (float)acc[p * N + n];
            float u1 = fmaf(zc, (float)rs[p * N + n], a);
            float u2 = fmaf(zcw[n], t, u1);
            float s = alpha * c_w[n];
            float y = fmaf(u2, s, bias ? bias[n] : 0.0f);
            if (y_f32) y_f32[p * N + n] = y;
            if (y_bf16) y_bf16[p * N + n] = oq_bf16_rne(y);
        }
    }
}

/*
 * The 3x3 convolution with asymmetric weights by its definition, in fp64:
 * x_hat = alpha * (s_x + zc) inside the image and 0 in the padding,
 * w_hat = c * (Q_b - z) with Q_b = mask_b(s_w) + 128 and the quantizer's z.
 */
void oq_conv3x3_zp_def_f64(const int8_t* s_x, float alpha, float zc, int B, int H, int W, int Cin,
                           const int8_t* s_w, const float* c_w, const float* z, const float* bias, int Cout, int b,
                           double* y) {
    int64_t P = (int64_t)B * H * W;
    int K = 9 * Cin;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < P; ++p) {
        int bb = (int)(p / ((int64_t)H * W));
        int h = (int)((p / W) % H);
        int w = (int)(p % W);
        for (int n = 0; n < Cout; ++n) {
            double sum = 0.0;
            for (int kh = 0; kh < 3; ++kh) {
                for (int kw = 0; kw < 3; ++kw) {
                    int ih = h + kh - 1, iw = w + kw - 1;
                    for (int c = 0; c < Cin; ++c) {
                        double xh = 0.0;
                        if (ih >= 0 && ih < H && iw >= 0 && iw < W)
                            xh = (double)alpha *
                                 ((double)s_x[(((int64_t)bb * H + ih) * W + iw) * Cin + c] + (double)zc);
                        double qb = (double)oq_mask(s_w[(int64_t)n * K + (kh * 3 + kw) * Cin + c], b) + 128.0;
                        double wh = (double)c_w[n] * (qb - (double)z[n]);
                        sum += xh * wh;
                    }
                }
            }
            y[p * Cout + n] = sum + (bias ? (double)bias[n] : 0.0);
        }
    }
}

/* Threads of the OpenMP loops above: n (n <= 0: every processor); and the
 * number the next parallel loop will use.  Timing helpers, no arithmetic. */
void oq_set_threads(int n) {
#ifdef _OPENMP
    omp_set_num_threads(n > 0 ? n : omp_get_num_procs());
#else
    (void)n;
#endif
}

int oq_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
