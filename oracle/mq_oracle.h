/*
 * mq_oracle.h -- plain, slow, single-threaded CPU oracle for the integer-only
 * quantized linear layer of MobileQuant (arXiv 2408.13933).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may include, link,
 * load or call this code: only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg do.  It shares no header, helper, table or
 * constant with the CUDA library; it is written from the paper's definitions:
 *
 *   - Sec. 3.1 (mobile-friendly design choices): integer (fixed-point) weights
 *     and activations, per-tensor/per-channel static quantization, int8 x int8.
 *   - Sec. 4.2, eqs. 2-4: the asymmetric uniform quantizer
 *       q_max = 2^bw - 1, alpha = (f_max - f_min)/q_max, beta = f_min/alpha,
 *       X_int = min(max(round(X/alpha) - beta, 0), q_max).
 *     Applied to the layer output with a static (alpha, beta) it is the
 *     requantization below; shifted by -128 to signed int8 its offset is the
 *     output zero point zy (the integer zero point round(-f_min / alpha)
 *     of the unsigned range, minus 128).
 *   - Sec. 5.1 and Appendix A: symmetric per-output-channel weights (int8, or
 *     int4 in [-8, 7]), so the weight zero point is 0.
 *
 * Conventions: M tokens, K input features, N output features.  x is int8
 * [M][ldx], weights are int8 [N][K] (K contiguous) or int4 packed two per byte
 * [N][K/2] with the low nibble holding the even k.  Output y is int8 [M][ldy].
 *
 * Every accumulation is done in int64 and every rounding is done on exact
 * integers (__int128), so the oracle's result is the mathematical definition.
 *
 * Parity status of each function is stated beside it.
 */
#ifndef MQ_ORACLE_H
#define MQ_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Return codes of the oracle (its own, not the library's). */
#define ORACLE_OK 0
#define ORACLE_EINVAL 1    /* bad argument */
#define ORACLE_EOVERFLOW 2 /* an accumulator left the int32 range */

/*
 * Fixed-point multiplier for the per-channel real scale
 *     M[n] = (sx * sw[n]) / sy          (double, in that order)
 * written as M[n] ~= M0[n] * 2^-shift[n] with M0 in [2^30, 2^31) and
 * shift in [1, 62].  Multipliers below 2^-32 (whose product with any int32
 * accumulator is under 1/2 in magnitude) are returned as M0 = 0, shift = 1.
 * Multipliers >= 2^30 are rejected (shift would be < 1).
 * Follows the fixed-point statement of Sec. 3.1 / Sec. 1 (all operations in
 * fixed point); the paper names no rounding mode, and one rounding, half
 * up, is taken.
 * Pinned by: power-of-two closed forms, relative-error bound 2^-31.
 */
int oracle_requant_params(float sx, const float *sw, int N, float sy,
                          int32_t *M0, int32_t *shift);

/*
 * Pack int8 weight values w[N][K] for `bits` = 8 (copy) or 4 (two's-complement
 * nibbles, low nibble = even k; values must lie in [-8, 7]) and compute
 * colsum[n] = sum_k w[n][k] in int32.  Pinned by: round trip, golden bytes,
 * brute-force sums.
 */
int oracle_pack(const int8_t *w, int N, int K, int bits, uint8_t *packed,
                int32_t *colsum);

/* Inverse of oracle_pack: packed -> int8 values [N][K]. */
int oracle_unpack(const uint8_t *packed, int N, int K, int bits, int8_t *w);

/*
 * The integer-only linear layer, straight from its definition:
 *   acc[m][n] = sum_k (x[m][k] - zx) * w[n][k]                (int64)
 *   v         = acc * M0[n]                                    (exact)
 *   q         = floor(v / 2^s + 1/2)     (round half up, s = shift[n])
 *   y[m][n]   = clamp(zy + q, -128, 127)
 * acc_out (may be NULL) receives acc as int32 [M][N] (row stride N).
 * Returns ORACLE_EOVERFLOW if any |acc| >= 2^31.
 * Pinned by: exhaustive K=1 brute force, zero-point identity, exact
 * dequantization invariant, closed-form requant and exact-rational ties.
 */
int oracle_linear(const int8_t *x, int M, int K, int ldx, int32_t zx,
                  const uint8_t *packed, int bits, int N, const int32_t *M0,
                  const int32_t *shift, int32_t zy, int8_t *y, int ldy,
                  int32_t *acc_out);

/*
 * The same layer evaluated only at the listed output coordinates
 * (m = pts[2i], n = pts[2i+1]); y_out[i] / acc_out[i] receive the results.
 * Used to check full-size problems on a sample of outputs.
 */
int oracle_linear_points(const int8_t *x, int M, int K, int ldx, int32_t zx,
                         const uint8_t *packed, int bits, int N,
                         const int32_t *M0, const int32_t *shift, int32_t zy,
                         const int64_t *pts, int count, int8_t *y_out,
                         int32_t *acc_out);

/*
 * The same layer with asymmetric weights: a per-output-channel weight zero
 * point zw[n] (zw == NULL: all zero, i.e. oracle_linear).  The paper's main
 * W8A8 / W4A8 runs quantize weights asymmetrically with the quantizer of
 * Sec. 4.2, eqs. 2-4 (per tensor, and per channel for the down projection,
 * Sec. 5.1); a per-tensor zero point is the case of equal zw[n].
 *   acc[m][n] = sum_k (x[m][k] - zx) * (w[n][k] - zw[n])           (int64)
 * then requantized exactly as in oracle_linear.  zw[n] must lie in the
 * weight code range ([-128, 127] for bits 8, [-8, 7] for bits 4).
 * Pinned by: exhaustive K=1 brute force over x and w for several zero points,
 * the expanded identity sum(xw) - zx colsum - zw rowsum(x) + K zx zw,
 * reduction to oracle_linear at zw = 0, exact dequantization.
 */
int oracle_linear_asym(const int8_t *x, int M, int K, int ldx, int32_t zx,
                       const uint8_t *packed, int bits, int N,
                       const int32_t *zw, const int32_t *M0,
                       const int32_t *shift, int32_t zy, int8_t *y, int ldy,
                       int32_t *acc_out);

/* oracle_linear_asym at listed output coordinates (as oracle_linear_points). */
int oracle_linear_points_asym(const int8_t *x, int M, int K, int ldx, int32_t zx,
                              const uint8_t *packed, int bits, int N,
                              const int32_t *zw, const int32_t *M0,
                              const int32_t *shift, int32_t zy,
                              const int64_t *pts, int count, int8_t *y_out,
                              int32_t *acc_out);

/*
 * The layer with 16-bit activations (W8A16 / W4A16): the paper keeps the
 * activations of its 16-bit baselines, and those around non-linear operators,
 * in 16-bit integers (Sec. 4.1 challenge i; Sec. 5.6 on-device settings
 * W8A16 and W4A16, Table 5).  The 16-bit unsigned code range is shifted by
 * -32768 to signed int16, as the 8-bit codes are by -128: x is int16 [M][ldx]
 * with zx in [-32768, 32767], the output y is int16 [M][ldy] with zy in
 * [-32768, 32767]; weights as in oracle_linear (symmetric per channel).
 *   acc[m][n] = sum_k (x[m][k] - zx) * w[n][k]      (int64; |acc| < 2^40)
 *   v         = acc * M0[n]                          (exact, __int128)
 *   q         = floor(v / 2^s + 1/2)                 (round half up)
 *   y[m][n]   = clamp(zy + q, -32768, 32767)
 * acc_out (may be NULL) receives acc as int64 [M][N] (row stride N).
 * K must not exceed 65536 (ORACLE_EINVAL).
 * Pinned by: brute force on Python integers and exact rationals, exhaustive
 * K=1 over all int16 activation codes, reduction to oracle_linear on int8
 * codes, the split into two int8 planes, exact dequantization, saturation.
 */
int oracle_linear_a16(const int16_t *x, int M, int K, int ldx, int32_t zx,
                      const uint8_t *packed, int bits, int N, const int32_t *M0,
                      const int32_t *shift, int32_t zy, int16_t *y, int ldy,
                      int64_t *acc_out);

/*
 * 8-bit inputs, 16-bit output: the product of two 8-bit activations (or
 * activations and weights) whose result feeds a non-linear operator, which
 * MobileQuant keeps in 16-bit integers (Sec. 4.1), e.g. the attention scores
 * Q K^T ahead of the softmax.  With int8 x [M][ldx], int8 / int4 w [N][K]
 * (packed as in oracle_linear) and an optional per-channel zero point zw
 * (NULL: 0):
 *   acc[m][n] = sum_k (x[m][k] - zx) * (w[n][k] - zw[n])      (int64)
 *   y[m][n]   = clamp(zy + floor(acc M0[n] / 2^s + 1/2), -32768, 32767)
 * zx in [-128, 127], zy in [-32768, 32767]; y is int16 [M][ldy].
 * Pinned by: its accumulator equals oracle_linear_asym's, its outputs are
 * oracle_requant_one_a16 of it, exhaustive K=1 with outputs checked against
 * exact rationals, saturation at the int16 ends.
 */
int oracle_linear_o16(const int8_t *x, int M, int K, int ldx, int32_t zx,
                      const uint8_t *packed, int bits, int N, const int32_t *zw,
                      const int32_t *M0, const int32_t *shift, int32_t zy, int16_t *y,
                      int ldy);

/*
 * 16-bit activations against weights (or 8-bit activations used as the
 * "weights" operand) with a per-channel zero point: the matmul of self-
 * attention in the paper's W8A16 setting, between 8-bit and 16-bit activations
 * (Sec. 5.6, on-device setup), and asymmetric weights (Sec. 5.1) under 16-bit
 * activations.  With x int16 [M][ldx], int8 / int4 w [N][K] and zw [N] in the
 * weight code range (NULL: 0):
 *   acc[m][n] = sum_k (x[m][k] - zx) * (w[n][k] - zw[n])      (int64)
 *   y[m][n]   = oracle_requant_one_a16(acc[m][n], M0[n], shift[n], zy)
 * Pinned by: exhaustive K=1 over every int16 code and every int8 weight code
 * with zero points at the range ends, against exact integers and rationals;
 * numpy's int64 matmul of the shifted operands; oracle_linear_a16 at zw = 0.
 */
int oracle_linear_a16_asym(const int16_t *x, int M, int K, int ldx, int32_t zx,
                           const uint8_t *packed, int bits, int N, const int32_t *zw,
                           const int32_t *M0, const int32_t *shift, int32_t zy, int16_t *y,
                           int ldy, int64_t *acc_out);

/* oracle_linear_a16 at listed output coordinates (as oracle_linear_points). */
int oracle_linear_points_a16(const int16_t *x, int M, int K, int ldx, int32_t zx,
                             const uint8_t *packed, int bits, int N,
                             const int32_t *M0, const int32_t *shift, int32_t zy,
                             const int64_t *pts, int count, int16_t *y_out,
                             int64_t *acc_out);

/* One 16-bit output: clamp(zy + floor(acc*M0 / 2^s + 1/2), -32768, 32767). */
int32_t oracle_requant_one_a16(int64_t acc, int32_t M0, int32_t shift, int32_t zy);

/*
 * Boundary quantizers between the float, int16 and int8 domains of an
 * integer block: the activations of linears are 8-bit, those around
 * non-linear operators 16-bit (Sec. 4.1, Sec. 1); every step is a static
 * per-tensor quantizer (Sec. 3.1).  `bits` selects int8 (8) or int16 (16)
 * codes, stored as int8_t / int16_t arrays.
 *
 * oracle_quantize_f32: the forward quantizer of eqs. 2-4, shifted to the
 * signed range: q = clamp(rint(x / alpha) + z, qmin, qmax).  The paper fixes
 * no precision or tie rule; the integer decision is taken in f32: x / alpha is the
 * correctly rounded f32 quotient and rint rounds ties to even; a NaN input
 * gives z.  alpha must be finite and > 0, z inside the code range.
 * Pinned by: exact rationals (f32 rounding of the true quotient, then ties to
 * even), dequantization within half a step, monotonicity, saturation.
 */
int oracle_quantize_f32(const float *x, int64_t n, float alpha, int32_t z, int bits,
                        void *q);

/*
 * Dequantization f = (q - z) * alpha, rounded once to f32 (the product of
 * an integer below 2^17 and an f32 is exact in double).
 * Pinned by: exact rationals, round trip with oracle_quantize_f32.
 */
int oracle_dequantize(const void *q, int bits, int64_t n, float alpha, int32_t z, float *f);

/*
 * Fixed-point requantization between integer domains (int8 / int16 in,
 * int8 / int16 out), the output quantizer of eq. 4 with the multiplier
 * alpha_in / alpha_out in the fixed-point form of oracle_requant_params:
 *   y = clamp(zy + floor(((q - zx) M0 + 2^(s-1)) / 2^s), ymin, ymax).
 * zx and zy lie in their domains' code ranges.
 * Pinned by: exhaustive sweeps over every int16 / int8 code against exact
 * rationals, the power-of-two closed form, eq. 4 with the real multiplier.
 */
int oracle_requantize(const void *q, int in_bits, int64_t n, int32_t zx, int32_t M0,
                      int32_t shift, int32_t zy, void *y, int out_bits);

/*
 * Offline weight preparation, step 1: the equivalent transform of eq. 1
 * folded into the weights.  With weights stored [N out][K in] (the transpose
 * of the paper's W), eq. 1's S W scales input channel k by s_in[k], and the
 * S^-1 of the next transform (Figure 3: S0 W1 S1^-1, S1 W2) scales output
 * channel n by 1 / s_out[n]:
 *   w_out[n][k] = (w[n][k] * s_in[k]) / s_out[n]
 * in f32, multiply first, each operation rounded to nearest; s_in or s_out
 * may be NULL (that factor is skipped).
 * Pinned by: exact rationals, float equivalence of eq. 1 through one layer
 * and through norm + two layers (Figure 3).
 */
int oracle_fold_weights(const float *w, int N, int K, const float *s_in, const float *s_out,
                        float *w_out);

/*
 * Step 2: weight quantization of f32 weights [N][K], the integer decisions
 * taken in f32 (the paper fixes no precision), per output channel or per tensor:
 *   scheme 0, symmetric per channel: amax = max|w[n]| (1e-8 if 0),
 *     sw = amax / qmax, q = clamp(rint(w / sw), -qmax, qmax) for int8
 *     (qmax 127) and clamp(., -8, 7) with qmax 7 for int4; zw = 0.
 *   scheme 1 / 2, asymmetric per channel / per tensor (eqs. 2-4 on weights,
 *     Sec. 5.1): lo = min(min w, 0), hi = max(max w, 0), span = hi - lo
 *     (1e-8 if 0), sw = span / (qmax - qmin), zw = clamp(rint(qmin - lo / sw)),
 *     q = clamp(rint(w / sw) + zw, qmin, qmax) with [qmin, qmax] the code range.
 * codes: int8 [N][K] (values in the bits' range), sw: f32 [N], zw: int32 [N]
 * (may be NULL for scheme 0).
 * Pinned by: exact rationals (every f32 operation rounded by hand), the code
 * range reached, the half-step bound, zero mapping to zw, per-tensor sharing.
 */
int oracle_quantize_weights(const float *w, int N, int K, int bits, int scheme, int8_t *codes,
                            float *sw, int32_t *zw);

/*
 * The norm's affine A before the first transformed linear absorbs S0^-1
 * (Figure 3): gamma'[k] = gamma[k] / s[k], beta'[k] = beta[k] / s[k] in f32.
 * beta / beta_out may be NULL (RMSNorm has no shift).
 */
int oracle_fold_norm(const float *gamma, const float *beta, const float *s, int K,
                     float *gamma_out, float *beta_out);

/*
 * Requantize one accumulator: clamp(zy + floor(acc*M0 / 2^s + 1/2), -128, 127).
 * Exposed so that tests can sweep accumulators around rounding ties.
 */
int32_t oracle_requant_one(int64_t acc, int32_t M0, int32_t shift, int32_t zy);

/*
 * Saturating int8 residual add, out[i] = clamp(a[i] + b[i], -128, 127): the
 * glue between chained layers of the 22-layer stack.
 */
void oracle_residual_add(const int8_t *a, const int8_t *b, int64_t n,
                         int8_t *out);

#ifdef __cplusplus
}
#endif
#endif
