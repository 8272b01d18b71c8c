/*
 * mq_oracle.c -- plain CPU oracle for the integer-only quantized linear layer
 * (MobileQuant, arXiv 2408.13933).  TEST INFRASTRUCTURE ONLY: the product path
 * never includes, links or calls this file.  See mq_oracle.h for the paper
 * passages each function follows.
 *
 * Written for readability, not speed: one output at a time, int64
 * accumulation, exact integer rounding with __int128.  No blocking, no
 * reordering beyond the definition.
 */
#include "mq_oracle.h"

#include <math.h>
#include <stddef.h>
#include <string.h>

/* One weight value w[n][k] from the packed buffer (int8 copy or int4 nibbles,
 * low nibble = even k, two's complement). */
static int oracle_weight_at(const uint8_t *packed, int bits, int K, int n,
                            int k) {
    if (bits == 8) {
        return (int)(int8_t)packed[(size_t)n * (size_t)K + (size_t)k];
    }
    uint8_t byte = packed[(size_t)n * (size_t)(K / 2) + (size_t)(k / 2)];
    int nibble = (k % 2 == 0) ? (byte & 0x0F) : (byte >> 4);
    return nibble >= 8 ? nibble - 16 : nibble;
}

/* floor(a / b) for b > 0, exact on 128-bit integers. */
static __int128 oracle_floor_div(__int128 a, __int128 b) {
    __int128 q = a / b;
    __int128 r = a % b;
    if (r != 0 && a < 0) q -= 1;
    return q;
}

int32_t oracle_requant_one(int64_t acc, int32_t M0, int32_t shift, int32_t zy) {
    /* v = acc * M0, exact (|acc| < 2^31, 0 <= M0 < 2^31). */
    __int128 v = (__int128)acc * (__int128)M0;
    /* q = floor(v / 2^s + 1/2) = floor((2v + 2^s) / 2^(s+1)): round half up. */
    __int128 two_s = (__int128)1 << shift;
    __int128 q = oracle_floor_div(2 * v + two_s, 2 * two_s);
    __int128 out = (__int128)zy + q;
    if (out < -128) out = -128;
    if (out > 127) out = 127;
    return (int32_t)out;
}

int oracle_requant_params(float sx, const float *sw, int N, float sy,
                          int32_t *M0, int32_t *shift) {
    if (N < 0 || (N > 0 && (!sw || !M0 || !shift))) return ORACLE_EINVAL;
    if (!(isfinite(sx) && sx > 0.0f) || !(isfinite(sy) && sy > 0.0f))
        return ORACLE_EINVAL;
    for (int n = 0; n < N; ++n) {
        if (!(isfinite(sw[n]) && sw[n] > 0.0f)) return ORACLE_EINVAL;
        /* Real per-channel multiplier: output scale sy maps the dequantized
         * product sx*sw[n]*acc back to the output grid. */
        double m = ((double)sx * (double)sw[n]) / (double)sy;
        int e = 0;
        double f = frexp(m, &e); /* m = f * 2^e, f in [0.5, 1) */
        long long m0 = llround(ldexp(f, 31));
        if (m0 == (1LL << 31)) { /* f rounded up to 1.0 */
            m0 = 1LL << 30;
            e += 1;
        }
        int s = 31 - e;
        if (s > 62) { /* |acc * m| < 1/2 for every int32 acc: output is zy */
            M0[n] = 0;
            shift[n] = 1;
            continue;
        }
        if (s < 1) return ORACLE_EINVAL;
        M0[n] = (int32_t)m0;
        shift[n] = s;
    }
    return ORACLE_OK;
}

int oracle_pack(const int8_t *w, int N, int K, int bits, uint8_t *packed,
                int32_t *colsum) {
    if (N < 0 || K < 0 || (bits != 8 && bits != 4)) return ORACLE_EINVAL;
    if (bits == 4 && K % 2 != 0) return ORACLE_EINVAL;
    for (int n = 0; n < N; ++n) {
        int64_t sum = 0;
        for (int k = 0; k < K; ++k) {
            int v = w[(size_t)n * (size_t)K + (size_t)k];
            if (bits == 4 && (v < -8 || v > 7)) return ORACLE_EINVAL;
            sum += v;
        }
        if (colsum) colsum[n] = (int32_t)sum;
        if (bits == 8) {
            memcpy(packed + (size_t)n * (size_t)K, w + (size_t)n * (size_t)K,
                   (size_t)K);
        } else {
            for (int j = 0; j < K / 2; ++j) {
                int lo = w[(size_t)n * (size_t)K + (size_t)(2 * j)];
                int hi = w[(size_t)n * (size_t)K + (size_t)(2 * j + 1)];
                packed[(size_t)n * (size_t)(K / 2) + (size_t)j] =
                    (uint8_t)((lo & 0x0F) | ((hi & 0x0F) << 4));
            }
        }
    }
    return ORACLE_OK;
}

int oracle_unpack(const uint8_t *packed, int N, int K, int bits, int8_t *w) {
    if (N < 0 || K < 0 || (bits != 8 && bits != 4)) return ORACLE_EINVAL;
    if (bits == 4 && K % 2 != 0) return ORACLE_EINVAL;
    for (int n = 0; n < N; ++n)
        for (int k = 0; k < K; ++k)
            w[(size_t)n * (size_t)K + (size_t)k] =
                (int8_t)oracle_weight_at(packed, bits, K, n, k);
    return ORACLE_OK;
}

/* acc = sum_k (x[m][k] - zx) * w[n][k] in int64. */
static int64_t oracle_dot(const int8_t *x, int K, int ldx, int32_t zx,
                          const uint8_t *packed, int bits, int m, int n) {
    int64_t acc = 0;
    for (int k = 0; k < K; ++k) {
        int64_t xv = (int64_t)x[(size_t)m * (size_t)ldx + (size_t)k] - zx;
        int64_t wv = oracle_weight_at(packed, bits, K, n, k);
        acc += xv * wv;
    }
    return acc;
}

static int oracle_check_args(int M, int K, int ldx, int bits, int N,
                             int32_t zx, int32_t zy) {
    if (M < 0 || K < 0 || N < 0) return ORACLE_EINVAL;
    if (bits != 8 && bits != 4) return ORACLE_EINVAL;
    if (bits == 4 && K % 2 != 0) return ORACLE_EINVAL;
    if (ldx < K) return ORACLE_EINVAL;
    if (zx < -128 || zx > 127 || zy < -128 || zy > 127) return ORACLE_EINVAL;
    return ORACLE_OK;
}

int oracle_linear(const int8_t *x, int M, int K, int ldx, int32_t zx,
                  const uint8_t *packed, int bits, int N, const int32_t *M0,
                  const int32_t *shift, int32_t zy, int8_t *y, int ldy,
                  int32_t *acc_out) {
    int rc = oracle_check_args(M, K, ldx, bits, N, zx, zy);
    if (rc != ORACLE_OK) return rc;
    if (ldy < N) return ORACLE_EINVAL;
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            int64_t acc = oracle_dot(x, K, ldx, zx, packed, bits, m, n);
            if (acc >= ((int64_t)1 << 31) || acc < -((int64_t)1 << 31))
                return ORACLE_EOVERFLOW;
            if (acc_out) acc_out[(size_t)m * (size_t)N + (size_t)n] = (int32_t)acc;
            if (y)
                y[(size_t)m * (size_t)ldy + (size_t)n] =
                    (int8_t)oracle_requant_one(acc, M0[n], shift[n], zy);
        }
    }
    return ORACLE_OK;
}

int oracle_linear_points(const int8_t *x, int M, int K, int ldx, int32_t zx,
                         const uint8_t *packed, int bits, int N,
                         const int32_t *M0, const int32_t *shift, int32_t zy,
                         const int64_t *pts, int count, int8_t *y_out,
                         int32_t *acc_out) {
    int rc = oracle_check_args(M, K, ldx, bits, N, zx, zy);
    if (rc != ORACLE_OK) return rc;
    for (int i = 0; i < count; ++i) {
        int64_t m = pts[2 * i], n = pts[2 * i + 1];
        if (m < 0 || m >= M || n < 0 || n >= N) return ORACLE_EINVAL;
        int64_t acc = oracle_dot(x, K, ldx, zx, packed, bits, (int)m, (int)n);
        if (acc >= ((int64_t)1 << 31) || acc < -((int64_t)1 << 31))
            return ORACLE_EOVERFLOW;
        if (acc_out) acc_out[i] = (int32_t)acc;
        if (y_out) y_out[i] = (int8_t)oracle_requant_one(acc, M0[n], shift[n], zy);
    }
    return ORACLE_OK;
}

/* sum_k (x[m][k] - zx) * (w[n][k] - zw), the asymmetric-weight dot product. */
static int64_t oracle_dot_asym(const int8_t *x, int K, int ldx, int32_t zx,
                               const uint8_t *packed, int bits, int m, int n,
                               int32_t zw) {
    int64_t acc = 0;
    for (int k = 0; k < K; ++k) {
        int64_t xv = (int64_t)x[(size_t)m * (size_t)ldx + (size_t)k] - zx;
        int64_t wv = oracle_weight_at(packed, bits, K, n, k) - zw;
        acc += xv * wv;
    }
    return acc;
}

static int oracle_check_zw(const int32_t *zw, int N, int bits) {
    if (!zw) return ORACLE_OK;
    const int32_t lo = bits == 8 ? -128 : -8, hi = bits == 8 ? 127 : 7;
    for (int n = 0; n < N; ++n)
        if (zw[n] < lo || zw[n] > hi) return ORACLE_EINVAL;
    return ORACLE_OK;
}

int oracle_linear_asym(const int8_t *x, int M, int K, int ldx, int32_t zx,
                       const uint8_t *packed, int bits, int N,
                       const int32_t *zw, const int32_t *M0,
                       const int32_t *shift, int32_t zy, int8_t *y, int ldy,
                       int32_t *acc_out) {
    int rc = oracle_check_args(M, K, ldx, bits, N, zx, zy);
    if (rc != ORACLE_OK) return rc;
    if (ldy < N) return ORACLE_EINVAL;
    rc = oracle_check_zw(zw, N, bits);
    if (rc != ORACLE_OK) return rc;
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            int64_t acc = oracle_dot_asym(x, K, ldx, zx, packed, bits, m, n, zw ? zw[n] : 0);
            if (acc >= ((int64_t)1 << 31) || acc < -((int64_t)1 << 31))
                return ORACLE_EOVERFLOW;
            if (acc_out) acc_out[(size_t)m * (size_t)N + (size_t)n] = (int32_t)acc;
            if (y)
                y[(size_t)m * (size_t)ldy + (size_t)n] =
                    (int8_t)oracle_requant_one(acc, M0[n], shift[n], zy);
        }
    }
    return ORACLE_OK;
}

int oracle_linear_points_asym(const int8_t *x, int M, int K, int ldx, int32_t zx,
                              const uint8_t *packed, int bits, int N,
                              const int32_t *zw, const int32_t *M0,
                              const int32_t *shift, int32_t zy,
                              const int64_t *pts, int count, int8_t *y_out,
                              int32_t *acc_out) {
    int rc = oracle_check_args(M, K, ldx, bits, N, zx, zy);
    if (rc != ORACLE_OK) return rc;
    rc = oracle_check_zw(zw, N, bits);
    if (rc != ORACLE_OK) return rc;
    for (int i = 0; i < count; ++i) {
        int64_t m = pts[2 * i], n = pts[2 * i + 1];
        if (m < 0 || m >= M || n < 0 || n >= N) return ORACLE_EINVAL;
        int64_t acc = oracle_dot_asym(x, K, ldx, zx, packed, bits, (int)m, (int)n,
                                      zw ? zw[n] : 0);
        if (acc >= ((int64_t)1 << 31) || acc < -((int64_t)1 << 31))
            return ORACLE_EOVERFLOW;
        if (acc_out) acc_out[i] = (int32_t)acc;
        if (y_out) y_out[i] = (int8_t)oracle_requant_one(acc, M0[n], shift[n], zy);
    }
    return ORACLE_OK;
}

/* floor(acc * M0 / 2^s + 1/2) on exact integers (|acc| < 2^40, M0 < 2^31,
 * so |2 acc M0 + 2^s| < 2^73). */
static __int128 oracle_round_shift(int64_t acc, int32_t M0, int32_t shift) {
    __int128 v = (__int128)acc * (__int128)M0;
    __int128 two_s = (__int128)1 << shift;
    return oracle_floor_div(2 * v + two_s, 2 * two_s);
}

int32_t oracle_requant_one_a16(int64_t acc, int32_t M0, int32_t shift, int32_t zy) {
    __int128 out = (__int128)zy + oracle_round_shift(acc, M0, shift);
    if (out < -32768) out = -32768;
    if (out > 32767) out = 32767;
    return (int32_t)out;
}

/* acc = sum_k (x[m][k] - zx) * w[n][k] in int64, 16-bit activations. */
static int64_t oracle_dot_a16(const int16_t *x, int K, int ldx, int32_t zx,
                              const uint8_t *packed, int bits, int m, int n) {
    int64_t acc16 = 0;
    for (int k = 0; k < K; ++k) {
        int64_t x16 = (int64_t)x[(size_t)m * (size_t)ldx + (size_t)k] - (int64_t)zx;
        int64_t w16 = oracle_weight_at(packed, bits, K, n, k);
        acc16 += x16 * w16;
    }
    return acc16;
}

static int oracle_check_args_a16(int M, int K, int ldx, int bits, int N,
                                 int32_t zx, int32_t zy) {
    if (M < 0 || K < 0 || N < 0 || K > 65536) return ORACLE_EINVAL;
    if (bits != 8 && bits != 4) return ORACLE_EINVAL;
    if (bits == 4 && K % 2 != 0) return ORACLE_EINVAL;
    if (ldx < K) return ORACLE_EINVAL;
    if (zx < -32768 || zx > 32767 || zy < -32768 || zy > 32767) return ORACLE_EINVAL;
    return ORACLE_OK;
}

int oracle_linear_a16(const int16_t *x, int M, int K, int ldx, int32_t zx,
                      const uint8_t *packed, int bits, int N, const int32_t *M0,
                      const int32_t *shift, int32_t zy, int16_t *y, int ldy,
                      int64_t *acc_out) {
    int rc = oracle_check_args_a16(M, K, ldx, bits, N, zx, zy);
    if (rc != ORACLE_OK) return rc;
    if (ldy < N) return ORACLE_EINVAL;
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            int64_t acc = oracle_dot_a16(x, K, ldx, zx, packed, bits, m, n);
            if (acc_out) acc_out[(size_t)m * (size_t)N + (size_t)n] = acc;
            if (y)
                y[(size_t)m * (size_t)ldy + (size_t)n] =
                    (int16_t)oracle_requant_one_a16(acc, M0[n], shift[n], zy);
        }
    }
    return ORACLE_OK;
}

int oracle_linear_a16_asym(const int16_t *x, int M, int K, int ldx, int32_t zx,
                           const uint8_t *packed, int bits, int N, const int32_t *zw,
                           const int32_t *M0, const int32_t *shift, int32_t zy, int16_t *y,
                           int ldy, int64_t *acc_out) {
    int rc = oracle_check_args_a16(M, K, ldx, bits, N, zx, zy);
    if (rc != ORACLE_OK) return rc;
    if (ldy < N) return ORACLE_EINVAL;
    rc = oracle_check_zw(zw, N, bits);
    if (rc != ORACLE_OK) return rc;
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            const int64_t zwn = zw ? (int64_t)zw[n] : 0;
            int64_t acc = 0;
            for (int k = 0; k < K; ++k) {
                int64_t xv = (int64_t)x[(size_t)m * (size_t)ldx + (size_t)k] - (int64_t)zx;
                int64_t wv = oracle_weight_at(packed, bits, K, n, k) - zwn;
                acc += xv * wv;
            }
            if (acc_out) acc_out[(size_t)m * (size_t)N + (size_t)n] = acc;
            if (y)
                y[(size_t)m * (size_t)ldy + (size_t)n] =
                    (int16_t)oracle_requant_one_a16(acc, M0[n], shift[n], zy);
        }
    }
    return ORACLE_OK;
}

int oracle_linear_points_a16(const int16_t *x, int M, int K, int ldx, int32_t zx,
                             const uint8_t *packed, int bits, int N,
                             const int32_t *M0, const int32_t *shift, int32_t zy,
                             const int64_t *pts, int count, int16_t *y_out,
                             int64_t *acc_out) {
    int rc = oracle_check_args_a16(M, K, ldx, bits, N, zx, zy);
    if (rc != ORACLE_OK) return rc;
    for (int i = 0; i < count; ++i) {
        int64_t m = pts[2 * i], n = pts[2 * i + 1];
        if (m < 0 || m >= M || n < 0 || n >= N) return ORACLE_EINVAL;
        int64_t acc = oracle_dot_a16(x, K, ldx, zx, packed, bits, (int)m, (int)n);
        if (acc_out) acc_out[i] = acc;
        if (y_out) y_out[i] = (int16_t)oracle_requant_one_a16(acc, M0[n], shift[n], zy);
    }
    return ORACLE_OK;
}

int oracle_linear_o16(const int8_t *x, int M, int K, int ldx, int32_t zx,
                      const uint8_t *packed, int bits, int N, const int32_t *zw,
                      const int32_t *M0, const int32_t *shift, int32_t zy, int16_t *y,
                      int ldy) {
    if (M < 0 || K < 0 || N < 0 || (bits != 8 && bits != 4) || ldx < K || ldy < N)
        return ORACLE_EINVAL;
    if (bits == 4 && K % 2 != 0) return ORACLE_EINVAL;
    if (zx < -128 || zx > 127 || zy < -32768 || zy > 32767) return ORACLE_EINVAL;
    int rc = oracle_check_zw(zw, N, bits);
    if (rc != ORACLE_OK) return rc;
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            int64_t wide = oracle_dot_asym(x, K, ldx, zx, packed, bits, m, n, zw ? zw[n] : 0);
            y[(size_t)m * (size_t)ldy + (size_t)n] =
                (int16_t)oracle_requant_one_a16(wide, M0[n], shift[n], zy);
        }
    }
    return ORACLE_OK;
}

static int oracle_code_range(int bits, int32_t *lo, int32_t *hi) {
    if (bits == 8) {
        *lo = -128;
        *hi = 127;
        return ORACLE_OK;
    }
    if (bits == 16) {
        *lo = -32768;
        *hi = 32767;
        return ORACLE_OK;
    }
    return ORACLE_EINVAL;
}

static int32_t oracle_code_at(const void *q, int bits, int64_t i) {
    return bits == 8 ? (int32_t)((const int8_t *)q)[i] : (int32_t)((const int16_t *)q)[i];
}

static void oracle_code_store(void *q, int bits, int64_t i, int32_t v) {
    if (bits == 8)
        ((int8_t *)q)[i] = (int8_t)v;
    else
        ((int16_t *)q)[i] = (int16_t)v;
}

int oracle_quantize_f32(const float *x, int64_t n, float alpha, int32_t z, int bits,
                        void *q) {
    int32_t lo, hi;
    if (oracle_code_range(bits, &lo, &hi) != ORACLE_OK || n < 0) return ORACLE_EINVAL;
    if (!(isfinite(alpha) && alpha > 0.0f) || z < lo || z > hi) return ORACLE_EINVAL;
    for (int64_t i = 0; i < n; ++i) {
        float quotient = x[i] / alpha; /* f32 division, rounded to nearest */
        int32_t code;
        if (isnan(quotient)) {
            code = z;
        } else {
            double t = (double)rintf(quotient) + (double)z; /* ties to even */
            if (t < lo) t = lo;
            if (t > hi) t = hi;
            code = (int32_t)t;
        }
        oracle_code_store(q, bits, i, code);
    }
    return ORACLE_OK;
}

int oracle_dequantize(const void *q, int bits, int64_t n, float alpha, int32_t z, float *f) {
    int32_t lo, hi;
    if (oracle_code_range(bits, &lo, &hi) != ORACLE_OK || n < 0) return ORACLE_EINVAL;
    if (!isfinite(alpha) || z < lo || z > hi) return ORACLE_EINVAL;
    for (int64_t i = 0; i < n; ++i) {
        double exact = (double)(oracle_code_at(q, bits, i) - z) * (double)alpha;
        f[i] = (float)exact;
    }
    return ORACLE_OK;
}

int oracle_requantize(const void *q, int in_bits, int64_t n, int32_t zx, int32_t M0,
                      int32_t shift, int32_t zy, void *y, int out_bits) {
    int32_t ilo, ihi, olo, ohi;
    if (oracle_code_range(in_bits, &ilo, &ihi) != ORACLE_OK ||
        oracle_code_range(out_bits, &olo, &ohi) != ORACLE_OK || n < 0)
        return ORACLE_EINVAL;
    if (zx < ilo || zx > ihi || zy < olo || zy > ohi) return ORACLE_EINVAL;
    if (M0 < 0 || shift < 1 || shift > 62) return ORACLE_EINVAL;
    for (int64_t i = 0; i < n; ++i) {
        int64_t centered = (int64_t)oracle_code_at(q, in_bits, i) - zx;
        __int128 rounded = oracle_round_shift(centered, M0, shift);
        __int128 out = (__int128)zy + rounded;
        if (out < olo) out = olo;
        if (out > ohi) out = ohi;
        oracle_code_store(y, out_bits, i, (int32_t)out);
    }
    return ORACLE_OK;
}

int oracle_fold_weights(const float *w, int N, int K, const float *s_in, const float *s_out,
                        float *w_out) {
    if (N < 0 || K < 0) return ORACLE_EINVAL;
    for (int n = 0; n < N; ++n)
        for (int k = 0; k < K; ++k) {
            float v = w[(size_t)n * (size_t)K + (size_t)k];
            if (s_in) v = v * s_in[k];   /* S W: input channel k */
            if (s_out) v = v / s_out[n]; /* S^-1 of the next transform: output channel n */
            w_out[(size_t)n * (size_t)K + (size_t)k] = v;
        }
    return ORACLE_OK;
}

int oracle_quantize_weights(const float *w, int N, int K, int bits, int scheme, int8_t *codes,
                            float *sw, int32_t *zw) {
    if (N < 0 || K < 0 || (bits != 8 && bits != 4) || scheme < 0 || scheme > 2)
        return ORACLE_EINVAL;
    if (scheme != 0 && !zw) return ORACLE_EINVAL;
    const int32_t qmin = bits == 8 ? -128 : -8, qmax = bits == 8 ? 127 : 7;
    /* per-tensor statistics (scheme 2) */
    float tlo = 0.0f, thi = 0.0f;
    for (int n = 0; scheme == 2 && n < N; ++n)
        for (int k = 0; k < K; ++k) {
            float v = w[(size_t)n * (size_t)K + (size_t)k];
            if (v < tlo) tlo = v;
            if (v > thi) thi = v;
        }
    for (int n = 0; n < N; ++n) {
        const float *row = w + (size_t)n * (size_t)K;
        float lo = 0.0f, hi = 0.0f;
        if (scheme == 2) {
            lo = tlo;
            hi = thi;
        } else {
            for (int k = 0; k < K; ++k) {
                if (row[k] < lo) lo = row[k];
                if (row[k] > hi) hi = row[k];
            }
        }
        float scale;
        int32_t zero = 0;
        if (scheme == 0) {
            float amax = -lo > hi ? -lo : hi;
            if (!(amax > 0.0f)) amax = 1e-8f;
            scale = amax / (float)qmax;
        } else {
            float span = hi - lo;
            if (!(span > 0.0f)) span = 1e-8f;
            scale = span / (float)(qmax - qmin);
            float zf = rintf((float)qmin - lo / scale);
            zero = (int32_t)(zf < qmin ? qmin : (zf > qmax ? qmax : zf));
        }
        const int32_t cmin = (scheme == 0 && bits == 8) ? -qmax : qmin;
        for (int k = 0; k < K; ++k) {
            double c = (double)rintf(row[k] / scale) + (double)zero;
            if (c < cmin) c = cmin;
            if (c > qmax) c = qmax;
            codes[(size_t)n * (size_t)K + (size_t)k] = (int8_t)c;
        }
        sw[n] = scale;
        if (zw) zw[n] = zero;
    }
    return ORACLE_OK;
}

int oracle_fold_norm(const float *gamma, const float *beta, const float *s, int K,
                     float *gamma_out, float *beta_out) {
    if (K < 0 || (K > 0 && (!gamma || !s || !gamma_out))) return ORACLE_EINVAL;
    for (int k = 0; k < K; ++k) {
        gamma_out[k] = gamma[k] / s[k];
        if (beta && beta_out) beta_out[k] = beta[k] / s[k];
    }
    return ORACLE_OK;
}

void oracle_residual_add(const int8_t *a, const int8_t *b, int64_t n,
                         int8_t *out) {
    for (int64_t i = 0; i < n; ++i) {
        int v = (int)a[i] + (int)b[i];
        out[i] = (int8_t)(v < -128 ? -128 : (v > 127 ? 127 : v));
    }
}
