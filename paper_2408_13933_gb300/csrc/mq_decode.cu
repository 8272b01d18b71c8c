// mq_decode.cu -- weight-streaming kernel for the integer-only quantized
// linear layer at decode sizes (M <= 16 tokens), bit-exact.
//
// At M <= 16 the layer reads each weight once and does at most 16 MACs with
// it, so its speed is the weight stream (the paper notes that autoregressive
// generation is memory-bound, Sec. 5.6 and Appendix A.2).
//
// Schedule (stream-K).  The work of up to DECODE_MAX_PROBLEMS linears is cut
// into 64-row units and each unit into stages of KSTAGE values of k; the
// global sequence of stages is split evenly among the CTAs of a persistent
// grid (two per SM), so every SM streams the same number of weight bytes no
// matter how the linears' sizes differ.  A unit whose stages fall to several
// CTAs is finished by its first CTA, which reaches the unit at the end of its
// range; the later contributors, which process the unit's tail at the start
// of theirs, store their int32 partial sums in their own workspace slot as
// 8-byte words {sum, launch epoch} (a thread's words adjacent) and go on
// without waiting.  The first CTA reads a contributor's words before its own
// last stage of the unit, polls only words that do not carry the epoch yet,
// adds them, requantizes, and stores zero back, so the workspace is left zero.
//
// Data path.  In each CTA one producer thread streams the weight rows of its
// stages with TMA into a 7-stage (one token tile) or 6-stage (two) shared-
// memory ring, continuing across unit boundaries.  A stage holds 64 weight
// rows x 128 bytes and the matching k slice of the 16 (zero-padded) token rows
// of x, both 128-byte swizzled, so up to 56 KB of weights per CTA are in
// flight and the activation fragments come from shared memory without bank
// conflicts.
// Eight consumer warps read the ring, widen weights in registers to f16 and multiply with warp-level
// mma.sync m16n8k16 (f16 x f16 -> f32): weights are the 16-row A operand, the
// (zero-padded) tokens the 8-column B operand.  Warp w of the consumers owns
// the 16-byte chunk w of every row of a stage (conflict-free under the
// swizzle) for all four 16-row tiles of the unit, so one activation fragment
// serves four weight tiles.
//
// Widening.  A weight code is made unsigned (u = w + 8 for int4, u = w + 128
// for int8) and placed unchanged in the low mantissa bits of an f16 whose
// exponent field is zero: that is the f16 subnormal u * 2^-24, exact, made by
// one LOP3 per two weights.  int4 nibbles at bits 4-7 of a half become
// 16 u * 2^-24; they are multiplied with activations scaled by 1/16 (exact in
// f16), so every product lands on the common scale 2^-24.  The accumulator
// holds S = sum(u x) * 2^-24 exactly while |sum(u x)| < 2^24 (int4: 8738
// values of k per warp, int8: 514); int8 partials are flushed to int32 every
// 512 values of k per warp, int4 never needs a flush (a warp sees at most
// MQ_MAX_K / 8 = 8192 values of k).  The bias is removed exactly in the
// epilogue with the token's activation sum: sum(w x) = sum(u x) - 8 sum(x)
// (int4) or - 128 sum(x) (int8).
//
// The reduction order over k inside one mma is free, so each fragment slot's
// k index is whatever the unpacking yields; the activation fragments use the
// same assignment.
//
// Epilogue (per unit): each warp writes its int32 partials and activation sums
// to its own shared-memory slice; every thread then sums a fixed set of slots
// over the eight warps; acc = sum(u x) - bias sum(x) - zx colsum[n], then
// fixed-point requant (round half up), saturation, optional residual, store.
// Launches use programmatic dependent launch: the first ring stages' weights
// are requested before waiting for the previous kernel in the stream.
// All mbarrier waits are bounded (mq_wait_parity).
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <atomic>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {
namespace decode {

constexpr int CONS_WARPS = 8;
constexpr int CONS_THREADS = CONS_WARPS * 32;
constexpr int PROD_WARP = CONS_WARPS;  // warp 8
constexpr int THREADS = CONS_THREADS + 32;
constexpr int UNIT_ROWS = 64;          // four 16-row mma tiles
constexpr int ROW_BYTES = 128;         // weight bytes per row per stage
constexpr int W_BYTES = UNIT_ROWS * ROW_BYTES;  // 8 KB of weights
constexpr int X_BOX = 16 * 128;                 // one x box: 16 tokens x 128 k
constexpr int X16_BOX = 8 * 128;                // one 16-bit x box: 8 tokens x 64 codes
constexpr int STAGE_BYTES = W_BYTES + 2 * X_BOX;
// Ring depth: the cross-warp reduction buffer grows with the token tiles, so
// the ring shrinks to keep two CTAs per SM.
template <int NT>
constexpr int stages_for() { return NT == 1 ? 7 : 6; }
constexpr int CONS_BARRIER = 1;        // named barrier among the consumer warps

struct Params {
    CUtensorMap tmap_w[DECODE_MAX_PROBLEMS];  // weight bytes [N][K*bits/8], box 128 x 64, 128B swizzle
    CUtensorMap tmap_x[DECODE_MAX_PROBLEMS];  // x [M][ldx], box 128 x 16, 128B swizzle
    Problem p[DECODE_MAX_PROBLEMS];  // tile_begin = first global stage, tiles_m = stages per unit
    int count;
    int total_stages;
    int2 *ws;            // [gridDim.x][UNIT_ROWS * 16] 8-byte {sum, epoch} words (zero between calls)
    uint32_t epoch;      // nonzero, different for every launch
    int wide;            // total_stages * gridDim.x >= 2^32: 64-bit range arithmetic
    int pre_w;           // 1: load weights before griddep_wait (all constant)
    int skip_cta;        // failure-detection test: this CTA stores no split-unit sums (-1: none)
    int *status;
    uint64_t wait_ns;    // limit of every bounded wait
};

// What the kernel reads of a problem, kept in shared memory (the TMA tensor
// maps replace x and the weights).
struct DecProb {
    const int32_t *colsum;
    const int32_t *M0;
    const int32_t *shift;
    const int8_t *residual;
    const int32_t *zw;
    int8_t *y;
    int32_t M, N, K, ldy, zx, zy;
    int32_t tile_begin;  // first global stage
    int32_t tiles_m;     // stages per unit
};

__device__ __forceinline__ DecProb dec_prob(const Problem &p) {
    DecProb d;
    d.colsum = p.colsum;
    d.M0 = p.M0;
    d.shift = p.shift;
    d.residual = p.residual;
    d.zw = p.zw;
    d.y = p.y;
    d.M = p.M;
    d.N = p.N;
    d.K = p.K;
    d.ldy = p.ldy;
    d.zx = p.zx;
    d.zy = p.zy;
    d.tile_begin = p.tile_begin;
    d.tiles_m = p.tiles_m;
    return d;
}

template <int NT>
struct Smem {
    static constexpr int STAGES = stages_for<NT>();
    uint8_t ring[STAGES][STAGE_BYTES];
    uint64_t full[STAGES];
    uint64_t empty[STAGES];
    // each consumer warp's int32 partial sums of a piece, by mma fragment
    // element e = (rt * NT + nt) * 4 + i and lane (conflict-free both ways)
    int32_t part[CONS_WARPS][16 * NT][32];
    int32_t xpart[CONS_WARPS][16];  // each warp's activation sums per token
    int32_t row_corr[UNIT_ROWS];  // zx * colsum[n] - K zx zw[n] of the current unit's rows
    int32_t row_zw[UNIT_ROWS];    // weight zero points of the current unit's rows
    int32_t row_m0[UNIT_ROWS];
    int32_t row_shift[UNIT_ROWS];
    DecProb prob[DECODE_MAX_PROBLEMS];  // the kernel's problem table, read once
    int abort;
};

template <int NT>
constexpr size_t smem_bytes() { return sizeof(Smem<NT>) + 1024; }

__device__ __forceinline__ void cons_sync() {
    asm volatile("bar.sync %0, %1;" ::"n"(CONS_BARRIER), "n"(CONS_THREADS) : "memory");
}

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ int dp4a_sum(uint32_t w, int acc) {
    return __dp4a((int)w, 0x01010101, acc);
}

__device__ __forceinline__ uint32_t lds32(const uint8_t *p) {
    return *reinterpret_cast<const uint32_t *>(p);
}

// Two chosen activation bytes of the word pair (a, b) -> an exact f16 pair:
// byte ^ 0x80 = x + 128 as mantissa of 1024, minus 1152.  `scaled` gives
// (x/16) instead: (1024 + x + 128)/16 - 72.
__device__ __forceinline__ uint32_t x_pair(uint32_t a, uint32_t b, uint32_t sel, bool scaled) {
    const uint32_t t = prmt(a ^ 0x80808080u, b ^ 0x80808080u, sel);  // bytes [p, q, ., .]
    const uint32_t h = prmt(t, 0x64646464u, 0x5140u);                // bytes [p, 64, q, 64]
    return scaled ? hfma2(h, 0x2C002C00u, 0xD480D480u) : hsub2(h, F16X2_1152);
}

template <int BITS>
struct Cfg;
template <>
struct Cfg<4> {
    static constexpr int KSTAGE = 256;       // k per stage (128 bytes per row)
    static constexpr int KWARP = 32;         // k per consumer warp per stage
    static constexpr bool FLUSH = false;     // 15 * 128 * 8192 < 2^24
    static constexpr int FLUSH_STAGES = 1;
    static constexpr int BIAS = 8;
};
template <>
struct Cfg<8> {
    static constexpr int KSTAGE = 128;
    static constexpr int KWARP = 16;
    static constexpr bool FLUSH = true;
    static constexpr int FLUSH_STAGES = 32;  // 512 k per warp: 255 * 128 * 512 < 2^24
    static constexpr int BIAS = 128;
};

// First global stage of CTA c when S stages are split among G CTAs.  With
// S * G < 2^32 (the launcher sets `wide` otherwise) the products fit 32 bits:
// a 64-bit division is a long software sequence, and these run in every
// CTA's prologue and for every split unit.
__device__ __forceinline__ int range_begin(int c, int S, int G, bool wide) {
    return wide ? (int)(((long long)c * S) / G)
                : (int)(((uint32_t)c * (uint32_t)S) / (uint32_t)G);
}

// The CTA whose range holds global stage s.
__device__ __forceinline__ int cta_of(int s, int S, int G, bool wide) {
    int c = wide ? (int)(((long long)s * G) / S) : (int)(((uint32_t)s * (uint32_t)G) / (uint32_t)S);
    while (c + 1 < G && range_begin(c + 1, S, G, wide) <= s) ++c;
    while (c > 0 && range_begin(c, S, G, wide) > s) --c;
    return c;
}

// Problem holding global stage s, searching forward from `pi` (stages are
// visited in increasing order, so the walk is amortized O(1)).
template <class SM>
__device__ __forceinline__ int problem_from(const SM &sm, int count, int pi, int s) {
    while (pi + 1 < count && s >= sm.prob[pi + 1].tile_begin) ++pi;
    return pi;
}

// Split-unit entries in the workspace: per CTA slot, consumer thread t's
// 2 NT sums at words [2 NT t, 2 NT t + 2 NT), each one 8-byte word {sum in the
// low half, launch epoch in the high half}.  An aligned 8-byte access is
// single-copy atomic, so a reader sees either zero or the whole entry; a
// thread's words are adjacent, so a pair of them is one 16-byte access.  The
// mapping from a thread to its outputs depends only on the thread index, so
// thread t of the finishing CTA reads exactly what thread t of a contributor
// wrote.
template <int NT>
__device__ __forceinline__ uint64_t *unit_entries(const Params &P, int c) {
    return reinterpret_cast<uint64_t *>(P.ws) + (size_t)c * UNIT_ROWS * 16 +
           (size_t)threadIdx.x * (2 * NT);
}

__device__ __forceinline__ uint64_t pack_entry(uint32_t v, uint32_t epoch) {
    return (uint64_t)v | ((uint64_t)epoch << 32);
}

__device__ __forceinline__ void st_pair(uint64_t *p, uint64_t a, uint64_t b) {
    asm volatile("st.relaxed.gpu.global.v2.b64 [%0], {%1, %2};" ::"l"(p), "l"(a), "l"(b)
                 : "memory");
}

__device__ __forceinline__ void ld_pair(const uint64_t *p, uint64_t &a, uint64_t &b) {
    asm volatile("ld.relaxed.gpu.global.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "l"(p)
                 : "memory");
}

// Wait (bounded, like every wait in this library) until the word carries
// `epoch`; the word is returned in `w`.
__device__ __forceinline__ bool poll_word(const uint64_t *p, uint32_t epoch, uint64_t &w,
                                          volatile int *abort, int *status, uint64_t limit_ns) {
    uint64_t t0 = 0;
    while (true) {
        asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(w) : "l"(p) : "memory");
        if ((uint32_t)(w >> 32) == epoch) return true;
        if (*abort) return false;
        const uint64_t t = global_timer_ns();
        if (t0 == 0) {
            t0 = t;
        } else if (t - t0 > limit_ns) {
            *abort = 1;
            atomicOr(status, MQ_DEVICE_STATUS_TIMEOUT);
            return false;
        }
        __nanosleep(128);
    }
}

// A contributor's sums, stored with this launch's epoch; it does not wait.
// (The failure-detection test names one CTA that skips its stores, so that
// the finishing CTA's bounded wait for them runs out.)
template <int NT>
__device__ __forceinline__ void put_partials(const Params &P, int cta, const uint32_t (&v)[2 * NT]) {
    if (cta == P.skip_cta) return;
    uint64_t *m = unit_entries<NT>(P, cta);
#pragma unroll
    for (int q = 0; q < 2 * NT; q += 2)
        st_pair(m + q, pack_entry(v[q], P.epoch), pack_entry(v[q + 1], P.epoch));
}

// A read of CTA c's entries for this thread (possibly before they are written).
template <int NT>
__device__ __forceinline__ void read_partials(const Params &P, int c, uint64_t (&e)[2 * NT]) {
    const uint64_t *src = unit_entries<NT>(P, c);
#pragma unroll
    for (int q = 0; q < 2 * NT; q += 2) ld_pair(src + q, e[q], e[q + 1]);
}

// The finishing CTA adds the sums of contributors cf + 1 .. cl into v.  `first`
// is an earlier read of CTA cf + 1's entries; words that do not carry this
// launch's epoch yet are polled.  Every entry read is stored back as zero.
template <int NT>
__device__ __forceinline__ bool gather_partials(const Params &P, volatile int *abort, int cf,
                                                int cl, const uint64_t (&first)[2 * NT],
                                                uint32_t (&v)[2 * NT]) {
    bool got = true;
    for (int c = cf + 1; got && c <= cl; ++c) {
        uint64_t e[2 * NT];
        if (c == cf + 1) {
#pragma unroll
            for (int q = 0; q < 2 * NT; ++q) e[q] = first[q];
        } else {
            read_partials<NT>(P, c, e);
        }
        const uint64_t *src = unit_entries<NT>(P, c);
#pragma unroll
        for (int q = 0; q < 2 * NT; ++q) {
            if ((uint32_t)(e[q] >> 32) != P.epoch)
                got = got && poll_word(src + q, P.epoch, e[q], abort, P.status, P.wait_ns);
            v[q] += (uint32_t)e[q];
        }
    }
    if (got)
        for (int c = cf + 1; c <= cl; ++c) {
            uint64_t *src = unit_entries<NT>(P, c);
#pragma unroll
            for (int q = 0; q < 2 * NT; q += 2) st_pair(src + q, 0ull, 0ull);
        }
    return got;
}

// Requantize one output of tile row `row` (global row n, token tok) from
// sum(w x): acc = sum(w x) - zx colsum[n], fixed point, saturate, optional
// residual; with O16 to a 16-bit output (no residual).
template <bool O16, class SM>
__device__ __forceinline__ void store_out(const DecProb &p, const SM &sm, int row, int n,
                                          int tok, int32_t sum_wx) {
    // two's-complement wrap is exact: the true value fits in int32
    const int32_t a = (int32_t)((uint32_t)sum_wx - (uint32_t)sm.row_corr[row]);
    if constexpr (O16) {
        reinterpret_cast<int16_t *>(p.y)[(size_t)tok * (size_t)p.ldy + n] =
            (int16_t)mq_requant16((int64_t)a, sm.row_m0[row], sm.row_shift[row], p.zy);
        return;
    }
    int32_t y = mq_requant(a, sm.row_m0[row], sm.row_shift[row], p.zy);
    if (p.residual)
        y = min(127, max(-128, y + (int32_t)p.residual[(size_t)tok * (size_t)p.ldy + n]));
    p.y[(size_t)tok * (size_t)p.ldy + n] = (int8_t)y;
}

// One plane of four 16-bit codes held in two words (codes 2i, 2i+1 in word
// i): the high bytes (plane 0) or the low bytes - 128 (plane 1).
__device__ __forceinline__ uint32_t code_plane(uint32_t w0, uint32_t w1, bool low) {
    return low ? (__byte_perm(w0, w1, 0x6420) ^ 0x80808080u) : __byte_perm(w0, w1, 0x7531);
}

// One stage of one warp: activation fragment and weight words from the ring
// slot, widening, mma.  Returns nothing; accumulates into acc and xs.
template <int BITS, int NT, bool A16>
__device__ __forceinline__ void compute_stage(const uint8_t *ring, int warp, int g, int t,
                                              float (&acc)[4][NT][4], int (&xs)[NT]) {
    using C = Cfg<BITS>;
    // activation fragment of this warp's k range, token g (+8): the bytes at
    // stage offset warp * KWARP + t * KWARP/4 of token row m (zero outside M
    // and K: TMA fill)
    uint32_t xa[NT], xb[NT];
    if constexpr (A16) {
        // 16-bit codes: plane row m is token m >> 1, plane m & 1 (high bytes,
        // low bytes - 128).  Box h of the stage holds 64 codes of the 8
        // tokens (128-byte rows, 128-byte swizzle); this lane's KWARP/4 codes
        // start at stage offset `off`.
        const int off = warp * C::KWARP + t * (C::KWARP / 4);
        const uint8_t *xbox = ring + W_BYTES + (off >> 6) * X16_BOX;
        const int c = (off & 63) >> 3, inner = (off & 7) * 2;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            const int m = nt * 8 + g, tok = m >> 1;
            const uint8_t *src = xbox + tok * 128 + ((c ^ (tok & 7)) << 4) + inner;
            if (BITS == 4) {
                const uint4 v = *reinterpret_cast<const uint4 *>(src);
                xa[nt] = code_plane(v.x, v.y, m & 1);
                xb[nt] = code_plane(v.z, v.w, m & 1);
            } else {
                const uint2 v = *reinterpret_cast<const uint2 *>(src);
                xa[nt] = code_plane(v.x, v.y, m & 1);
                xb[nt] = 0u;
            }
        }
    } else {
        const int off = warp * C::KWARP + t * (C::KWARP / 4);
        const uint8_t *xbox = ring + W_BYTES + (off >> 7) * X_BOX;
        const int c = (off & 127) >> 4, inner = off & 15;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            const int m = nt * 8 + g;
            const uint8_t *src = xbox + m * 128 + ((c ^ (m & 7)) << 4) + inner;
            if (BITS == 4) {
                const uint2 v = *reinterpret_cast<const uint2 *>(src);
                xa[nt] = v.x;
                xb[nt] = v.y;
            } else {
                xa[nt] = lds32(src);
                xb[nt] = 0u;
            }
        }
    }
    // weight word t of chunk `warp` of rows g and g+8 of the four tiles
    uint32_t wv[4][2];
#pragma unroll
    for (int rt = 0; rt < 4; ++rt)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int row = rt * 16 + h * 8 + g;
            wv[rt][h] = lds32(ring + row * ROW_BYTES + ((warp ^ (row & 7)) << 4) + t * 4);
        }
    if constexpr (BITS == 4) {
        // x bytes k0..k7 = xa (k0..k3), xb (k4..k7): pairs (k0,k4) (k2,k6) at
        // scale 1, (k1,k5) (k3,k7) at scale 1/16
        uint32_t b04[NT], b26[NT], b15[NT], b37[NT];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            b04[nt] = x_pair(xa[nt], xb[nt], 0x0040u, false);
            b26[nt] = x_pair(xa[nt], xb[nt], 0x0062u, false);
            b15[nt] = x_pair(xa[nt], xb[nt], 0x0051u, true);
            b37[nt] = x_pair(xa[nt], xb[nt], 0x0073u, true);
            xs[nt] = dp4a_sum(xa[nt], dp4a_sum(xb[nt], xs[nt]));
        }
#pragma unroll
        for (int rt = 0; rt < 4; ++rt) {
            uint32_t pa0[2], pa1[2], pb0[2], pb1[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const uint32_t w = wv[rt][h], w2 = w >> 8;
                pa0[h] = lop3_sel_xor(w, 0x000F000Fu, 0x00080008u);   // u0, u4
                pb0[h] = lop3_sel_xor(w, 0x00F000F0u, 0x00800080u);   // 16 u1, 16 u5
                pa1[h] = lop3_sel_xor(w2, 0x000F000Fu, 0x00080008u);  // u2, u6
                pb1[h] = lop3_sel_xor(w2, 0x00F000F0u, 0x00800080u);  // 16 u3, 16 u7
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                mma16816(acc[rt][nt], pa0[0], pa0[1], pa1[0], pa1[1], b04[nt], b26[nt]);
                mma16816(acc[rt][nt], pb0[0], pb0[1], pb1[0], pb1[1], b15[nt], b37[nt]);
            }
        }
    } else {
        // x bytes k0..k3: pairs (k0,k2), (k1,k3)
        uint32_t b02[NT], b13[NT];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            b02[nt] = x_pair(xa[nt], xa[nt], 0x0020u, false);
            b13[nt] = x_pair(xa[nt], xa[nt], 0x0031u, false);
            xs[nt] = dp4a_sum(xa[nt], xs[nt]);
        }
#pragma unroll
        for (int rt = 0; rt < 4; ++rt) {
            uint32_t pa[2], pb[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const uint32_t w = wv[rt][h];
                pa[h] = lop3_sel_xor(w, 0x00FF00FFu, 0x00800080u);       // u0, u2
                pb[h] = lop3_sel_xor(w >> 8, 0x00FF00FFu, 0x00800080u);  // u1, u3
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
                mma16816(acc[rt][nt], pa[0], pa[1], pb[0], pb[1], b02[nt], b13[nt]);
        }
    }
}

// Exchange buffer of the 16-bit epilogue, laid over the reduction buffer
// (free once every thread has read its slots): the final sums per plane row
// and unit row, row stride 68 words (conflict-free for both the fragment-
// ordered writes and the row-ordered reads).
constexpr int YV_STRIDE = UNIT_ROWS + 4;

// The 16-bit epilogue of one piece.  Every consumer thread calls it (its
// barriers are unconditional); `ok` / `tok` say whether the thread holds
// valid slots.  Sums are formed as in the int8 epilogue (including the split
// unit protocol), then the CTA that finishes the unit writes them to the
// exchange buffer and combines plane rows 2j, 2j + 1 of every unit row:
// sum((x - zx) w) = 256 S(2j) + S(2j + 1) + (128 - zx) colsum, requantized
// to int16.
template <int BITS, int NT, class SM>
__device__ __forceinline__ void a16_epilogue(const Params &P, SM &s, const DecProb &p, int rb,
                                             bool whole, bool ok, int tok, int32_t xsum, int e0,
                                             int ln, bool finisher, int cl, int cta) {
    using C = Cfg<BITS>;
    const int cf = cta;  // read only by the finisher
    bool have = ok && tok < p.M;
    uint32_t v[2 * NT];
    int rows[2 * NT];
#pragma unroll
    for (int q = 0; q < 2 * NT; ++q) {
        const int e = e0 + 8 * q;
        rows[q] = ((e >> 2) / NT) * 16 + (ln >> 2) + ((e & 2) ? 8 : 0);
        int32_t sum = 0;
        if (have) {
#pragma unroll
            for (int w = 0; w < CONS_WARPS; ++w) sum += s.part[w][e][ln];
        }
        // sum(plane (w - zw)) = sum(u plane) - (bias + zw) sum(plane)
        v[q] = (uint32_t)sum - (uint32_t)((C::BIAS + s.row_zw[rows[q]]) * xsum);
    }
    if (have && !whole) {
        if (!finisher) {
            put_partials<NT>(P, cta, v);
            have = false;
        } else {
            uint64_t first[2 * NT];
            read_partials<NT>(P, cf + 1, first);
            have = gather_partials<NT>(P, &s.abort, cf, cl, first, v);
        }
    }
    int32_t *yv = &s.part[0][0][0];
    cons_sync();  // every read of the reduction buffer is done
    if (finisher && have) {
#pragma unroll
        for (int q = 0; q < 2 * NT; ++q) yv[tok * YV_STRIDE + rows[q]] = (int32_t)v[q];
    }
    cons_sync();
    if (finisher && !s.abort) {
        const int ntok = p.M >> 1;
        int16_t *y = reinterpret_cast<int16_t *>(p.y);
        // The codes past K are zero-filled, so each of the unit's n_oob
        // missing k has low plane -128 against a zero weight code: with a
        // weight zero point it adds (0 - zw)(-128) to the low plane's sum,
        // which the combine takes back (per row, like the colsum term).
        const int64_t oob128 = p.K > 0 ? 128 * (int64_t)(p.tiles_m * C::KSTAGE - p.K) : 0;
        for (int i = threadIdx.x; i < UNIT_ROWS * ntok; i += CONS_THREADS) {
            const int row = i & (UNIT_ROWS - 1), j = i / UNIT_ROWS;
            const int n = rb * UNIT_ROWS + row;
            if (n >= p.N) continue;
            const int64_t a = 256 * (int64_t)yv[(2 * j) * YV_STRIDE + row] +
                              (int64_t)yv[(2 * j + 1) * YV_STRIDE + row] +
                              (int64_t)(128 - p.zx) * (int64_t)s.row_corr[row] -
                              oob128 * (int64_t)s.row_zw[row];
            y[(size_t)j * (size_t)p.ldy + n] =
                (int16_t)mq_requant16(a, s.row_m0[row], s.row_shift[row], p.zy);
        }
    }
}

// A16: every problem has 16-bit activations (Problem::a16): x is the plane
// matrix (rows 2m, 2m + 1 = high and low planes of token m) and the outputs
// are int16, formed from row pairs after an exchange through shared memory.
// O16: every problem has 8-bit inputs and a 16-bit output (Problem::o16).
template <int BITS, int NT, bool A16, bool O16>
__global__ void __launch_bounds__(THREADS, 2) decode_kernel(const __grid_constant__ Params P) {
    using C = Cfg<BITS>;
    using SM = Smem<NT>;
    constexpr int STAGES = SM::STAGES;
    extern __shared__ uint8_t smem_raw[];
    SM &s = *reinterpret_cast<SM *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = P.total_stages, G = gridDim.x, cta = blockIdx.x;
    const bool wide = P.wide != 0;
    const int s_begin = range_begin(cta, S, G, wide), s_end = range_begin(cta + 1, S, G, wide);

    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], CONS_WARPS);
        }
        s.abort = 0;
        fence_mbar_init();
    }
    for (int i = threadIdx.x; i < P.count; i += THREADS) s.prob[i] = dec_prob(P.p[i]);
    __syncthreads();
    if (threadIdx.x == 0) griddep_launch_dependents();
    const int count = P.count;

    if (warp == PROD_WARP) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            for (int i = 0; i < P.count; ++i)
                if (P.p[i].K > 0) {
                    prefetch_tensormap(&P.tmap_w[i]);
                    prefetch_tensormap(&P.tmap_x[i]);
                }
            constexpr int XBOXES = C::KSTAGE / 128;  // x boxes per stage (int4: 2, int8: 1)
            // Packed weights are constant inputs (unless a problem says they are
            // written by earlier work, pre_w == 0): the weight boxes of the
            // first ring stages are requested before waiting for the previous
            // grid in the stream; activations only after it.
            const int npre = !P.pre_w ? 0 : s_end - s_begin < STAGES ? s_end - s_begin : STAGES;
            int pi = 0;
            for (int i = 0; i < npre; ++i) {
                const int gs = s_begin + i;
                pi = problem_from(s, count, pi, gs);
                const DecProb &p = s.prob[pi];
                if (p.K == 0) continue;
                const int local = gs - p.tile_begin;
                const int rb = local / p.tiles_m, j = local % p.tiles_m;
                mbar_arrive_expect_tx(&s.full[i], W_BYTES + XBOXES * X_BOX);
                tma_load_2d(s.ring[i], &P.tmap_w[pi], j * ROW_BYTES, rb * UNIT_ROWS, &s.full[i]);
            }
            griddep_wait();
            uint32_t it = 0;
            pi = 0;
            for (int gs = s_begin; gs < s_end; ++gs, ++it) {
                pi = problem_from(s, count, pi, gs);
                const DecProb &p = s.prob[pi];
                const int local = gs - p.tile_begin;
                const int rb = local / p.tiles_m, j = local % p.tiles_m;
                const int slot = it % STAGES;
                if (!mq_wait_parity(&s.empty[slot], ((it / STAGES) & 1) ^ 1, &s.abort, P.status,
                                    P.wait_ns)) {
                    // Given up: let the loads already issued land before the
                    // CTA can leave (stages below `it` were issued whole -- the
                    // waits of the first STAGES stages cannot fail -- and only
                    // the last STAGES of them can still be in flight).
                    for (uint32_t i = it > (uint32_t)STAGES ? it - STAGES : 0u; i < it; ++i)
                        mq_wait_parity_drain(&s.full[i % STAGES], (i / STAGES) & 1, P.status,
                                             P.wait_ns);
                    break;
                }
                if (p.K == 0) {  // an empty stage: nothing to load
                    mbar_arrive(&s.full[slot]);
                    continue;
                }
                if ((int)it >= npre) {
                    mbar_arrive_expect_tx(&s.full[slot], W_BYTES + XBOXES * X_BOX);
                    tma_load_2d(s.ring[slot], &P.tmap_w[pi], j * ROW_BYTES, rb * UNIT_ROWS,
                                &s.full[slot]);
                }
                if constexpr (A16) {
                    // 16-bit codes: KSTAGE / 64 boxes of 8 tokens x 64 codes
                    // (the same bytes as the 8-bit boxes)
#pragma unroll
                    for (int h = 0; h < C::KSTAGE / 64; ++h)
                        tma_load_2d(s.ring[slot] + W_BYTES + h * X16_BOX, &P.tmap_x[pi],
                                    j * C::KSTAGE + h * 64, 0, &s.full[slot]);
                } else {
#pragma unroll
                    for (int h = 0; h < XBOXES; ++h)
                        tma_load_2d(s.ring[slot] + W_BYTES + h * X_BOX, &P.tmap_x[pi],
                                    j * C::KSTAGE + h * 128, 0, &s.full[slot]);
                }
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------ consumers
        griddep_wait();  // before the first global access (parameters, workspace, y)
        const int g = lane >> 2, t = lane & 3;
        uint32_t it = 0;
        bool ok = true;  // after a failed wait the warps still walk the barriers
        int gs = s_begin;
        int pi = 0;
        int par = 0;  // piece parity: selects xsum / last buffers
        while (gs < s_end) {
            // the piece [gs, piece_end) of one unit that this CTA owns
            pi = problem_from(s, count, pi, gs);
            const DecProb &p = s.prob[pi];
            const int nst = p.tiles_m;
            const int local = gs - p.tile_begin;
            const int rb = local / nst;
            const int u_begin = p.tile_begin + rb * nst, u_end = u_begin + nst;
            const int piece_end = u_end < s_end ? u_end : s_end;
            const bool whole = u_begin >= s_begin && u_end <= s_end;
            // this thread's slots j + 256 q share one fragment element i, one
            // token tile and one lane: the token is fixed
            const int e0 = threadIdx.x >> 5, ln = threadIdx.x & 31;
            const int tok = (NT == 2 ? ((e0 >> 2) & 1) * 8 : 0) + 2 * (ln & 3) + (e0 & 1);
            // a split unit is finished by its first CTA (the one holding its
            // first stage), at the end of that CTA's range; the contributors
            // cf + 1 .. cl store their sums at the start of theirs.  The
            // finishing CTA reads the first contributor's entries before its
            // last stage, so that the round trip overlaps that stage.
            const bool finisher = u_begin >= s_begin;
            const int cf = cta;  // read only when finisher
            const int cl = (whole || !finisher) ? cta : cta_of(u_end - 1, S, G, wide);
            const bool early = !A16 && !whole && finisher && tok < p.M;
            uint64_t first[2 * NT];
#pragma unroll
            for (int q = 0; q < 2 * NT; ++q) first[q] = 0;
            // requant parameters of the unit's rows: loaded now, published to
            // shared memory when the piece is done, so the loads overlap the
            // stage loop instead of stalling the warp here
            int32_t prm_cs = 0, prm_m0 = 0, prm_sh = 33, prm_zw = 0;
            if (threadIdx.x < UNIT_ROWS) {
                const int n = rb * UNIT_ROWS + threadIdx.x;
                if (n < p.N) {
                    prm_cs = __ldg(p.colsum + n);
                    prm_m0 = __ldg(p.M0 + n);
                    prm_sh = __ldg(p.shift + n);
                    if (p.zw) prm_zw = __ldg(p.zw + n);
                }
            }
            float acc[4][NT][4];
            int32_t iacc[4][NT][4];
            int xs[NT];
#pragma unroll
            for (int rt = 0; rt < 4; ++rt)
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        acc[rt][nt][i] = 0.f;
                        iacc[rt][nt][i] = 0;
                    }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) xs[nt] = 0;
            for (int q = gs; ok && q < piece_end; ++q, ++it) {
                const int slot = it % STAGES;
                if (early && q == piece_end - 1) read_partials<NT>(P, cf + 1, first);
                bool got = true;
                if (lane == 0)
                    got = mq_wait_parity(&s.full[slot], (it / STAGES) & 1, &s.abort, P.status,
                                         P.wait_ns);
                if (!__shfl_sync(0xffffffffu, got ? 1 : 0, 0)) {
                    ok = false;
                    break;
                }
                if (p.K > 0) compute_stage<BITS, NT, A16>(s.ring[slot], warp, g, t, acc, xs);
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.empty[slot]);
                if constexpr (C::FLUSH) {
                    if ((q - gs + 1) % C::FLUSH_STAGES == 0) {
#pragma unroll
                        for (int rt = 0; rt < 4; ++rt)
#pragma unroll
                            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                                for (int i = 0; i < 4; ++i) {
                                    iacc[rt][nt][i] +=
                                        __float2int_rn(acc[rt][nt][i] * 16777216.0f);
                                    acc[rt][nt][i] = 0.f;
                                }
                    }
                }
            }
            // ---- this CTA's partial of the unit.  Fragment element i of tile
            // (rt, nt) is row rt*16 + g (+8 for i >= 2), token nt*8 + 2t + (i & 1);
            // each warp writes its partials to its own slice, then every
            // thread sums a fixed set of slots over the eight warps.
            if (ok) {
#pragma unroll
                for (int rt = 0; rt < 4; ++rt)
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            int32_t v = __float2int_rn(acc[rt][nt][i] * 16777216.0f);
                            if constexpr (C::FLUSH) v += iacc[rt][nt][i];
                            s.part[warp][(rt * NT + nt) * 4 + i][lane] = v;
                        }
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                    int v = xs[nt];
                    v += __shfl_xor_sync(0xffffffffu, v, 1);
                    v += __shfl_xor_sync(0xffffffffu, v, 2);
                    if (t == 0) s.xpart[warp][nt * 8 + g] = v;
                }
            }
            if (threadIdx.x < UNIT_ROWS) {
                // sum((x - zx)(w - zw)) = sum(x w) - zx colsum - zw sum(x) + K zx zw;
                // the zw sum(x) term is taken per piece with the bias below
                // (16-bit activations: colsum - K zw, the combine applies (128 - zx))
                s.row_corr[threadIdx.x] =
                    A16 ? (int32_t)((uint32_t)prm_cs - (uint32_t)p.K * (uint32_t)prm_zw)
                        : (int32_t)((uint32_t)(p.zx * prm_cs) -
                                    (uint32_t)p.K * (uint32_t)(p.zx * prm_zw));
                s.row_zw[threadIdx.x] = prm_zw;
                s.row_m0[threadIdx.x] = prm_m0;
                s.row_shift[threadIdx.x] = prm_sh;
            }
            cons_sync();
            int32_t xsum = 0;
            if (ok && tok < p.M) {
#pragma unroll
                for (int w = 0; w < CONS_WARPS; ++w) xsum += s.xpart[w][tok];
            }
            if constexpr (A16) {
                a16_epilogue<BITS, NT>(P, s, p, rb, whole, ok, tok, xsum, e0, ln, finisher, cl, cta);
            } else if (ok && whole) {
                // the unit is entirely this CTA's: requantize and store
#pragma unroll
                for (int q = 0; q < 2 * NT; ++q) {
                    const int e = e0 + 8 * q;
                    const int row = ((e >> 2) / NT) * 16 + (ln >> 2) + ((e & 2) ? 8 : 0);
                    const int n = rb * UNIT_ROWS + row;
                    if (tok >= p.M || n >= p.N) continue;
                    int32_t sum = 0;
#pragma unroll
                    for (int w = 0; w < CONS_WARPS; ++w) sum += s.part[w][e][ln];
                    // sum((x - zx)(w - zw)) = sum(u x) - (bias + zw) sum(x) - corr
                    store_out<O16>(p, s, row, n, tok,
                              (int32_t)((uint32_t)sum -
                                        (uint32_t)((C::BIAS + s.row_zw[row]) * xsum)));
                }
            } else if (ok) {
                // a split unit (see above): contributors store, the first CTA
                // gathers, requantizes and stores
                if (tok < p.M) {
                    uint32_t v[2 * NT];
                    int rows[2 * NT];
#pragma unroll
                    for (int q = 0; q < 2 * NT; ++q) {
                        const int e = e0 + 8 * q;
                        rows[q] = ((e >> 2) / NT) * 16 + (ln >> 2) + ((e & 2) ? 8 : 0);
                        int32_t sum = 0;
#pragma unroll
                        for (int w = 0; w < CONS_WARPS; ++w) sum += s.part[w][e][ln];
                        v[q] = (uint32_t)sum - (uint32_t)((C::BIAS + s.row_zw[rows[q]]) * xsum);
                    }
                    if (!finisher) {
                        put_partials<NT>(P, cta, v);
                    } else {
                        if (!early) read_partials<NT>(P, cf + 1, first);
                        if (gather_partials<NT>(P, &s.abort, cf, cl, first, v)) {
#pragma unroll
                            for (int q = 0; q < 2 * NT; ++q) {
                                const int n = rb * UNIT_ROWS + rows[q];
                                if (n < p.N) store_out<O16>(p, s, rows[q], n, tok, (int32_t)v[q]);
                            }
                        }
                    }
                }
            }
            cons_sync();  // every read of part / xpart / row params is done
            par ^= 1;
            gs = piece_end;
        }
    }
    __syncthreads();
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

// uint8 tensor [rows][cols] with row pitch `pitch`, box 128 x box_rows, 128-byte swizzle.
bool encode_sw128(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows,
                  uint64_t pitch, uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {pitch};
    const cuuint32_t box[2] = {ROW_BYTES, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

// int16 tensor [rows][cols] with row pitch `pitch` bytes, box 64 x 8, 128-byte swizzle.
bool encode_x16(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows, uint64_t pitch) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {pitch};
    const cuuint32_t box[2] = {64, 8};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, const_cast<void *>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

// Launch epochs: nonzero and different for consecutive launches (wraps after
// 2^32 - 1 launches; entries are zeroed after use, so an old epoch never
// lingers in the workspace).
uint32_t next_epoch() {
    static std::atomic<uint32_t> counter{0};
    uint32_t e = counter.fetch_add(1, std::memory_order_relaxed) + 1;
    if (e == 0) e = counter.fetch_add(1, std::memory_order_relaxed) + 1;
    return e;
}

// The kernel's dynamic shared-memory limit, raised once per device (the
// attribute belongs to the device's context) and instantiation; safe to call
// from several host threads.
template <int BITS, int NT, bool A16, bool O16>
int prepare_t(int dev) {
    static std::atomic<uint64_t> done{0};  // bit d: device d prepared
    if (dev < 0 || dev >= 64) return MQ_ERR_CUDA;
    const uint64_t bit = 1ull << dev;
    if (done.load(std::memory_order_acquire) & bit) return MQ_OK;
    if (cudaFuncSetAttribute(decode_kernel<BITS, NT, A16, O16>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem_bytes<NT>()) != cudaSuccess)
        return MQ_ERR_CUDA;
    done.fetch_or(bit, std::memory_order_release);
    return MQ_OK;
}

template <int BITS, int NT, bool A16, bool O16>
int launch_t(const Problem *probs, int count, int32_t *workspace, cudaStream_t stream) {
    using C = Cfg<BITS>;
    auto kern = decode_kernel<BITS, NT, A16, O16>;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return MQ_ERR_CUDA;
    if (prepare_t<BITS, NT, A16, O16>(dev) != MQ_OK) return MQ_ERR_CUDA;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MQ_ERR_CUDA;
    for (int begin = 0; begin < count; begin += DECODE_MAX_PROBLEMS) {
        const int n = count - begin < DECODE_MAX_PROBLEMS ? count - begin : DECODE_MAX_PROBLEMS;
        Params P{};
        P.pre_w = 1;
        long long stages = 0;
        for (int i = 0; i < n; ++i) {
            Problem &q = P.p[i];
            q = probs[begin + i];
            if (q.wdynamic) P.pre_w = 0;
            const int nst = q.K > 0 ? (q.K + C::KSTAGE - 1) / C::KSTAGE : 1;
            q.tile_begin = (int)stages;
            q.tiles_m = nst;
            stages += (long long)((q.N + UNIT_ROWS - 1) / UNIT_ROWS) * nst;
            const uint64_t wcols = (uint64_t)q.K * BITS / 8;
            // 16-bit codes: q.M counts plane rows, the tensor has q.M / 2 tokens
            if (q.K > 0 &&
                (!encode_sw128(&P.tmap_w[i], q.w, wcols, (uint64_t)q.N, (uint64_t)q.ldw, UNIT_ROWS) ||
                 !(A16 ? encode_x16(&P.tmap_x[i], q.x, (uint64_t)q.K, (uint64_t)(q.M / 2),
                                    2 * (uint64_t)q.ldx)
                       : encode_sw128(&P.tmap_x[i], q.x, (uint64_t)q.K, (uint64_t)q.M,
                                      (uint64_t)q.ldx, 16))))
                return MQ_ERR_CUDA;
        }
        if (stages == 0) continue;
        if (stages > 0x7fffffffLL) return MQ_ERR_UNSUPPORTED_SHAPE;
        P.count = n;
        P.total_stages = (int)stages;
        P.ws = reinterpret_cast<int2 *>(workspace);
        P.epoch = next_epoch();
        P.status = device_status_ptr();
        P.wait_ns = wait_limit_ns();
        P.skip_cta = test_skip_cta();
        long long grid = 2LL * sms;
        if (grid > DECODE_MAX_GRID) grid = DECODE_MAX_GRID;
        if (grid > stages) grid = stages;
        P.wide = (unsigned long long)stages * (unsigned long long)grid >= (1ull << 32);
        // programmatic stream serialization: this launch may start while the
        // previous kernel in the stream finishes (see griddep_wait)
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)grid, 1, 1);
        cfg.blockDim = dim3(THREADS, 1, 1);
        cfg.dynamicSmemBytes = smem_bytes<NT>();
        cfg.stream = stream;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaLaunchKernelEx(&cfg, kern, P) != cudaSuccess) return MQ_ERR_CUDA;
    }
    return MQ_OK;
}

}  // namespace decode

// Both token-tile variants of the W4A8 decode kernel (8-bit activations and
// output) prepared on the current device.
int prepare_decode_w4a8() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return MQ_ERR_CUDA;
    if (decode::prepare_t<4, 1, false, false>(dev) != MQ_OK ||
        decode::prepare_t<4, 2, false, false>(dev) != MQ_OK)
        return MQ_ERR_CUDA;
    return MQ_OK;
}

// All problems passed here have the same bits, a16 and o16 and M <= DECODE_MAX_M;
// `workspace` holds DECODE_WS_BYTES, zero-filled.
int launch_decode(const Problem *probs, int count, void *workspace, void *stream) {
    using namespace decode;
    if (count <= 0) return MQ_OK;
    // one or two tokens: the row-tile kernel (mq_gemv.cu) when the launch suits it
    const int which = test_decode_kernel();
    if (which != 2) {
        int dev = 0, sms = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            return MQ_ERR_CUDA;
        if (gemv_suits(probs, count, sms, which == 1)) return launch_gemv(probs, count, stream);
    }
    int max_m = 0;
    for (int i = 0; i < count; ++i) max_m = probs[i].M > max_m ? probs[i].M : max_m;
    const bool nt2 = max_m > 8;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int32_t *ws = static_cast<int32_t *>(workspace);
    const bool a16 = probs[0].a16, o16 = probs[0].o16, i4 = probs[0].bits == 4;
#define MQ_DECODE_CASE(A, O)                                                              \
    if (a16 == A && o16 == O) {                                                           \
        if (i4) return nt2 ? launch_t<4, 2, A, O>(probs, count, ws, s)                    \
                           : launch_t<4, 1, A, O>(probs, count, ws, s);                   \
        return nt2 ? launch_t<8, 2, A, O>(probs, count, ws, s)                            \
                   : launch_t<8, 1, A, O>(probs, count, ws, s);                           \
    }
    MQ_DECODE_CASE(true, false)
    MQ_DECODE_CASE(false, true)
    MQ_DECODE_CASE(false, false)
#undef MQ_DECODE_CASE
    return MQ_ERR_INVALID_ARG;
}

}  // namespace mq
