// mq_decode.cu -- weight-streaming kernel for the integer-only quantized
// linear layer at decode sizes (M <= 16 tokens), bit-exact.
//
// At M <= 16 the layer reads each weight once and does at most 16 MACs with
// it, so its speed is the weight stream (the paper notes that autoregressive
// generation is memory-bound, Sec. 5.6 and Appendix A.2).  Each warp streams
// 16-row weight tiles straight from HBM into registers with 128-bit loads,
// widens them in registers to f16 (exact for int8 and int4), and multiplies
// with legacy warp-level mma.sync m16n8k16 (f16 x f16 -> f32): the weights
// are the 16-row A operand, the (zero-padded) tokens the 8-column B operand.
// Register-resident operands keep the weight stream out of shared memory;
// on sm_103a the f16 mma.sync rate is 4x its int8 rate.
//
// Exactness: every product is an integer of magnitude <= 2^14 (int8) or
// 2^10 (int4); a warp converts its f32 accumulators to int32 every 1024
// (int8) or 16384 (int4) values of k, so no f32 partial sum exceeds 2^24.
//
// The reduction order over k inside one mma is free, so the k index of each
// fragment slot is permuted to whatever the cheapest in-register unpacking
// yields (int4: nibble pairs (p, p+4) of a 32-bit word), and the activation
// fragments use the same permutation.
//
// CTA = 8 warps on one 32-row block of one problem; the warps split K
// (step-cyclic) and reduce their int32 partials in shared memory; the
// epilogue subtracts zx * colsum, requantizes (round half up), saturates,
// adds the optional residual and stores int8.
#include <cuda_runtime.h>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {
namespace decode {

constexpr int WARPS = 8;
constexpr int THREADS = WARPS * 32;
constexpr int R = 2;              // 16-row mma tiles per warp (rows per CTA = 16 * R)
constexpr int ROWS = 16 * R;

struct Params {
    Problem p[DECODE_MAX_PROBLEMS];
    int count;
    int total_blocks;
    int *status;
};

__device__ __forceinline__ uint4 ldg16(const void *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

__device__ __forceinline__ uint4 ldg16_keep(const void *p) {
    uint4 v;
    asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Activation int8 words (k0..k3) and (k4..k7) -> f16 pairs (k0,k4) (k1,k5)
// (k2,k6) (k3,k7), matching the int4 weight pairs below.
__device__ __forceinline__ void x8_pairs_int4order(uint32_t a, uint32_t b, uint32_t (&o)[4]) {
    const uint32_t ua = a ^ 0x80808080u, ub = b ^ 0x80808080u;
    const uint32_t u = prmt(ua, ub, 0x5140u);  // a0 b0 a1 b1
    const uint32_t v = prmt(ua, ub, 0x7362u);  // a2 b2 a3 b3
    o[0] = hsub2(prmt(u, 0x64646464u, 0x4140u), F16X2_1152);
    o[1] = hsub2(prmt(u, 0x64646464u, 0x4342u), F16X2_1152);
    o[2] = hsub2(prmt(v, 0x64646464u, 0x4140u), F16X2_1152);
    o[3] = hsub2(prmt(v, 0x64646464u, 0x4342u), F16X2_1152);
}

// int4 word (nibble p = k offset p) -> f16 pairs (k0,k4) (k1,k5) (k2,k6) (k3,k7).
// Pair (p, p+4) sits at bits 4p and 16+4p.  Even p: mantissa = nibble, value
// 1024 + (e + 8), minus 1032.  Odd p: mantissa = 16 * nibble, value
// 1024 + 16 (e + 8), times 1/16 minus 72.
__device__ __forceinline__ void w4_pairs(uint32_t w, uint32_t (&o)[4]) {
    const uint32_t F16X2_1032 = 0x64086408u;
    const uint32_t SCALE16 = 0x2C002C00u;  // (1/16, 1/16)
    const uint32_t OFF72 = 0xD480D480u;    // (-72, -72)
    const uint32_t w2 = w >> 8;
    o[0] = hsub2(lop3_sel_xor(w, 0x000F000Fu, 0x64086408u), F16X2_1032);
    o[1] = hfma2(lop3_sel_xor(w, 0x00F000F0u, 0x64806480u), SCALE16, OFF72);
    o[2] = hsub2(lop3_sel_xor(w2, 0x000F000Fu, 0x64086408u), F16X2_1032);
    o[3] = hfma2(lop3_sel_xor(w2, 0x00F000F0u, 0x64806480u), SCALE16, OFF72);
}

template <int BITS>
struct Cfg;
template <>
struct Cfg<4> {
    static constexpr int KSTEP = 128;       // k per warp step (4 threads x 32)
    static constexpr int KTHREAD = 32;      // k per thread per step
    static constexpr int CHUNK_STEPS = 128; // 16384 k between f32 -> int32 flushes
    static constexpr int MMAS = 8;          // mma k16 per step
};
template <>
struct Cfg<8> {
    static constexpr int KSTEP = 64;
    static constexpr int KTHREAD = 16;
    static constexpr int CHUNK_STEPS = 16;  // 1024 k
    static constexpr int MMAS = 4;
};

template <int BITS, int NT>
struct StepRegs {
    uint4 w[R][2];                     // rows g and g+8 of each 16-row tile
    uint4 x[NT][BITS == 4 ? 2 : 1];    // this thread's k segment of token g (+8)
};

template <int BITS, int NT>
__device__ __forceinline__ void load_step(const Problem &p, int n_base, int step, int g, int t,
                                          StepRegs<BITS, NT> &r) {
    using C = Cfg<BITS>;
    const int k = step * C::KSTEP + t * C::KTHREAD;
    const bool kin = k < p.K;
    const size_t row_bytes = (size_t)p.K * BITS / 8;
    const size_t kbyte = (size_t)k * BITS / 8;
#pragma unroll
    for (int rr = 0; rr < R; ++rr)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int n = n_base + rr * 16 + h * 8 + g;
            r.w[rr][h] = (kin && n < p.N) ? ldg16(p.w + (size_t)n * row_bytes + kbyte)
                                          : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        const int m = nt * 8 + g;
        const bool ok = kin && m < p.M;
        const int8_t *src = p.x + (size_t)m * (size_t)p.ldx + k;
#pragma unroll
        for (int q = 0; q < (BITS == 4 ? 2 : 1); ++q)
            r.x[nt][q] = ok ? ldg16_keep(src + 16 * q) : make_uint4(0, 0, 0, 0);
    }
}

template <int BITS, int NT>
__device__ __forceinline__ void compute_step(const StepRegs<BITS, NT> &r,
                                             float (&acc)[R][NT][4]) {
    if constexpr (BITS == 4) {
        // x: 32 int8 per token = words x0..x7 (k 0..31); word pair (2j, 2j+1)
        // holds k 8j..8j+7.
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            uint32_t xb[NT][4];
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const uint4 &lo = r.x[nt][j >> 1];
                const uint32_t wa = (j & 1) ? lo.z : lo.x;
                const uint32_t wb = (j & 1) ? lo.w : lo.y;
                x8_pairs_int4order(wa, wb, xb[nt]);
            }
#pragma unroll
            for (int rr = 0; rr < R; ++rr) {
                const uint32_t w0 = j == 0 ? r.w[rr][0].x : j == 1 ? r.w[rr][0].y
                                  : j == 2 ? r.w[rr][0].z : r.w[rr][0].w;
                const uint32_t w1 = j == 0 ? r.w[rr][1].x : j == 1 ? r.w[rr][1].y
                                  : j == 2 ? r.w[rr][1].z : r.w[rr][1].w;
                uint32_t pg[4], ph[4];
                w4_pairs(w0, pg);
                w4_pairs(w1, ph);
                const uint32_t a0[4] = {pg[0], ph[0], pg[1], ph[1]};
                const uint32_t a1[4] = {pg[2], ph[2], pg[3], ph[3]};
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                    mma16816(acc[rr][nt], a0, xb[nt][0], xb[nt][1]);
                    mma16816(acc[rr][nt], a1, xb[nt][2], xb[nt][3]);
                }
            }
        }
    } else {
        // int8: word j of the 16-byte segment holds k 4j..4j+3 (natural pairs).
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            uint32_t xb[NT][2];
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const uint4 &v = r.x[nt][0];
                const uint32_t xw = j == 0 ? v.x : j == 1 ? v.y : j == 2 ? v.z : v.w;
                i8x4_to_f16x4(xw, xb[nt][0], xb[nt][1]);
            }
#pragma unroll
            for (int rr = 0; rr < R; ++rr) {
                const uint32_t w0 = j == 0 ? r.w[rr][0].x : j == 1 ? r.w[rr][0].y
                                  : j == 2 ? r.w[rr][0].z : r.w[rr][0].w;
                const uint32_t w1 = j == 0 ? r.w[rr][1].x : j == 1 ? r.w[rr][1].y
                                  : j == 2 ? r.w[rr][1].z : r.w[rr][1].w;
                uint32_t g0, g1, h0, h1;
                i8x4_to_f16x4(w0, g0, g1);
                i8x4_to_f16x4(w1, h0, h1);
                const uint32_t a[4] = {g0, h0, g1, h1};
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) mma16816(acc[rr][nt], a, xb[nt][0], xb[nt][1]);
            }
        }
    }
}

template <int BITS, int NT>
__device__ __forceinline__ void flush(float (&acc)[R][NT][4], int32_t (&iacc)[R][NT][4]) {
#pragma unroll
    for (int rr = 0; rr < R; ++rr)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                iacc[rr][nt][i] += __float2int_rn(acc[rr][nt][i]);
                acc[rr][nt][i] = 0.f;
            }
}

template <int BITS, int NT>
__global__ void __launch_bounds__(THREADS) decode_kernel(const __grid_constant__ Params P) {
    using C = Cfg<BITS>;
    __shared__ int32_t red[ROWS][16];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, t = lane & 3;

    int pi = 0;
    while (pi + 1 < P.count && (int)blockIdx.x >= P.p[pi + 1].tile_begin) ++pi;
    const Problem &p = P.p[pi];
    const int n_base = ((int)blockIdx.x - p.tile_begin) * ROWS;

    for (int i = threadIdx.x; i < ROWS * 16; i += THREADS) (&red[0][0])[i] = 0;
    __syncthreads();

    float acc[R][NT][4];
    int32_t iacc[R][NT][4];
#pragma unroll
    for (int rr = 0; rr < R; ++rr)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                acc[rr][nt][i] = 0.f;
                iacc[rr][nt][i] = 0;
            }

    const int nsteps = (p.K + C::KSTEP - 1) / C::KSTEP;
    StepRegs<BITS, NT> cur, nxt;
    int step = warp;
    if (step < nsteps) load_step<BITS, NT>(p, n_base, step, g, t, nxt);
    int local = 0;
    while (step < nsteps) {
        cur = nxt;
        const int next = step + WARPS;
        if (next < nsteps) load_step<BITS, NT>(p, n_base, next, g, t, nxt);
        compute_step<BITS, NT>(cur, acc);
        if (++local == C::CHUNK_STEPS) {
            flush<BITS, NT>(acc, iacc);
            local = 0;
        }
        step = next;
    }
    flush<BITS, NT>(acc, iacc);

    // cross-warp reduction of the int32 partials: fragment element i of tile
    // (rr, nt) is row rr*16 + g (+8 for i >= 2), token nt*8 + 2t + (i & 1)
#pragma unroll
    for (int rr = 0; rr < R; ++rr)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int row = rr * 16 + g + (i >= 2 ? 8 : 0);
                const int tok = nt * 8 + 2 * t + (i & 1);
                if (tok < p.M) atomicAdd(&red[row][tok], iacc[rr][nt][i]);
            }
    __syncthreads();

    for (int idx = threadIdx.x; idx < ROWS * p.M; idx += THREADS) {
        const int row = idx % ROWS, tok = idx / ROWS;
        const int n = n_base + row;
        if (n >= p.N) continue;
        const int32_t cs = __ldg(p.colsum + n);
        const int32_t m0 = __ldg(p.M0 + n);
        const int32_t sh = __ldg(p.shift + n);
        const int32_t a = (int32_t)((uint32_t)red[row][tok] - (uint32_t)(p.zx * cs));
        const int64_t v = (int64_t)a * (int64_t)m0;
        const int64_t q = (v + ((int64_t)1 << (sh - 1))) >> sh;
        int64_t yv = (int64_t)p.zy + q;
        yv = yv < -128 ? -128 : (yv > 127 ? 127 : yv);
        if (p.residual) {
            yv += (int64_t)p.residual[(size_t)tok * (size_t)p.ldy + n];
            yv = yv < -128 ? -128 : (yv > 127 ? 127 : yv);
        }
        p.y[(size_t)tok * (size_t)p.ldy + n] = (int8_t)yv;
    }
}

template <int BITS, int NT>
int launch_t(const Problem *probs, int count, cudaStream_t stream) {
    for (int begin = 0; begin < count; begin += DECODE_MAX_PROBLEMS) {
        const int n = count - begin < DECODE_MAX_PROBLEMS ? count - begin : DECODE_MAX_PROBLEMS;
        Params P{};
        int blocks = 0;
        for (int i = 0; i < n; ++i) {
            P.p[i] = probs[begin + i];
            P.p[i].tile_begin = blocks;
            blocks += (P.p[i].N + ROWS - 1) / ROWS;
        }
        P.count = n;
        P.total_blocks = blocks;
        P.status = device_status_ptr();
        if (blocks == 0) continue;
        decode_kernel<BITS, NT><<<blocks, THREADS, 0, stream>>>(P);
        if (cudaGetLastError() != cudaSuccess) return MQ_ERR_CUDA;
    }
    return MQ_OK;
}

}  // namespace decode

// All problems passed here have the same bits and M <= DECODE_MAX_M.
int launch_decode(const Problem *probs, int count, void *stream) {
    using namespace decode;
    if (count <= 0) return MQ_OK;
    int max_m = 0;
    for (int i = 0; i < count; ++i) max_m = probs[i].M > max_m ? probs[i].M : max_m;
    const bool nt2 = max_m > 8;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (probs[0].bits == 4)
        return nt2 ? launch_t<4, 2>(probs, count, s) : launch_t<4, 1>(probs, count, s);
    return nt2 ? launch_t<8, 2>(probs, count, s) : launch_t<8, 1>(probs, count, s);
}

}  // namespace mq
