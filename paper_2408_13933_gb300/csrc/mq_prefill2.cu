// mq_prefill2.cu -- tensor-core kernel for the integer-only quantized linear
// layer at prefill sizes with 256-token pair tiles, bit-exact, and the token
// pre-pass it reads.
//
// Same arithmetic as mq_prefill.cu (Sec. 3.1: int8 x int8 products summed in
// int32, then the zero-point correction and the fixed-point requant of the
// layer's output): the operands are widened to f16, which holds every int8
// and int4 value exactly, the pair MMAs (tcgen05 cta_group::2, kind::f16)
// sum the exact products in f32, and the f32 sums are integers that are
// exact while no partial sum exceeds 2^24 in magnitude.
//
// What differs is the tile and where the widening happens:
//   * A pair tile is 256 output channels x 256 tokens (MMA M = 256, N = 256):
//     each stage of weights widened into tensor memory feeds twice the MMA
//     work of a 128-token tile, and the L2 -> SM bytes per MMA drop by a
//     third.
//   * The tokens are widened once per call, by the pre-pass below, into an
//     f16 copy in the caller's workspace, which TMA loads straight into the
//     MMA's 128-byte-swizzled operand layout.  Only the weights pass through
//     the converter warps.
//   * The pre-pass also writes every token row's sum of squares X2[m].  By
//     Cauchy-Schwarz, every partial sum over a run of L k's satisfies
//     |sum x w| <= sqrt(X2[m]) * wmax * sqrt(L), where wmax bounds |w - zw|
//     (128 for int8, 255 with a zero point, 8 and 15 for int4).  A tile whose
//     rows all satisfy X2 * wmax^2 * L <= 2^48 can therefore accumulate a
//     run of L k's in one f32 chunk.  Each tile takes the longer of that run
//     and the data-independent one (1024 k for int8 and so on); activations
//     quantized from real data give one chunk for the whole K.
//   * The f32 accumulator F (256 columns) is single: at the end of a chunk
//     each epilogue thread loads its 64 sums 32 at a time, requantizes and
//     packs them four tokens a word, and releases F, so the MMAs of the next
//     tile wait only for that; the stores follow from the packed words (a
//     4 x 4 byte transpose across lanes gives 4-byte stores of four channels).
//     A tile with several chunks adds the earlier chunks' int32 sums through
//     local memory.
//
// Data path per CTA and stage of 128 k:
//   weights: HBM/L2 --TMA--> int8 / int4 staging ring (S8 stages)
//            --converters--> A: TMEM ring (SF stages of 64 columns)
//   tokens:  f16 copy --TMA--> B: shared-memory ring (SF stages, 128 rows x
//            128 k, two 64-k swizzle atoms)
//   pair MMA (issued by the even CTA) --> F: TMEM columns 0-255
// TMEM columns: F 0-255, A stages 256 + 64 s.
// Warp roles (both CTAs), warpgroup-aligned for setmaxnreg:
//   warp 0      : weight TMA producer (one lane)
//   warp 1      : TMEM allocation; in the even CTA the MMA loop (converged
//                 warp, one elected lane issues)
//   warp 2      : token TMA producer (one lane)
//   warp 3      : idle
//   warps 4-11  : converters, two groups of four on alternate stages: warp w
//                 widens TMEM lanes 32 (w % 4) .. +31 (its weight rows, all
//                 128 k of the stage)
//   warps 12-27 : epilogue: thread = one output channel (TMEM lane) x 64 of
//                 the tile's 256 tokens
// All mbarrier waits are bounded (mq_wait_parity / mq_wait_parity_cluster).
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <queue>
#include <vector>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {

// cuTensorMapEncodeTiled through the runtime's driver entry point (defined in
// mq_prefill.cu).
namespace prefill {
PFN_cuTensorMapEncodeTiled_v12000 encode_fn();
bool encode_2d(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows, uint64_t pitch,
               uint32_t box_cols, uint32_t box_rows);
}  // namespace prefill

namespace prefill2 {

constexpr int TM = 256;  // output channels per pair tile (MMA M, operand A)
constexpr int TN = 256;  // tokens per pair tile (MMA N, operand B)
constexpr int CM = 128;  // weight rows per CTA
constexpr int CN = 128;  // token rows per CTA
constexpr int KS = 128;  // k per stage
constexpr int S8 = 5;    // weight staging stages
constexpr int SF = 4;    // operand stages (A in TMEM, B in shared memory)
constexpr int WPROD_WARP = 0;
constexpr int MMA_WARP = 1;
constexpr int XPROD_WARP = 2;
constexpr int CONV_WARP0 = 4;
constexpr int CONV_WARPS = 8;
constexpr int EPI_WARP0 = 12;
constexpr int EPI_WARPS = 16;
constexpr int TPT = TN / (EPI_WARPS / 4);  // tokens per epilogue thread
constexpr int NUM_WARPS = 28;
constexpr int THREADS = NUM_WARPS * 32;
constexpr int STA = CM * KS;       // weight staging bytes (int4 uses half)
constexpr int XATOM = CN * 128;    // one 64-k swizzle atom of the f16 token tile
constexpr int OPB = 2 * XATOM;     // f16 token tile of one stage
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t A_COL0 = 256;   // A stage s at A_COL0 + 64 s; F at 0
// Register split after set-up (setmaxnreg, per warpgroup): control warps,
// converters, epilogue.  The launch gives every thread LAUNCH_REGS, and
// setmaxnreg.inc draws only on what the CTA's warps give back with
// setmaxnreg.dec: the split must fit THREADS * LAUNCH_REGS, or the epilogue
// warps would wait for registers forever.  The launcher checks the compiled
// kernel's register count against it before every first launch on a device.
constexpr int LAUNCH_REGS = 72;
constexpr int REG_CTRL = 24;
constexpr int REG_CONV = 64;
constexpr int REG_EPI = 88;
constexpr int REG_SPLIT = 128 * REG_CTRL + 32 * CONV_WARPS * REG_CONV + 32 * EPI_WARPS * REG_EPI;
static_assert(THREADS * LAUNCH_REGS <= 65536, "launch register budget");
static_assert(REG_SPLIT <= THREADS * LAUNCH_REGS, "register split above the launch allocation");
constexpr int MAX_SCHED = 4096;
constexpr int MAX_PAIRS = 128;

struct Params {
    CUtensorMap tmap_w[PREFILL_MAX_PROBLEMS];  // int8 [N][K] box 128 B x 128, or int4 64 B x 128
    CUtensorMap tmap_x[PREFILL_MAX_PROBLEMS];  // f16 [M][K] box 64 x 128 (128-byte swizzle)
    Problem p[PREFILL_MAX_PROBLEMS];           // tile_begin: first tile; tiles_m: token tiles
    const int32_t *rowsq[PREFILL_MAX_PROBLEMS];  // sum of squares of every token row
    uint16_t *y16[PREFILL_MAX_PROBLEMS];         // or null: y also written as f16 [M][N]
    int32_t *ysq[PREFILL_MAX_PROBLEMS];          // with y16: row sums of squares of y, added
    int count;
    int total_tiles;
    int npairs;
    int use_table;
    int pre_w;  // 1: load weights before griddep_wait (all constant)
    uint16_t pair_begin[MAX_PAIRS + 1];
    uint16_t sched[MAX_SCHED];
    uint8_t sched_pi[MAX_SCHED];
    int *status;
    uint64_t wait_ns;
};

struct Smem {
    uint8_t opb[SF][OPB];  // first: every atom 1024-byte aligned
    uint8_t sta[S8][STA];
    uint64_t ld_full[S8];
    uint64_t ld_empty[S8];
    uint64_t b_full[SF];    // this CTA's token tile landed (TMA transaction bytes)
    uint64_t op_full[SF];   // even CTA: its converter warps arrive (one announcing 16
                            // bytes), the odd CTA's converter warps signal 4 bytes each
    uint64_t op_empty[SF];  // both CTAs: multicast commit
    uint64_t f_full;        // both CTAs: multicast commit
    uint64_t f_empty;       // even CTA: both CTAs' epilogue warps arrive
    uint64_t done;
    uint32_t sink[CONV_WARPS];
    uint32_t tmem_base;
    int abort;
};

constexpr size_t SMEM_BYTES = sizeof(Smem) + 1024;

struct Tile {
    int pi;
    int ct, tt;  // channel tile, token tile
    int nkb;     // stages
};

__device__ __forceinline__ int problem_of(const Params &P, int tile) {
    int lo = 0, hi = P.count - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (P.p[mid].tile_begin <= tile)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

__device__ __forceinline__ Tile tile_of(const Params &P, int tile, int pi) {
    Tile t;
    t.pi = pi;
    const Problem &p = P.p[pi];
    const int local = tile - p.tile_begin;
    t.tt = local % p.tiles_m;
    t.ct = local / p.tiles_m;
    t.nkb = (p.K + KS - 1) / KS;
    return t;
}

__device__ __forceinline__ bool pair_tile_at(const Params &P, int pair, int i, Tile &t) {
    if (P.use_table) {
        const int j = P.pair_begin[pair] + i;
        if (j >= P.pair_begin[pair + 1]) return false;
        t = tile_of(P, P.sched[j], P.sched_pi[j]);
        return true;
    }
    const int tile = pair + i * P.npairs;
    if (tile >= P.total_tiles) return false;
    t = tile_of(P, tile, problem_of(P, tile));
    return true;
}

// Stages per exact f32 chunk of a tile (warp-collective; the MMA warp and the
// epilogue warps compute the same value).  The data-independent chunk bounds
// |x (w - zw)| by 128 wmax per product; the data-dependent one uses the
// tile's largest token-row sum of squares X2: a run of L k's is exact when
// X2 wmax^2 L <= 2^48 (every partial sum is then at most 2^24 in magnitude),
// or, given the weights' sums of squares (symmetric weights), the whole K
// when X2 max_n wsq[n] <= 2^48.
__device__ __forceinline__ int chunk_stages(const Params &P, const Tile &t, int lane) {
    const Problem &p = P.p[t.pi];
    const bool zw = p.zw != nullptr;
    const int fixed = p.bits == 8 ? (zw ? 512 / KS : 1024 / KS) : (zw ? 8192 / KS : 16384 / KS);
    const int32_t *rq = P.rowsq[t.pi];
    const int m0 = t.tt * TN;
    uint32_t mx = 0;
    for (int i = lane; i < TN; i += 32)
        if (m0 + i < p.M) mx = max(mx, (uint32_t)__ldg(rq + m0 + i));
    mx = __reduce_max_sync(0xffffffffu, mx);
    if (p.wsq && !zw) {
        // both operands' norms: every partial sum over any part of K is at most
        // sqrt(X2 W2), so X2 W2 <= 2^48 sums the whole K in one run
        const int n0 = t.ct * TM;
        uint32_t wm = 0;
        for (int i = lane; i < TM; i += 32)
            if (n0 + i < p.N) wm = max(wm, (uint32_t)__ldg(p.wsq + n0 + i));
        wm = __reduce_max_sync(0xffffffffu, wm);
        if ((uint64_t)mx * (uint64_t)wm <= (1ull << 48)) return t.nkb < 1 ? 1 : t.nkb;
    }
    const uint64_t wmax = p.bits == 8 ? (zw ? 255u : 128u) : (zw ? 15u : 8u);
    const uint64_t per_stage = (uint64_t)mx * wmax * wmax * (uint64_t)KS;  // < 2^54
    uint64_t data = per_stage ? (1ull << 48) / per_stage : (uint64_t)t.nkb;
    if (data > (uint64_t)t.nkb) data = (uint64_t)t.nkb;
    const int L = max((int)data, fixed);
    return L < 1 ? 1 : L;
}

__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, Smem &s,
                                          const Params &P) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0) ok = mq_wait_parity(bar, parity, &s.abort, P.status, P.wait_ns);
    return __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
}

__device__ __forceinline__ void abort_pair(Smem &s, uint32_t rank) {
    s.abort = 1;
    asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(cluster_addr(&s.abort, rank ^ 1u)),
                 "r"(1u) : "memory");
}

__device__ __forceinline__ uint4 lds16(const uint8_t *p) {
    return *reinterpret_cast<const uint4 *>(p);
}

template <uint32_t N>
__device__ __forceinline__ void reg_dec() {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}
template <uint32_t N>
__device__ __forceinline__ void reg_inc() {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}

// Four int32 values saturated to int8 and packed, value i in byte i.
__device__ __forceinline__ uint32_t pack4_sat_s8(int32_t v0, int32_t v1, int32_t v2, int32_t v3) {
    uint32_t hi, d;
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(hi) : "r"(v3), "r"(v2), "r"(0u));
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(v1), "r"(v0), "r"(hi));
    return d;
}

// Requantize 32 sums of one channel (32 consecutive tokens) and pack them,
// four tokens a word, into w[0..7].  FAST: the shift is at least 33, so the
// round-half-up shift is a multiply-high, an add and a shift; the saturation
// to int8 happens in the pack.
template <bool FAST>
__device__ __forceinline__ void requant_pack32(const uint32_t (&f)[32], int32_t corr, int32_t m0,
                                               int32_t sh, int32_t zy, uint32_t *w) {
    const int32_t rnd = FAST ? (1 << (sh - 33)) : 0;
    const int32_t rs = FAST ? sh - 32 : 0;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        int32_t o[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int32_t a = (int32_t)(f[4 * q + i] - (uint32_t)corr);
            o[i] = FAST ? ((__mulhi(a, m0) + rnd) >> rs) + zy : mq_requant(a, m0, sh, zy);
        }
        w[q] = pack4_sat_s8(o[0], o[1], o[2], o[3]);
    }
}

// Store the packed outputs of this warp's 32 channels x TPT tokens four bytes
// at a time: a 4 x 4 byte transpose among the four lanes of a group (two
// shuffles) leaves lane r of the group with token 4q + r of the group's four
// consecutive channels, stored (the residual added bytewise, saturating) as
// one 32-bit word.  The whole warp calls it (the shuffles); `nch` (0..4) is
// the number of the group's channels below N; y0 / r0 point at token tok0 and
// the group's first channel, and both, like ldy, are 4-byte aligned.
// With y16 (chained layers): the same words also go out as f16 (8 bytes: four
// channels of one token; y16 and ysq point at token tok0 and the group's
// first channel / at token tok0, row pitch ldy16 elements), and each token's
// sum of squares over the warp's 32 channels is added into ysq (dp4a over
// the group's four channels, shuffles over the eight groups).
template <bool CHAIN>
__device__ __forceinline__ void store_words_v4(const uint32_t (&w)[TPT / 4], int8_t *y0,
                                               const int8_t *r0, size_t ldy, int ntok, int lane,
                                               int nch, uint16_t *y16, int32_t *ysq,
                                               size_t ldy16) {
    const int r = lane & 3;
    const uint32_t sel1 = (r & 1) ? 0x3715u : 0x6240u;
    const uint32_t sel2 = (r & 2) ? 0x3276u : 0x5410u;
    // the bytes of this lane's group that are channels below N
    const uint32_t valid = nch >= 4 ? 0xFFFFFFFFu : (nch <= 0 ? 0u : (1u << (8 * nch)) - 1u);
#pragma unroll
    for (int q = 0; q < TPT / 4; ++q) {
        if (4 * q >= ntok) break;
        uint32_t v = prmt(w[q], __shfl_xor_sync(0xffffffffu, w[q], 1), sel1);
        v = prmt(v, __shfl_xor_sync(0xffffffffu, v, 2), sel2);
        const int tok = 4 * q + r;
        const bool live = tok < ntok && nch > 0;
        if (live && r0) {
            const int8_t *rp = r0 + (size_t)tok * ldy;
            uint32_t res = 0;
            if (nch == 4) {
                res = *reinterpret_cast<const uint32_t *>(rp);
            } else {
                for (int c = 0; c < nch; ++c) res |= (uint32_t)(uint8_t)rp[c] << (8 * c);
            }
            v = __vaddss4(v, res);
        }
        if (live) {
            int8_t *yp = y0 + (size_t)tok * ldy;
            if (nch == 4) {
                *reinterpret_cast<uint32_t *>(yp) = v;
            } else {
                for (int c = 0; c < nch; ++c) yp[c] = (int8_t)(v >> (8 * c));
            }
        }
        if (CHAIN && y16) {
            const uint32_t vm = live ? v & valid : 0u;
            if (live && nch == 4) {  // N % 16 == 0: a group is whole or past N
                uint32_t h0, h1;
                i8x4_to_f16x4(vm, h0, h1);
                *reinterpret_cast<uint2 *>(y16 + (size_t)tok * ldy16) = make_uint2(h0, h1);
            }
            int sq = __dp4a((int)vm, (int)vm, 0);
            sq += __shfl_xor_sync(0xffffffffu, sq, 4);
            sq += __shfl_xor_sync(0xffffffffu, sq, 8);
            sq += __shfl_xor_sync(0xffffffffu, sq, 16);
            if (lane < 4 && tok < ntok) atomicAdd(ysq + tok, sq);
        }
    }
}

// The same outputs one byte at a time (y, the residual or ldy not 4-byte
// aligned): this lane's channel, tokens tok0 .. tok0 + ntok - 1.
__device__ __forceinline__ void store_words_b(const uint32_t (&w)[TPT / 4], int8_t *yp,
                                              const int8_t *rp, size_t ldy, int ntok) {
#pragma unroll
    for (int q = 0; q < TPT / 4; ++q) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int tok = 4 * q + i;
            if (tok < ntok) {
                int32_t out = (int32_t)(int8_t)(w[q] >> (8 * i));
                if (rp) out = min(127, max(-128, out + (int32_t)rp[(size_t)tok * ldy]));
                yp[(size_t)tok * ldy] = (int8_t)out;
            }
        }
    }
}

// ZW: problems may have a weight zero point, folded into the widening of the
// weights (w - zw); without it the widening offsets are immediate constants.
// CHAIN: some problem's output also goes out as f16 with its row sums of
// squares (a separate instantiation: the extra epilogue code slowed launches
// that do not use it by ~5%).
template <bool ZW, bool CHAIN>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
    prefill2_kernel(const __grid_constant__ Params P) {
    extern __shared__ uint8_t smem_raw[];
    Smem &s = *reinterpret_cast<Smem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();  // 0: even CTA (issues the MMAs), 1: odd
    const int pair = (int)(blockIdx.x >> 1);

    if (threadIdx.x == 0) {
        for (int i = 0; i < S8; ++i) {
            mbar_init(&s.ld_full[i], 1);
            mbar_init(&s.ld_empty[i], CONV_WARPS / 2);
        }
        for (int i = 0; i < SF; ++i) {
            mbar_init(&s.b_full[i], 1);
            mbar_init(&s.op_full[i], CONV_WARPS / 2);
            mbar_init(&s.op_empty[i], 1);
        }
        mbar_init(&s.f_full, 1);
        mbar_init(&s.f_empty, 2 * EPI_WARPS);
        mbar_init(&s.done, 32);  // one commit from every lane of the MMA warp
        s.abort = 0;
        fence_mbar_init();
    }
    if (warp == MMA_WARP) {
        tmem_alloc2(&s.tmem_base, TMEM_COLS);
        tmem_relinquish2();
    }
    tc_fence_before();
    cluster_sync();  // barriers of both CTAs initialised before any remote arrive
    tc_fence_after();
    if (threadIdx.x == 0) griddep_launch_dependents();
    const uint32_t tmem = s.tmem_base;

    if (warp < CONV_WARP0) {
        reg_dec<REG_CTRL>();
        if (warp == WPROD_WARP) {
            // ------------------------------------------------ weight TMA producer
            if (lane == 0) {
                for (int i = 0; i < P.count; ++i)
                    if (P.p[i].K > 0) prefetch_tensormap(&P.tmap_w[i]);
                // packed weights are constant inputs (unless a problem says they
                // are written by earlier work, pre_w == 0): the first S8 stages
                // are requested before waiting for the previous grid
                uint32_t npre = 0;
                if (P.pre_w) {
                    Tile t;
                    for (int ti = 0; npre < (uint32_t)S8 && pair_tile_at(P, pair, ti, t); ++ti) {
                        const bool i4 = P.p[t.pi].bits == 4;
                        const int wrow = t.ct * TM + (int)rank * CM;
                        for (int kb = 0; kb < t.nkb && npre < (uint32_t)S8; ++kb, ++npre) {
                            mbar_arrive_expect_tx(&s.ld_full[npre], i4 ? STA / 2 : STA);
                            tma_load_2d(s.sta[npre], &P.tmap_w[t.pi], i4 ? kb * (KS / 2) : kb * KS,
                                        wrow, &s.ld_full[npre]);
                        }
                    }
                }
                griddep_wait();
                uint32_t it = 0;
                bool ok = true;
                Tile t;
                for (int ti = 0; ok && pair_tile_at(P, pair, ti, t); ++ti) {
                    const bool i4 = P.p[t.pi].bits == 4;
                    const int wrow = t.ct * TM + (int)rank * CM;
                    for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                        if (it < npre) continue;
                        const int slot = it % S8;
                        if (!mq_wait_parity(&s.ld_empty[slot], ((it / S8) & 1) ^ 1, &s.abort,
                                            P.status, P.wait_ns)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(&s.ld_full[slot], i4 ? STA / 2 : STA);
                        tma_load_2d(s.sta[slot], &P.tmap_w[t.pi], i4 ? kb * (KS / 2) : kb * KS,
                                    wrow, &s.ld_full[slot]);
                    }
                }
                if (!ok) {
                    // let the loads already issued land before this CTA can leave
                    abort_pair(s, rank);
                    for (uint32_t i = it > (uint32_t)S8 ? it - S8 : 0u; i < it; ++i)
                        mq_wait_parity_drain(&s.ld_full[i % S8], (i / S8) & 1, P.status,
                                             P.wait_ns);
                }
            }
            __syncwarp();
        } else if (warp == XPROD_WARP) {
            // ------------------------------------------------- token TMA producer
            if (lane == 0) {
                for (int i = 0; i < P.count; ++i)
                    if (P.p[i].K > 0) prefetch_tensormap(&P.tmap_x[i]);
                griddep_wait();  // the f16 tokens are written by the pre-pass
                uint32_t it = 0;
                bool ok = true;
                Tile t;
                for (int ti = 0; ok && pair_tile_at(P, pair, ti, t); ++ti) {
                    const int xrow = t.tt * TN + (int)rank * CN;
                    for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                        const int sf = it % SF;
                        // the MMAs that read slot sf last have completed
                        if (!mq_wait_parity(&s.op_empty[sf], ((it / SF) & 1) ^ 1, &s.abort,
                                            P.status, P.wait_ns)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(&s.b_full[sf], OPB);
                        tma_load_2d(s.opb[sf], &P.tmap_x[t.pi], kb * KS, xrow, &s.b_full[sf]);
                        tma_load_2d(s.opb[sf] + XATOM, &P.tmap_x[t.pi], kb * KS + KS / 2, xrow,
                                    &s.b_full[sf]);
                    }
                }
                if (!ok) {
                    abort_pair(s, rank);
                    for (uint32_t i = it > (uint32_t)SF ? it - SF : 0u; i < it; ++i)
                        mq_wait_parity_drain(&s.b_full[i % SF], (i / SF) & 1, P.status,
                                             P.wait_ns);
                }
            }
            __syncwarp();
        } else if (warp == MMA_WARP) {
            // ------------------------------------------------------- MMA issuer
            // The whole warp runs the loop (warp-uniform control flow) and one
            // elected lane issues the MMAs and commits.
            if (rank == 0) {
                griddep_wait();  // the chunk plan reads the pre-pass's row sums
                const uint32_t idesc = idesc_f16_f32(TM, TN);
                uint32_t it = 0, chunks = 0;
                bool ok = true;
                Tile t;
                for (int ti = 0; ok && pair_tile_at(P, pair, ti, t); ++ti) {
                    const int L = t.nkb ? chunk_stages(P, t, lane) : 1;
                    int kc = 0;  // stage within the exact-f32 chunk
                    for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                        const bool chunk_start = kc == 0;
                        if (chunk_start &&
                            !warp_wait(&s.f_empty, (chunks & 1) ^ 1, s, P)) {  // F copied out
                            ok = false;
                            break;
                        }
                        const int slot = it % SF;
                        if (!warp_wait(&s.op_full[slot], (it / SF) & 1, s, P)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t acol = tmem + A_COL0 + 64 * slot;
                        const uint64_t bd0 = smem_desc_sw128(smem_u32(s.opb[slot]));
                        const uint64_t bd1 = smem_desc_sw128(smem_u32(s.opb[slot] + XATOM));
                        const bool chunk_end = ++kc == L || kb + 1 == t.nkb;
                        if (elect_one()) {
#pragma unroll
                            for (int j = 0; j < KS / 16; ++j)  // +32 B along K: +2 in the (addr >> 4) field
                                tc_mma2_f16_ts(tmem, acol + 8 * j,
                                               (j < 4 ? bd0 : bd1) + 2 * (j & 3), idesc,
                                               (chunk_start && j == 0) ? 0u : 1u);
                            tc_commit2_mc(&s.op_empty[slot], 3);
                            if (chunk_end) tc_commit2_mc(&s.f_full, 3);
                        }
                        __syncwarp();
                        if (chunk_end) {
                            ++chunks;
                            kc = 0;
                        }
                    }
                }
                if (!ok && lane == 0) abort_pair(s, rank);
                // every MMA issued above has completed once `done` fires (every
                // lane commits, so the phase follows whichever lane issued)
                tc_commit2_mc(&s.done, 1);
                if (lane == 0) mq_wait_parity_drain(&s.done, 0, P.status, P.wait_ns);
            }
            __syncwarp();
        }
    } else if (warp < EPI_WARP0) {
        reg_dec<REG_CONV>();
        // ------------------------------------------------------------ converters
        // Two groups of four warps take alternate stages; in its stage warp w
        // widens all 128 k of weight rows 32 (w % 4) .. +31 into TMEM.
        const int grp = (warp - CONV_WARP0) >> 2;            // 0 or 1
        const int gt = threadIdx.x - (CONV_WARP0 + 4 * grp) * 32;  // 0..127 in the group
        const int quad = warp & 3;
        const int arow = quad * 32 + lane;
        const uint32_t a_lane = tmem + ((uint32_t)(quad * 32) << 16);
        uint32_t a8_src[8], a4_src[4];
#pragma unroll
        for (int i = 0; i < 8; ++i) a8_src[i] = (uint32_t)(arow * 128 + ((i ^ (arow & 7)) << 4));
#pragma unroll
        for (int i = 0; i < 4; ++i)
            a4_src[i] = (uint32_t)(arow * 64 + ((i ^ ((arow >> 1) & 3)) << 4));
        if constexpr (ZW) griddep_wait();  // the weight zero points are read below
        const uint32_t leader_op_full = cluster_addr(&s.op_full[0], 0);
        const uint32_t leader_sink = cluster_addr(&s.sink[warp - CONV_WARP0], 0);
        uint32_t it = 0;
        bool ok = true;
        Tile t;
        for (int ti = 0; ok && pair_tile_at(P, pair, ti, t); ++ti) {
            const bool i4 = P.p[t.pi].bits == 4;
            uint32_t aoff = i4 ? 0xD480E408u : F16X2_1152;
            if constexpr (ZW) {
                const int32_t *zwp = P.p[t.pi].zw;
                const int wch = t.ct * TM + (int)rank * CM + arow;
                const int32_t zwr = (zwp && wch < P.p[t.pi].N) ? __ldg(zwp + wch) : 0;
                aoff = i4 ? f16x2_i4_offset(zwr) : f16x2_i8_offset(zwr);
            }
            for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                if ((int)(it & 1) != grp) continue;
                const int s8 = it % S8, sf = it % SF;
                if (!warp_wait(&s.ld_full[s8], (it / S8) & 1, s, P) ||
                    !warp_wait(&s.op_empty[sf], ((it / SF) & 1) ^ 1, s, P)) {
                    if (lane == 0) abort_pair(s, rank);
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint8_t *sa = s.sta[s8];
                const uint32_t acol = a_lane + A_COL0 + 64 * sf;
#pragma unroll
                for (int hk = 0; hk < 2; ++hk) {  // 64 k of the row per TMEM store
                    uint32_t a[32];
                    if (!i4) {
                        uint4 v[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i) v[i] = lds16(sa + a8_src[4 * hk + i]);
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            i8x4_to_f16x4(v[i].x, a[8 * i + 0], a[8 * i + 1], aoff);
                            i8x4_to_f16x4(v[i].y, a[8 * i + 2], a[8 * i + 3], aoff);
                            i8x4_to_f16x4(v[i].z, a[8 * i + 4], a[8 * i + 5], aoff);
                            i8x4_to_f16x4(v[i].w, a[8 * i + 6], a[8 * i + 7], aoff);
                        }
                    } else {
                        uint4 v[2];
#pragma unroll
                        for (int i = 0; i < 2; ++i) v[i] = lds16(sa + a4_src[2 * hk + i]);
#pragma unroll
                        for (int i = 0; i < 2; ++i) {
                            const uint32_t w4[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                uint32_t o[4];
                                i4x8_to_f16x8(w4[j], o, aoff);
#pragma unroll
                                for (int e = 0; e < 4; ++e) a[16 * i + 4 * j + e] = o[e];
                            }
                        }
                    }
                    tc_st_32x32b_x32(acol + 32 * hk, a);
                }
                // every value read from the staging slot now feeds an issued store
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.ld_empty[s8]);
                // the MMA also reads this CTA's token tile: one warp of the group
                // holds its signal back until the tile has landed
                if (quad == 0 && !warp_wait(&s.b_full[sf], (it / SF) & 1, s, P)) {
                    if (lane == 0) abort_pair(s, rank);
                    ok = false;
                    break;
                }
                tc_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    if (rank == 0 && gt == 0)  // also announces the odd CTA's signal bytes
                        mbar_arrive_expect_tx(&s.op_full[sf], 4 * (CONV_WARPS / 2));
                    else if (rank == 0)
                        mbar_arrive(&s.op_full[sf]);
                    else
                        st_async_signal(leader_sink, it, leader_op_full + 8u * (uint32_t)sf);
                }
            }
        }
    } else {
        reg_inc<REG_EPI>();
        // -------------------------------------------------------------- epilogue
        griddep_wait();  // before the first global access (row sums, parameters, y)
        const int quad = warp & 3;
        const int part_of = (warp - EPI_WARP0) >> 2;  // which TPT tokens of the tile
        const uint32_t t_lane = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(TPT * part_of);
        const uint32_t leader_f_empty = cluster_addr(&s.f_empty, 0);
        uint32_t chunks = 0;
        bool ok = true;
        Tile t;
        for (int ti = 0; ok && pair_tile_at(P, pair, ti, t); ++ti) {
            const Problem &p = P.p[t.pi];
            const int ch = t.ct * TM + (int)rank * CM + quad * 32 + lane;
            const bool ch_in = ch < p.N;
            const int32_t zw = (ch_in && p.zw) ? __ldg(p.zw + ch) : 0;
            // the chunks sum x (w - zw): sum((x - zx)(w - zw)) = that - zx (colsum - K zw)
            const int32_t corr =
                ch_in ? (int32_t)((uint32_t)(p.zx * __ldg(p.colsum + ch)) -
                                  (uint32_t)p.K * (uint32_t)(p.zx * zw))
                      : 0;
            const int32_t m0 = ch_in ? __ldg(p.M0 + ch) : 0;
            const int32_t sh = ch_in ? __ldg(p.shift + ch) : 33;
            const int L = t.nkb ? chunk_stages(P, t, lane) : 1;
            const int nchunks = t.nkb ? (t.nkb + L - 1) / L : 0;
            const bool fast = __all_sync(0xffffffffu, sh >= 33);
            uint32_t w[TPT / 4];  // requantized outputs, four tokens a word
            // int32 sums of the chunks before the last (rare: several chunks
            // only when some token row is far above anything quantized from
            // real data)
            volatile uint32_t part[TPT];
            for (int c = 0; c < nchunks; ++c, ++chunks) {
                if (!warp_wait(&s.f_full, chunks & 1, s, P)) {
                    if (lane == 0) abort_pair(s, rank);
                    ok = false;
                    break;
                }
                tc_fence_after();
                const bool last = c + 1 == nchunks;
                uint32_t f[TPT];
#pragma unroll
                for (int q = 0; q < TPT / 32; ++q)
                    tc_ld_32x32b_x32(t_lane + 32 * q, *reinterpret_cast<uint32_t(*)[32]>(&f[32 * q]));
                tc_wait_ld();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(leader_f_empty);  // F may be overwritten
#pragma unroll
                for (int i = 0; i < TPT; ++i) {
                    uint32_t v = (uint32_t)__float2int_rn(__uint_as_float(f[i]));
                    if (nchunks > 1) {
                        if (c > 0) v += part[i];
                        if (!last) part[i] = v;
                    }
                    f[i] = v;
                }
                if (last) {
#pragma unroll
                    for (int q = 0; q < TPT / 32; ++q) {
                        const uint32_t(&g)[32] = *reinterpret_cast<const uint32_t(*)[32]>(&f[32 * q]);
                        if (fast)
                            requant_pack32<true>(g, corr, m0, sh, p.zy, &w[8 * q]);
                        else
                            requant_pack32<false>(g, corr, m0, sh, p.zy, &w[8 * q]);
                    }
                }
            }
            if (!ok) break;
            if (nchunks == 0) {  // K = 0: every sum is 0
                uint32_t f[32];
#pragma unroll
                for (int i = 0; i < 32; ++i) f[i] = 0u;
#pragma unroll
                for (int q = 0; q < TPT / 32; ++q) {
                    if (fast)
                        requant_pack32<true>(f, corr, m0, sh, p.zy, &w[8 * q]);
                    else
                        requant_pack32<false>(f, corr, m0, sh, p.zy, &w[8 * q]);
                }
            }
            const int tok0 = t.tt * TN + TPT * part_of;
            const int ntok = min(TPT, p.M - tok0);
            if (ntok <= 0) continue;
            const size_t ldy = (size_t)p.ldy;
            const bool vec = ((ldy | reinterpret_cast<uintptr_t>(p.y) |
                               reinterpret_cast<uintptr_t>(p.residual)) & 3) == 0;
            if (vec) {  // the whole warp: the stores are transposed across lanes
                const int chg = ch - (lane & 3);  // first channel of this lane's group
                const int nch = max(0, min(4, p.N - chg));
                int8_t *y0 = p.y + (size_t)tok0 * ldy + chg;
                const int8_t *r0 = p.residual ? p.residual + (size_t)tok0 * ldy + chg : nullptr;
                uint16_t *y16 = CHAIN ? P.y16[t.pi] : nullptr;
                int32_t *ysq = y16 ? P.ysq[t.pi] + tok0 : nullptr;
                if (y16) y16 += (size_t)tok0 * (size_t)p.N + chg;
                store_words_v4<CHAIN>(w, y0, r0, ldy, ntok, lane, nch, y16, ysq, (size_t)p.N);
            } else if (ch_in) {
                int8_t *yp = p.y + (size_t)tok0 * ldy + ch;
                const int8_t *rp = p.residual ? p.residual + (size_t)tok0 * ldy + ch : nullptr;
                store_words_b(w, yp, rp, ldy, ntok);
            }
        }
    }

    tc_fence_before();
    cluster_sync();  // the pair's MMAs are done with both CTAs' TMEM and shared memory
    if (warp == MMA_WARP) {
        tc_fence_after();
        tmem_dealloc2(tmem, TMEM_COLS);
    }
}

// ---------------------------------------------------------------- pre-pass
// One CTA per token row: the f16 copy of the row (pitch K) and its sum of
// squares.  K is a multiple of 16 and every row 16-byte aligned.
struct WidenParams {
    Widen16Job job[WIDEN16_MAX_JOBS];
    int row_begin[WIDEN16_MAX_JOBS + 1];  // first global row of each job
    int count;
};

__global__ void __launch_bounds__(256) widen16_kernel(const __grid_constant__ WidenParams P) {
    __shared__ int part[8];
    griddep_launch_dependents();
    griddep_wait();  // x may be written by the previous kernel in the stream
    const int row = (int)blockIdx.x;
    int j = 0;
    while (row >= P.row_begin[j + 1]) ++j;
    const Widen16Job &J = P.job[j];
    const int m = row - P.row_begin[j];
    const int8_t *src = J.x + (size_t)m * (size_t)J.ldx;
    uint16_t *dst = J.out + (size_t)m * (size_t)J.K;
    int sq = 0;
    for (int k = 16 * (int)threadIdx.x; k < J.K; k += 16 * 256) {
        const uint4 v = *reinterpret_cast<const uint4 *>(src + k);
        uint32_t h[8];
        i8x4_to_f16x4(v.x, h[0], h[1]);
        i8x4_to_f16x4(v.y, h[2], h[3]);
        i8x4_to_f16x4(v.z, h[4], h[5]);
        i8x4_to_f16x4(v.w, h[6], h[7]);
        uint4 *o = reinterpret_cast<uint4 *>(dst + k);
        o[0] = make_uint4(h[0], h[1], h[2], h[3]);
        o[1] = make_uint4(h[4], h[5], h[6], h[7]);
        sq = __dp4a((int)v.x, (int)v.x, sq);
        sq = __dp4a((int)v.y, (int)v.y, sq);
        sq = __dp4a((int)v.z, (int)v.z, sq);
        sq = __dp4a((int)v.w, (int)v.w, sq);
    }
    sq = __reduce_add_sync(0xffffffffu, sq);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = sq;
    __syncthreads();
    if (threadIdx.x == 0) {
        int t = 0;
#pragma unroll
        for (int w = 0; w < 8; ++w) t += part[w];
        J.rowsq[m] = t;
    }
}

// One warp per weight row: wsq[n] = sum_k w[n][k]^2 of the codes (int4: both
// nibbles of a byte, sign-extended per byte).
__global__ void __launch_bounds__(256) wsq_kernel(const uint8_t *w, int N, int K, int bits, int ldw,
                                                  int32_t *wsq) {
    const int n = (int)blockIdx.x * 8 + (int)(threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (n >= N) return;
    const uint8_t *row = w + (size_t)n * (size_t)ldw;
    const int bytes = K * bits / 8;
    int sq = 0;
    for (int b = 16 * lane; b < bytes; b += 512) {
        const uint4 v = *reinterpret_cast<const uint4 *>(row + b);
        const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            if (bits == 8) {
                sq = __dp4a((int)u[i], (int)u[i], sq);
            } else {
                // nibble -> signed byte: ((x ^ 8) - 8) per byte
                const int lo = (int)__vsub4((u[i] & 0x0F0F0F0Fu) ^ 0x08080808u, 0x08080808u);
                const int hi = (int)__vsub4(((u[i] >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u, 0x08080808u);
                sq = __dp4a(lo, lo, sq);
                sq = __dp4a(hi, hi, sq);
            }
        }
    }
    sq = __reduce_add_sync(0xffffffffu, sq);
    if (lane == 0) wsq[n] = sq;
}

// Pairs the device can run at once (one CTA per SM, clusters of two).
int max_pairs(int dev) {
    static int cached[64] = {0};
    if (dev >= 0 && dev < 64 && cached[dev]) return cached[dev];
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    int n = sms / 2;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(2 * n, 1, 1);
    cfg.blockDim = dim3(THREADS, 1, 1);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, prefill2_kernel<false, false>, &cfg) == cudaSuccess &&
        clusters > 0 && clusters < n)
        n = clusters;
    if (n > MAX_PAIRS) n = MAX_PAIRS;
    if (dev >= 0 && dev < 64) cached[dev] = n;
    return n;
}

void lpt_schedule(Params &P, int npairs) {
    std::vector<std::pair<int, int>> work;  // (work, tile)
    std::vector<uint8_t> tile_pi(P.total_tiles);
    work.reserve(P.total_tiles);
    for (int pi = 0; pi < P.count; ++pi) {
        const Problem &q = P.p[pi];
        const int tiles = q.tiles_m * ((q.N + TM - 1) / TM);
        const int w = (q.K + KS - 1) / KS + 2;
        for (int i = 0; i < tiles; ++i) {
            work.emplace_back(w, q.tile_begin + i);
            tile_pi[q.tile_begin + i] = (uint8_t)pi;
        }
    }
    std::stable_sort(work.begin(), work.end(),
                     [](const std::pair<int, int> &a, const std::pair<int, int> &b) {
                         return a.first > b.first;
                     });
    using Load = std::pair<long long, int>;  // (load, pair)
    std::priority_queue<Load, std::vector<Load>, std::greater<Load>> heap;
    for (int i = 0; i < npairs; ++i) heap.emplace(0LL, i);
    std::vector<std::vector<int>> lists(npairs);
    for (const auto &wt : work) {
        Load l = heap.top();
        heap.pop();
        lists[l.second].push_back(wt.second);
        l.first += wt.first;
        heap.push(l);
    }
    int at = 0;
    for (int i = 0; i < npairs; ++i) {
        P.pair_begin[i] = (uint16_t)at;
        for (int tile : lists[i]) {
            P.sched_pi[at] = tile_pi[tile];
            P.sched[at++] = (uint16_t)tile;
        }
    }
    P.pair_begin[npairs] = (uint16_t)at;
}

// f16 [rows][cols] tensor map, box 64 x 128 elements, 128-byte swizzle.
bool encode_x16(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows) {
    auto fn = prefill::encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)CN};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(base), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace prefill2

int launch_weight_sq(const uint8_t *packed, int N, int K, int bits, int ldw, int32_t *wsq,
                     void *stream) {
    if (N <= 0) return MQ_OK;
    prefill2::wsq_kernel<<<(unsigned)((N + 7) / 8), 256, 0, static_cast<cudaStream_t>(stream)>>>(
        packed, N, K, bits, ldw, wsq);
    return cudaGetLastError() == cudaSuccess ? MQ_OK : MQ_ERR_CUDA;
}

int launch_widen16(const Widen16Job *jobs, int count, void *stream) {
    using namespace prefill2;
    for (int begin = 0; begin < count; begin += WIDEN16_MAX_JOBS) {
        const int n = count - begin < WIDEN16_MAX_JOBS ? count - begin : WIDEN16_MAX_JOBS;
        WidenParams P{};
        long long rows = 0;
        for (int i = 0; i < n; ++i) {
            P.job[i] = jobs[begin + i];
            P.row_begin[i] = (int)rows;
            rows += jobs[begin + i].M;
        }
        if (rows == 0) continue;
        if (rows > 0x7fffffffLL) return MQ_ERR_UNSUPPORTED_SHAPE;
        P.row_begin[n] = (int)rows;
        P.count = n;
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)rows, 1, 1);
        cfg.blockDim = dim3(256, 1, 1);
        cfg.stream = static_cast<cudaStream_t>(stream);
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaLaunchKernelEx(&cfg, widen16_kernel, P) != cudaSuccess) return MQ_ERR_CUDA;
    }
    return MQ_OK;
}

bool prefill2_ready() {
    using namespace prefill2;
    static std::atomic<uint64_t> attr_done{0};  // bit d: device d prepared
    static std::atomic<uint64_t> refused{0};    // bit d: device d cannot run the kernel
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
    if (refused.load(std::memory_order_acquire) & (1ull << dev)) return false;
    if (!(attr_done.load(std::memory_order_acquire) & (1ull << dev))) {
        const int smem = (int)SMEM_BYTES;
        const auto attr = cudaFuncAttributeMaxDynamicSharedMemorySize;
        bool ok = cudaFuncSetAttribute(prefill2_kernel<false, false>, attr, smem) == cudaSuccess &&
                  cudaFuncSetAttribute(prefill2_kernel<true, false>, attr, smem) == cudaSuccess &&
                  cudaFuncSetAttribute(prefill2_kernel<false, true>, attr, smem) == cudaSuccess &&
                  cudaFuncSetAttribute(prefill2_kernel<true, true>, attr, smem) == cudaSuccess;
        // the register split of the warpgroups must fit what the launch gives
        // the CTA (see REG_SPLIT): a build that compiled to fewer registers per
        // thread is never launched (the 128-token kernel serves instead)
        for (const void *k :
             {(const void *)prefill2_kernel<false, false>, (const void *)prefill2_kernel<true, false>,
              (const void *)prefill2_kernel<false, true>, (const void *)prefill2_kernel<true, true>}) {
            cudaFuncAttributes fa{};
            ok = ok && cudaFuncGetAttributes(&fa, k) == cudaSuccess &&
                 fa.numRegs * THREADS >= REG_SPLIT;
        }
        if (!ok) {
            cudaGetLastError();  // clear a failed attribute call's error state
            refused.fetch_or(1ull << dev, std::memory_order_release);
            return false;
        }
        attr_done.fetch_or(1ull << dev, std::memory_order_release);
    }
    return true;
}

int launch_prefill2(const Problem *probs, const uint16_t *const *x16, const int32_t *const *rowsq,
                    uint16_t *const *y16, int32_t *const *ysq, int count, void *stream) {
    using namespace prefill2;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return MQ_ERR_CUDA;
    if (!prefill2_ready()) return MQ_ERR_CUDA;
    if (count <= 0) return MQ_OK;
    const int pairs_max = max_pairs(dev);
    if (pairs_max < 1) return MQ_ERR_CUDA;
    for (int begin = 0; begin < count; begin += PREFILL_MAX_PROBLEMS) {
        const int n = count - begin < PREFILL_MAX_PROBLEMS ? count - begin : PREFILL_MAX_PROBLEMS;
        bool any_zw = false, any_chain = false;
        for (int i = begin; i < begin + n; ++i) {
            any_zw = any_zw || probs[i].zw != nullptr;
            any_chain = any_chain || (y16 && y16[i]);
        }
        auto kern = any_zw ? (any_chain ? prefill2_kernel<true, true> : prefill2_kernel<true, false>)
                           : (any_chain ? prefill2_kernel<false, true> : prefill2_kernel<false, false>);
        Params P{};
        P.pre_w = 1;
        long long tiles = 0;
        int order[PREFILL_MAX_PROBLEMS];
        for (int i = 0; i < n; ++i) order[i] = begin + i;
        for (int i = 1; i < n; ++i)
            for (int j = i; j > 0 && probs[order[j]].K > probs[order[j - 1]].K; --j) {
                const int tmp = order[j];
                order[j] = order[j - 1];
                order[j - 1] = tmp;
            }
        for (int i = 0; i < n; ++i) {
            Problem &q = P.p[i];
            q = probs[order[i]];
            P.rowsq[i] = rowsq[order[i]];
            P.y16[i] = y16 ? y16[order[i]] : nullptr;
            P.ysq[i] = y16 ? ysq[order[i]] : nullptr;
            if (q.wdynamic) P.pre_w = 0;
            q.tiles_m = (q.M + TN - 1) / TN;
            q.tile_begin = (int)tiles;
            tiles += (long long)q.tiles_m * ((q.N + TM - 1) / TM);
            if (q.K > 0) {
                const bool i4 = q.bits == 4;
                const uint64_t wcols = i4 ? (uint64_t)q.K / 2 : (uint64_t)q.K;
                if (!encode_x16(&P.tmap_x[i], x16[order[i]], (uint64_t)q.K, (uint64_t)q.M) ||
                    !prefill::encode_2d(&P.tmap_w[i], q.w, wcols, (uint64_t)q.N, (uint64_t)q.ldw,
                                        i4 ? KS / 2 : KS, CM))
                    return MQ_ERR_CUDA;
            }
        }
        if (tiles == 0) continue;
        if (tiles > 0x7fffffffLL) return MQ_ERR_UNSUPPORTED_SHAPE;
        P.count = n;
        P.total_tiles = (int)tiles;
        P.status = device_status_ptr();
        P.wait_ns = wait_limit_ns();
        P.npairs = tiles < pairs_max ? (int)tiles : pairs_max;
        P.use_table = tiles <= MAX_SCHED ? 1 : 0;
        if (P.use_table) lpt_schedule(P, P.npairs);
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)(2 * P.npairs), 1, 1);
        cfg.blockDim = dim3(THREADS, 1, 1);
        cfg.dynamicSmemBytes = SMEM_BYTES;
        cfg.stream = static_cast<cudaStream_t>(stream);
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaLaunchKernelEx(&cfg, kern, P) != cudaSuccess) return MQ_ERR_CUDA;
    }
    return MQ_OK;
}

}  // namespace mq
