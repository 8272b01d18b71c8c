// mq_prefill.cu -- tensor-core kernel for the integer-only quantized linear
// layer at prefill sizes (M > 16): y = requant(sum_k (x - zx) w), bit-exact.
//
// The contraction (Sec. 3.1: int8 x int8 operations with int32 accumulation)
// runs on sm_103a's 5th-generation tensor cores.  sm_103a has no integer MMA
// kind (ptxas rejects tcgen05.mma .kind::i8 for this target), so the operands
// are widened to f16, which represents every int8 and int4 value exactly; the
// products are then exact and an f32 accumulator stays exact while every
// partial sum is an integer of magnitude <= 2^24.  The K loop is therefore cut
// into chunks of 1024 (int8 weights: |x w| <= 2^14) or 16384 (int4: |x w| <=
// 2^10); after each chunk the epilogue converts the f32 chunk sum to int32
// and adds it to an int32 running sum.  With a weight zero point zw the
// converters widen w - zw instead (the widening's f16 offset absorbs zw), the
// chunks shrink to 512 and 8192 (|x (w - zw)| <= 128 * 255, 128 * 15) and the
// epilogue subtracts zx (colsum - K zw).
//
// The kernel runs on CTA pairs (clusters of two, one CTA per SM) with pair
// MMAs (tcgen05 cta_group::2, M = 256, N = 128, K = 16).  Operand A is the
// weights: 256 output channels per pair tile, 128 in each CTA, widened by the
// converter warps straight into tensor memory (tcgen05.st), so they never pass
// through shared memory as f16.  Operand B is the activations: 128 tokens per
// pair tile, 64 rows in each CTA's shared memory, 128-byte swizzled K-major.
// Shared-memory bandwidth is what the tensor cores' operand reads and the
// widening pass compete for; this split keeps the f16 traffic through shared
// memory to the 64 token rows per CTA.
//
// Data path, per CTA and stage of 128 k:
//   HBM/L2 --TMA--> int8 / int4 staging ring (S8 stages, zero fill outside
//   the tensors) --converters--> A: TMEM ring (SF stages), B: f16 ring in
//   shared memory (SF stages) --pair MMA, issued by the even CTA--> f32 chunk
//   accumulator F[b] in TMEM (two buffers, so the MMAs of chunk c+1 overlap
//   the drain of chunk c).
// TMEM columns: F[0] 0-127, F[1] 128-255, A stages 256 + 64 s.
// Warp roles (both CTAs):
//   warp 0     : TMA producer (one thread) for this CTA's weight and token rows.
//   warp 1     : TMEM allocation; in the even CTA the warp runs the MMA loop
//                and one elected lane issues the MMAs and the commits
//                (multicast to both CTAs' barriers).
//   warps 2-9  : converters, two groups of four taking alternate stages.  In
//                its stage warp w writes TMEM lanes 32 (w % 4) .. +31 (its
//                weight rows, all 128 k) and widens four 16-byte chunks of
//                the token tile into shared memory.
//   warps 10-17: epilogue.  Thread = one output channel (TMEM lane), 64 of
//                the tile's 128 tokens; the int32 sum of each chunk is kept
//                in registers; per tile: acc - zx*colsum[n], fixed-point
//                requant, saturate, optional residual, byte stores (one warp
//                writes 32 consecutive channels of a token row).
// Work: pair tiles (256 channels x 128 tokens) of up to PREFILL_MAX_PROBLEMS
// independent linears, assigned to pairs by the host (longest processing time
// first) or round-robin when there are too many tiles for the table.
// 16-bit activations (the A16 instantiation): x is the plane matrix, whose
// rows 2m and 2m + 1 hold the high bytes and the low bytes - 128 of token m,
// so a tile covers 64 tokens; the epilogue adds 256 times the first column of
// each pair and the second into an int64 sum per token and chunk, adds
// (128 - zx) colsum and stores the int16 result.
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
namespace prefill {

constexpr int TM = 256;  // output channels per pair tile (MMA M, operand A)
constexpr int TN = 128;  // tokens per pair tile (MMA N, operand B)
constexpr int CM = 128;  // weight rows per CTA
constexpr int CN = 64;   // token rows per CTA
constexpr int KS = 128;  // k per stage
constexpr int S8 = 6;    // staging stages
constexpr int SF = 4;    // operand stages (A in TMEM, B in shared memory)
constexpr int TMA_WARP = 0;
constexpr int MMA_WARP = 1;
constexpr int CONV_WARP0 = 2;
constexpr int CONV_WARPS = 8;
constexpr int EPI_WARP0 = 10;
constexpr int EPI_WARPS = 8;
constexpr int NUM_WARPS = 18;
constexpr int THREADS = NUM_WARPS * 32;
constexpr int STA = CM * KS;       // weight staging bytes (int4 uses half)
constexpr int STB = CN * KS;       // token staging bytes
constexpr int ATOM = CN * 128;     // one 64-k column of the f16 token tile
constexpr int OPB = 2 * ATOM;      // f16 token tile of one stage
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t F_COL0 = 0;     // F[b] at F_COL0 + 128 b
constexpr uint32_t A_COL0 = 256;   // A stage s at A_COL0 + 64 s
constexpr int KB_PER_CHUNK_I8 = 1024 / KS;   // |partial| <= 1024 * 2^14 = 2^24
constexpr int KB_PER_CHUNK_I4 = 16384 / KS;  // |partial| <= 16384 * 2^10 = 2^24
// with a weight zero point the widened weights are w - zw: |x (w - zw)| <=
// 128 * 255 (int8) or 128 * 15 (int4)
constexpr int KB_PER_CHUNK_I8Z = 512 / KS;   // |partial| <= 512 * 32640 < 2^24
constexpr int KB_PER_CHUNK_I4Z = 8192 / KS;  // |partial| <= 8192 * 1920 < 2^24
constexpr int MAX_SCHED = 4096;    // tile table entries (host LPT schedule)
constexpr int MAX_PAIRS = 128;

struct Params {
    CUtensorMap tmap_w[PREFILL_MAX_PROBLEMS];  // int8 [N][K] box 128 B x 128, or int4 bytes box 64 B x 128
    CUtensorMap tmap_x[PREFILL_MAX_PROBLEMS];  // int8 [M][ldx] box 128 x 64
    Problem p[PREFILL_MAX_PROBLEMS];           // tile_begin: first tile; tiles_m: token tiles
    int count;
    int total_tiles;
    int npairs;
    int use_table;                       // 1: sched / pair_begin, 0: round-robin
    int pre_w;                           // 1: load weights before griddep_wait (all constant)
    uint16_t pair_begin[MAX_PAIRS + 1];
    uint16_t sched[MAX_SCHED];
    uint8_t sched_pi[MAX_SCHED];  // the problem of each table entry
    int *status;
    uint64_t wait_ns;                    // limit of every bounded wait
};

struct Smem {
    uint8_t sta[S8][STA];
    uint8_t stb[S8][STB];
    uint8_t opb[SF][OPB];
    uint64_t ld_full[S8];
    uint64_t ld_empty[S8];
    uint64_t op_full[SF];   // even CTA: its converter warps arrive (one announcing 16
                            // bytes), the odd CTA's converter warps signal 4 bytes each
    uint64_t op_empty[SF];  // both CTAs: multicast commit
    uint64_t f_full[2];     // both CTAs: multicast commit
    uint64_t f_empty[2];    // even CTA: both CTAs' epilogue warps arrive
    uint64_t done;
    uint32_t sink[CONV_WARPS];  // even CTA: targets of the odd CTA's st.async signals
    uint32_t tmem_base;
    int abort;
};

constexpr size_t SMEM_BYTES = sizeof(Smem) + 1024;  // + alignment slack

struct Tile {
    int pi;
    int ct, tt;    // channel tile, token tile
    int nkb, kpc;  // stages, stages per exact f32 chunk
};

// The last problem whose first tile is <= tile (binary search: the problem
// table lives in the kernel parameters, whose reads are slow).
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
    const Problem &p = P.p[t.pi];
    const int local = tile - p.tile_begin;
    t.tt = local % p.tiles_m;
    t.ct = local / p.tiles_m;
    t.nkb = (p.K + KS - 1) / KS;
    t.kpc = p.bits == 8 ? (p.zw ? KB_PER_CHUNK_I8Z : KB_PER_CHUNK_I8)
                        : (p.zw ? KB_PER_CHUNK_I4Z : KB_PER_CHUNK_I4);
    return t;
}

// The i-th tile of pair `pair`, or -1 past its last one.
// The i-th tile of pair `pair` (false past its last one).  The table gives
// each entry's problem; round-robin tiles search for it.
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

// Warp-uniform bounded waits: lane 0 polls, the verdict is broadcast.
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, Smem &s,
                                          const Params &P) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0) ok = mq_wait_parity(bar, parity, &s.abort, P.status, P.wait_ns);
    return __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
}

// After a failed wait: raise the other CTA's abort word too, so that the pair
// gives up together instead of the peer waiting out its own limit.  The peer
// is still running: neither CTA leaves before the final cluster barrier, and
// this store is ordered before this thread's arrival there.
__device__ __forceinline__ void abort_pair(Smem &s, uint32_t rank) {
    s.abort = 1;
    asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(cluster_addr(&s.abort, rank ^ 1u)),
                 "r"(1u) : "memory");
}


__device__ __forceinline__ uint4 lds16(const uint8_t *p) {
    return *reinterpret_cast<const uint4 *>(p);
}

__device__ __forceinline__ void sts16(uint8_t *p, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
    *reinterpret_cast<uint4 *>(p) = make_uint4(a, b, c, d);
}

// What the epilogue needs of a tile's problem, copied into registers (the
// problem table lives in the kernel parameters, where dynamically indexed
// reads are slow).
struct EpiArgs {
    int8_t *y;
    const int8_t *residual;
    int M, ldy, zy;
};

// Requantize and store this thread's 64 outputs (one channel, 64 tokens
// `ldy` bytes apart), with the residual added when RES.  The shift is the
// thread's own (one channel), so its requant case is decided once; FULL
// tiles skip the per-token bound.  The residual bytes of 16 tokens are all
// loaded before their first store (the compiler cannot know that y and the
// residual do not alias), so each group of 16 costs one round trip.
template <bool RES, bool FULL, bool FAST>
__device__ __forceinline__ void store_channel(const uint32_t (&acc)[64], int32_t corr, int32_t m0,
                                              int32_t sh, int32_t zy, int8_t *yp,
                                              const int8_t *rp, size_t ldy, int ntok) {
    // FAST: shift >= 33, (mulhi + 2^(s-33)) >> (s-32); other shifts: mq_requant
    const int32_t rnd = FAST ? (1 << (sh - 33)) : 0;
    const int32_t rs = FAST ? sh - 32 : 0;
#pragma unroll
    for (int q4 = 0; q4 < 4; ++q4) {
        uint32_t res[4] = {0u, 0u, 0u, 0u};  // 4 bytes each
        if (RES) {
            const int8_t *r = rp;
#pragma unroll
            for (int i = 0; i < 16; ++i, r += ldy)
                if (FULL || 16 * q4 + i < ntok) res[i >> 2] |= (uint32_t)(uint8_t)*r << (8 * (i & 3));
            rp = r;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i, yp += ldy) {
            const int j = 16 * q4 + i;
            if (FULL || j < ntok) {
                const int32_t a = (int32_t)(acc[j] - (uint32_t)corr);
                int32_t out = FAST ? min(127, max(-128, ((__mulhi(a, m0) + rnd) >> rs) + zy))
                                   : mq_requant(a, m0, sh, zy);
                if (RES) {
                    const int32_t r = (int32_t)(int8_t)(res[i >> 2] >> (8 * (i & 3)));
                    out = min(127, max(-128, out + r));
                }
                *yp = (int8_t)out;
            }
        }
    }
}

// The 16-bit output of 8-bit inputs: the same 64 outputs requantized to int16
// (no residual).  The accumulator fits int32, so for shifts >= 33 the int8
// path's multiply-high form gives floor((acc M0 + 2^(sh-1)) / 2^sh) exactly
// (|q| <= 2^30, so q + zy cannot overflow); other shifts take mq_requant16.
template <bool FULL, bool FAST>
__device__ __forceinline__ void store_channel16(const uint32_t (&acc)[64], int32_t corr,
                                                int32_t m0, int32_t sh, int32_t zy, int16_t *yp,
                                                size_t ldy, int ntok) {
    const int32_t rnd = FAST ? (1 << (sh - 33)) : 0;
    const int32_t rs = FAST ? sh - 32 : 0;
#pragma unroll
    for (int j = 0; j < 64; ++j, yp += ldy)
        if (FULL || j < ntok) {
            const int32_t a = (int32_t)(acc[j] - (uint32_t)corr);
            *yp = (int16_t)(FAST ? min(32767, max(-32768, ((__mulhi(a, m0) + rnd) >> rs) + zy))
                                 : mq_requant16((int64_t)a, m0, sh, zy));
        }
}

// Barrier scopes: arrivals from the other CTA are releases at cluster scope
// (st.async complete_tx, mbarrier.arrive.release.cluster, multicast commits),
// so the data they publish is visible cluster-wide before the phase can
// complete; waiters acquire at CTA scope, which is far cheaper per wait.
// A16: every problem has 16-bit activations (Problem::a16): its x is the
// plane matrix, and the epilogue combines row pairs and stores int16.
// O16: every problem has 8-bit inputs and a 16-bit output (Problem::o16).
// ZW: problems may have a weight zero point, folded into the widening of the
// weights (w - zw); without it the widening offsets are immediate constants
// (a register offset in the converters' loop costs about 4% on symmetric
// blocks).
template <bool A16, bool O16, bool ZW>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
    prefill_kernel(const __grid_constant__ Params P) {
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
            mbar_init(&s.op_full[i], CONV_WARPS / 2);
            mbar_init(&s.op_empty[i], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&s.f_full[b], 1);
            mbar_init(&s.f_empty[b], 2 * EPI_WARPS);
        }
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

    if (warp == TMA_WARP) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            for (int i = 0; i < P.count; ++i) {
                if (P.p[i].K == 0) continue;  // no map was encoded
                prefetch_tensormap(&P.tmap_x[i]);
                prefetch_tensormap(&P.tmap_w[i]);
            }
            // Packed weights are constant inputs (unless a problem says they are
            // written by earlier work, pre_w == 0): the weight boxes of the first
            // S8 stages are requested before waiting for the previous grid in
            // the stream; activations only after it.
            uint32_t npre = 0;
            if (P.pre_w) {
                Tile t;
                for (int ti = 0; npre < (uint32_t)S8 && pair_tile_at(P, pair, ti, t); ++ti) {
                    const bool i4 = P.p[t.pi].bits == 4;
                    const int wrow = t.ct * TM + (int)rank * CM;
                    for (int kb = 0; kb < t.nkb && npre < (uint32_t)S8; ++kb, ++npre) {
                        mbar_arrive_expect_tx(&s.ld_full[npre], (i4 ? STA / 2 : STA) + STB);
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
                const uint32_t bytes = (i4 ? STA / 2 : STA) + STB;
                const int wrow = t.ct * TM + (int)rank * CM;
                const int xrow = t.tt * TN + (int)rank * CN;
                for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                    const int slot = it % S8;
                    if (!mq_wait_parity(&s.ld_empty[slot], ((it / S8) & 1) ^ 1, &s.abort,
                                        P.status, P.wait_ns)) {
                        ok = false;
                        break;
                    }
                    if (it >= npre) {
                        mbar_arrive_expect_tx(&s.ld_full[slot], bytes);
                        tma_load_2d(s.sta[slot], &P.tmap_w[t.pi], i4 ? kb * (KS / 2) : kb * KS,
                                    wrow, &s.ld_full[slot]);
                    }
                    tma_load_2d(s.stb[slot], &P.tmap_x[t.pi], kb * KS, xrow, &s.ld_full[slot]);
                }
            }
            if (!ok) {
                // Given up: let the loads already issued land before this CTA
                // can leave (stages below `it` were issued whole -- the waits
                // of the first S8 stages cannot fail -- and only the last S8
                // of them can still be in flight).
                abort_pair(s, rank);
                for (uint32_t i = it > (uint32_t)S8 ? it - S8 : 0u; i < it; ++i)
                    mq_wait_parity_drain(&s.ld_full[i % S8], (i / S8) & 1, P.status, P.wait_ns);
            }
        }
        __syncwarp();
    } else if (warp == MMA_WARP) {
        // ------------------------------------------------------ MMA issuer
        // The whole warp runs the loop (warp-uniform control flow: lane 0
        // waits, the verdict is broadcast) and one elected lane issues the
        // MMAs and commits.  Issued from a lone lane behind its waits, pair
        // MMAs of N = 128 ran at 86-94 cycles instead of 64 (measured).
        if (rank == 0) {
            const uint32_t idesc = idesc_f16_f32(TM, TN);
            uint32_t it = 0, chunks = 0;
            bool ok = true;
            Tile t;
            for (int ti = 0; ok && pair_tile_at(P, pair, ti, t); ++ti) {
                uint32_t fcol = 0;
                int kc = 0;  // stage within the exact-f32 chunk
                for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                    const bool chunk_start = kc == 0;
                    if (chunk_start) {
                        const uint32_t b = chunks & 1;
                        if (!warp_wait(&s.f_empty[b], ((chunks >> 1) & 1) ^ 1, s, P)) {
                            ok = false;
                            break;
                        }
                        fcol = F_COL0 + 128 * b;
                    }
                    const int slot = it % SF;
                    if (!warp_wait(&s.op_full[slot], (it / SF) & 1, s, P)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t acol = tmem + A_COL0 + 64 * slot;
                    const uint64_t bd0 = smem_desc_sw128(smem_u32(s.opb[slot]));
                    const uint64_t bd1 = smem_desc_sw128(smem_u32(s.opb[slot] + ATOM));
                    const bool chunk_end = ++kc == t.kpc || kb + 1 == t.nkb;
                    if (elect_one()) {
#pragma unroll
                        for (int j = 0; j < KS / 16; ++j)  // +32 B along K: +2 in the (addr >> 4) field
                            tc_mma2_f16_ts(tmem + fcol, acol + 8 * j,
                                           (j < 4 ? bd0 : bd1) + 2 * (j & 3), idesc,
                                           (chunk_start && j == 0) ? 0u : 1u);
                        tc_commit2_mc(&s.op_empty[slot], 3);
                        if (chunk_end) tc_commit2_mc(&s.f_full[chunks & 1], 3);
                    }
                    __syncwarp();
                    if (chunk_end) {
                        ++chunks;
                        kc = 0;
                    }
                }
            }
            if (!ok && lane == 0) abort_pair(s, rank);
            // every MMA issued above has completed once `done` fires; wait for
            // it even after giving up (bounded, ignoring the abort word): the
            // MMAs read both CTAs' operands and write their tensor memory,
            // which is released after the final cluster barrier.  Every lane
            // commits (`done` counts 32 arrivals), so the phase follows the
            // MMAs of whichever lane the elections picked.
            tc_commit2_mc(&s.done, 1);
            if (lane == 0) mq_wait_parity_drain(&s.done, 0, P.status, P.wait_ns);
        }
        __syncwarp();
    } else if (warp < EPI_WARP0) {
        // ------------------------------------------------------ converters
        // Two groups of four warps take alternate stages, so that the waits
        // and signals of one group overlap the widening work of the other.
        // In its stage, warp w widens all 128 k of weight rows 32 (w % 4) ..
        // +31 (TMEM lanes it may write) and four 16-byte token chunks.
        const int grp = (warp - CONV_WARP0) >> 2;          // 0 or 1
        const int gt = threadIdx.x - (CONV_WARP0 + 4 * grp) * 32;  // 0..127 in the group
        const int quad = warp & 3;                          // TMEM lane quarter of this warp
        const int arow = quad * 32 + lane;                  // weight row in this CTA
        const uint32_t a_lane = tmem + ((uint32_t)(quad * 32) << 16);
        // staging offsets of this thread's weight chunks (128B / 64B swizzle)
        uint32_t a8_src[8], a4_src[4];
#pragma unroll
        for (int i = 0; i < 8; ++i) a8_src[i] = (uint32_t)(arow * 128 + ((i ^ (arow & 7)) << 4));
#pragma unroll
        for (int i = 0; i < 4; ++i)
            a4_src[i] = (uint32_t)(arow * 64 + ((i ^ ((arow >> 1) & 3)) << 4));
        // token chunks g = gt + 128 i: row g >> 3, 16-k chunk g & 7; f16
        // destination: 64-k column g >> 2 & 1, 16-byte chunks 2 (g & 3), +1
        uint32_t b_src[4], b_dst[4][2];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int g = gt + 128 * i, row = g >> 3, kc = g & 7;
            b_src[i] = (uint32_t)(row * 128 + ((kc ^ (row & 7)) << 4));
            const uint32_t base = (uint32_t)((kc >> 2) * ATOM + row * 128);
            const int c0 = 2 * (kc & 3), c1 = c0 + 1;
            // lanes with kc >= 4 store their second chunk first: the eight lanes
            // of a row then hit eight different bank groups on each store
            const int first = (kc & 4) ? c1 : c0, second = (kc & 4) ? c0 : c1;
            b_dst[i][0] = base + (uint32_t)((first ^ (row & 7)) << 4);
            b_dst[i][1] = base + (uint32_t)((second ^ (row & 7)) << 4);
        }
        const bool swap_b = (gt & 4) != 0;
        if constexpr (ZW) griddep_wait();  // the weight zero points are read below
        const uint32_t leader_op_full = cluster_addr(&s.op_full[0], 0);
        const uint32_t leader_sink = cluster_addr(&s.sink[warp - CONV_WARP0], 0);
        uint32_t it = 0;
        bool ok = true;
        Tile t;
        for (int ti = 0; ok && pair_tile_at(P, pair, ti, t); ++ti) {
            const bool i4 = P.p[t.pi].bits == 4;
            // weight row arow widens to w - zw (zw = 0 for symmetric weights):
            // the MMA then sums x (w - zw) and the epilogue needs no rowsum(x)
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
                const uint8_t *sb = s.stb[s8];
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
                uint8_t *ob = s.opb[sf];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const uint4 vb = lds16(sb + b_src[i]);
                    uint32_t h[8];
                    i8x4_to_f16x4(vb.x, h[0], h[1]);
                    i8x4_to_f16x4(vb.y, h[2], h[3]);
                    i8x4_to_f16x4(vb.z, h[4], h[5]);
                    i8x4_to_f16x4(vb.w, h[6], h[7]);
                    if (!swap_b) {
                        sts16(ob + b_dst[i][0], h[0], h[1], h[2], h[3]);
                        sts16(ob + b_dst[i][1], h[4], h[5], h[6], h[7]);
                    } else {
                        sts16(ob + b_dst[i][0], h[4], h[5], h[6], h[7]);
                        sts16(ob + b_dst[i][1], h[0], h[1], h[2], h[3]);
                    }
                }
                // every value read from the staging slot now feeds an issued store
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.ld_empty[s8]);
                tc_wait_st();
                fence_proxy_async_smem();
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
        // ------------------------------------------------------ epilogue
        griddep_wait();  // before the first global access (parameters, residual, y)
        const int quad = warp & 3;                  // TMEM lane quarter of this warp
        const int half = (warp - EPI_WARP0) >> 2;   // token half of the tile
        const uint32_t t_lane = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(64 * half);
        const uint32_t leader_f_empty = cluster_addr(&s.f_empty[0], 0);
        uint32_t chunks = 0;
        bool ok = true;
        Tile t;
        for (int ti = 0; ok && pair_tile_at(P, pair, ti, t); ++ti) {
            const Problem &p = P.p[t.pi];
            const int ch = t.ct * TM + (int)rank * CM + quad * 32 + lane;
            const bool ch_in = ch < p.N;
            const int32_t zw = (ch_in && p.zw) ? __ldg(p.zw + ch) : 0;
            // the chunks sum x (w - zw) (the converters widen w - zw), so
            // sum((x - zx)(w - zw)) = that - zx (colsum - K zw)
            const int32_t corr =
                ch_in ? (int32_t)((uint32_t)(p.zx * __ldg(p.colsum + ch)) -
                                  (uint32_t)p.K * (uint32_t)(p.zx * zw))
                      : 0;
            const int32_t m0 = ch_in ? __ldg(p.M0 + ch) : 0;
            const int32_t sh = ch_in ? __ldg(p.shift + ch) : 33;
            uint32_t acc[64];
#pragma unroll
            for (int i = 0; i < 64; ++i) acc[i] = 0u;
            const int nchunks = t.nkb ? (t.nkb + t.kpc - 1) / t.kpc : 0;
            for (int c = 0; c < nchunks; ++c, ++chunks) {
                const uint32_t b = chunks & 1;
                if (!warp_wait(&s.f_full[b], (chunks >> 1) & 1, s, P)) {
                    if (lane == 0) abort_pair(s, rank);
                    ok = false;
                    break;
                }
                tc_fence_after();
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t f[16];
                    tc_ld_32x32b_x16(t_lane + F_COL0 + 128 * b + 16 * q, f);
                    tc_wait_ld();
                    if constexpr (A16) {
                        // token 8q + i: 256 S(hi) + S(lo) of the chunk, added to the
                        // token's int64 sum (halves in acc[16q + 2i], acc[16q + 2i + 1])
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int64_t d =
                                256 * (int64_t)__float2int_rn(__uint_as_float(f[2 * i])) +
                                (int64_t)__float2int_rn(__uint_as_float(f[2 * i + 1]));
                            uint64_t v = ((uint64_t)acc[16 * q + 2 * i + 1] << 32) | acc[16 * q + 2 * i];
                            v += (uint64_t)d;
                            acc[16 * q + 2 * i] = (uint32_t)v;
                            acc[16 * q + 2 * i + 1] = (uint32_t)(v >> 32);
                        }
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i)
                            acc[16 * q + i] += (uint32_t)__float2int_rn(__uint_as_float(f[i]));
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(leader_f_empty + 8u * b);
            }
            if (!ok) break;
            if (!ch_in) continue;
            const EpiArgs e{p.y, p.residual, p.M, p.ldy, p.zy};
            const int tok0 = t.tt * TN + 64 * half;
            const int ntok = min(64, e.M - tok0);
            if constexpr (A16) {
                // acc pairs hold each token's int64 sum 256 S(hi) + S(lo) of
                // x (w - zw) (the converters widen w - zw):
                // sum((x - zx)(w - zw)) = that + (128 - zx) (colsum - K zw)
                const int64_t cs = (int64_t)__ldg(p.colsum + ch);
                const int64_t c16 =
                    (int64_t)(128 - p.zx) * (ZW ? cs - (int64_t)p.K * zw : cs);
                int16_t *yp = reinterpret_cast<int16_t *>(e.y) + (size_t)(tok0 >> 1) * (size_t)e.ldy + ch;
                const int n16 = ntok >> 1;
                const size_t ldy16 = (size_t)e.ldy;
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (j < n16) {
                        const int64_t a =
                            (int64_t)(((uint64_t)acc[2 * j + 1] << 32) | acc[2 * j]) + c16;
                        yp[(size_t)j * ldy16] = (int16_t)mq_requant16(a, m0, sh, e.zy);
                    }
                continue;
            }
            const size_t ldy = (size_t)e.ldy;
            if constexpr (O16) {
                int16_t *yp16 = reinterpret_cast<int16_t *>(e.y) + (size_t)tok0 * ldy + ch;
                if (ntok == 64 && sh >= 33)
                    store_channel16<true, true>(acc, corr, m0, sh, e.zy, yp16, ldy, 64);
                else
                    store_channel16<false, false>(acc, corr, m0, sh, e.zy, yp16, ldy, ntok);
                continue;
            }
            int8_t *yp = e.y + (size_t)tok0 * ldy + ch;
            const int8_t *rp = e.residual ? e.residual + (size_t)tok0 * ldy + ch : nullptr;
            const bool full = ntok == 64, fast = sh >= 33;
            if (rp) {
                if (full && fast) store_channel<true, true, true>(acc, corr, m0, sh, e.zy, yp, rp, ldy, 64);
                else store_channel<true, false, false>(acc, corr, m0, sh, e.zy, yp, rp, ldy, ntok);
            } else {
                if (full && fast) store_channel<false, true, true>(acc, corr, m0, sh, e.zy, yp, rp, ldy, 64);
                else store_channel<false, false, false>(acc, corr, m0, sh, e.zy, yp, rp, ldy, ntok);
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

// cuTensorMapEncodeTiled through the runtime's driver entry point (no libcuda
// link dependency).
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

// 2-D uint8 tensor [rows][cols] with row pitch `pitch` bytes, box box_cols x
// box_rows, 128- or 64-byte swizzle (box_cols bytes per row).
bool encode_2d(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows, uint64_t pitch,
               uint32_t box_cols, uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {pitch};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle swz =
        box_cols == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
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
    if (cudaOccupancyMaxActiveClusters(&clusters, prefill_kernel<false, false, false>, &cfg) ==
            cudaSuccess &&
        clusters > 0 && clusters < n)
        n = clusters;
    if (n > MAX_PAIRS) n = MAX_PAIRS;
    if (dev >= 0 && dev < 64) cached[dev] = n;
    return n;
}

// Longest-processing-time-first assignment of tiles to pairs.  Tile ids are
// numbered problem by problem; work = stages + a fixed epilogue share.
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

}  // namespace prefill

int launch_prefill(const Problem *probs, int count, void *stream) {
    using namespace prefill;
    // the kernels' dynamic shared-memory limit, raised once per device (the
    // attribute belongs to the device's context)
    static std::atomic<uint64_t> attr_done{0};  // bit d: device d prepared
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return MQ_ERR_CUDA;
    if (!(attr_done.load(std::memory_order_acquire) & (1ull << dev))) {
        const int smem = (int)SMEM_BYTES;
        const auto attr = cudaFuncAttributeMaxDynamicSharedMemorySize;
        if (cudaFuncSetAttribute(prefill_kernel<false, false, false>, attr, smem) != cudaSuccess ||
            cudaFuncSetAttribute(prefill_kernel<false, false, true>, attr, smem) != cudaSuccess ||
            cudaFuncSetAttribute(prefill_kernel<true, false, false>, attr, smem) != cudaSuccess ||
            cudaFuncSetAttribute(prefill_kernel<true, false, true>, attr, smem) != cudaSuccess ||
            cudaFuncSetAttribute(prefill_kernel<false, true, true>, attr, smem) != cudaSuccess)
            return MQ_ERR_CUDA;
        attr_done.fetch_or(1ull << dev, std::memory_order_release);
    }
    if (count <= 0) return MQ_OK;
    const int pairs_max = max_pairs(dev);
    if (pairs_max < 1) return MQ_ERR_CUDA;
    for (int begin = 0; begin < count; begin += PREFILL_MAX_PROBLEMS) {
        const int n = count - begin < PREFILL_MAX_PROBLEMS ? count - begin : PREFILL_MAX_PROBLEMS;
        bool any_zw = false;
        for (int i = begin; i < begin + n; ++i) any_zw = any_zw || probs[i].zw != nullptr;
        // 16-bit outputs always take the zero-point variant (their time is the
        // epilogue's, not the widening's)
        auto kern = probs[0].a16   ? (any_zw ? prefill_kernel<true, false, true>
                                             : prefill_kernel<true, false, false>)
                    : probs[0].o16 ? prefill_kernel<false, true, true>
                    : any_zw       ? prefill_kernel<false, false, true>
                                   : prefill_kernel<false, false, false>;
        Params P{};
        P.pre_w = 1;
        long long tiles = 0;
        // longest K first (round-robin order; the table orders by work itself)
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
            if (q.wdynamic) P.pre_w = 0;
            q.tiles_m = (q.M + TN - 1) / TN;
            q.tile_begin = (int)tiles;
            tiles += (long long)q.tiles_m * ((q.N + TM - 1) / TM);
            if (q.K > 0) {
                const bool i4 = q.bits == 4;
                const uint64_t wcols = i4 ? (uint64_t)q.K / 2 : (uint64_t)q.K;
                if (!encode_2d(&P.tmap_x[i], q.x, (uint64_t)q.K, (uint64_t)q.M, (uint64_t)q.ldx,
                               KS, CN) ||
                    !encode_2d(&P.tmap_w[i], q.w, wcols, (uint64_t)q.N, (uint64_t)q.ldw,
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
        // programmatic stream serialization: this launch may start while the
        // previous kernel in the stream finishes (see griddep_wait)
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
