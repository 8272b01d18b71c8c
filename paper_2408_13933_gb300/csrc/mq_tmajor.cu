// mq_tmajor.cu -- the token-major tensor-core kernel: tokens are the MMA's M
// (128 per tile) and output channels its N, the transpose of the prefill
// kernels' roles.  It serves the shapes those kernels are not built for:
// short K or few channels, i.e. the attention matmuls of the integer block
// (Sec. 4.1; Q K^T at K = head dim 64 with int16 scores, P V with N = head
// dim 64).
//
// Both zero points are folded into the widening: the tensor cores contract
// x - zx and w - zw (f16 integers, |.| <= 255), so the accumulator is the
// corrected sum itself and the epilogue only requantizes.  Each f32 run of
// the contraction is exact: its partial sums stay below 2^24 (narrow tiles)
// or 2^22 (wide tiles, whose epilogue converts them to int32 with an add
// instead of a conversion instruction); the run length is that bound over the
// largest |x - zx| |w - zw|, in whole stages.
//
// A tile's accumulator lives in tensor memory with one token per lane, so an
// epilogue thread holds 32 consecutive channels of one token after one
// tcgen05.ld.  Where the 32 channels share M0 and shift (per-tensor scales,
// as in attention) the requantization is a multiply-high, an add, a shift and
// a saturating pack per value.  The warp writes its block of 32 tokens x 64
// channels into shared memory by rows and stores it to y by 16-byte chunks
// of whole row segments (each store instruction covers whole 128-byte rows
// of the int16 scores), with their parameters loaded one tile ahead.
//
//   global int8 --TMA (S8 stages, x: 128 x 64 B, w: TN x 64 B)--> shared
//   --converter warps: int8 -> f16 (x - zx, w - zw), 128-byte swizzled
//   K-major--> operand stages (SF) --MMA M128 x N(TN) x K16, one thread-->
//   F[b] in TMEM (two buffers) --8 epilogue warps--> y.
//
// Tile shapes: TN = 256 channels when K fits one exact run and N > 64 (the
// epilogue requantizes each tile straight out of tensor memory), else TN = 64
// (with several runs each epilogue thread keeps 64 running int32 sums).
//
// Transposed weights (w stored [K][N], e.g. attention's V read in place for
// P V): narrow tiles only.  TMA stages 64 k-rows x 64 channels; the
// converters widen them row by row into an f16 tile with channels contiguous
// (128-byte swizzled, N-major), which the MMA reads as an N-major B operand,
// so no transpose is made anywhere.
//
// Warp roles (one CTA per SM, persistent over a contiguous range of tiles):
//   warp 0      TMA producer (one thread)
//   warp 1      tensor-memory allocation, MMA issue (one elected lane)
//   then        converters: one group of four warps (wide tiles) or two
//               taking alternate stages (narrow): widen a stage of x and w
//               into an operand slot
//   then        epilogue: 16 warps (wide) or 4 (narrow); each drains TMEM
//               lanes 32 (w % 4) .. + 31 (its tokens) and 64 columns
// Every mbarrier wait is bounded (mq_wait_parity); a timeout raises the CTA's
// abort word and every role unwinds, waiting for issued MMAs and loads first.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <atomic>

#include "mq_internal.h"
#include "mq_ptx.cuh"
#include "mq_tmajor.h"

namespace mq {

namespace prefill {
PFN_cuTensorMapEncodeTiled_v12000 encode_fn();
}  // namespace prefill

namespace tmajor {

constexpr int TMT = 128;  // tokens per tile (MMA M)
constexpr int TNW = 256;  // channels per wide tile (one exact run)
constexpr int TNN = 64;   // channels per narrow tile (any K)
constexpr int KS = 64;    // k per stage: one 128-byte f16 row
constexpr int TMA_WARP = 0;
constexpr int MMA_WARP = 1;
constexpr int CONV_WARP0 = 2;
constexpr int GROUP_WARPS = 4;  // converter warps of one group
constexpr int GROUP_THREADS = GROUP_WARPS * 32;
constexpr int STX = TMT * KS;   // token staging bytes
constexpr int OPA = TMT * 128;  // f16 token operand
constexpr int OUTB = 32 * 128;  // one 32 x 64 output block (int16; int8 uses half)
constexpr uint32_t TMEM_COLS = 512;  // F[b] at column 256 b

// The two tile shapes, each its own kernel.  Wide: 256 channels, one stage
// per tile (the scores): a short pipeline, 16 epilogue warps for the
// requantization.  Narrow: 64 channels over many stages (long K): eight
// staging stages (the loads of P's 64-byte row segments take ~2 us to land),
// four operand slots and two converter groups taking alternate stages (each
// group's waits and signals overlap the other's widening), four epilogue
// warps.
template <bool NARROW>
struct Cfg {
    static constexpr int TN = NARROW ? TNN : TNW;
    static constexpr int S8 = NARROW ? 8 : 2;  // staging stages
    static constexpr int SF = NARROW ? 4 : 2;  // operand slots
    static constexpr int GROUPS = NARROW ? 2 : 1;
    static constexpr int EPI_WARP0 = CONV_WARP0 + GROUPS * GROUP_WARPS;
    static constexpr int EPI_WARPS = NARROW ? 4 : 16;
    static constexpr int THREADS = (EPI_WARP0 + EPI_WARPS) * 32;
    static constexpr int STW = TN * KS;   // weight staging bytes
    static constexpr int OPB = TN * 128;  // f16 weight operand
    // accumulator buffers F[b] at tensor-memory column b TN: two wide ones;
    // four narrow ones, so that the MMAs run ahead of the epilogue's drains
    static constexpr int NF = NARROW ? 4 : 2;
    // exact runs: partial sums below 2^22 for the wide epilogue's add-based
    // conversion, below 2^24 (f32's exact integers) for the narrow one's
    static constexpr int RUN_BITS = NARROW ? 24 : 22;
};

// ----------------------------------------------------------------- PTX helpers
__device__ __forceinline__ void tmem_alloc1(uint32_t *dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(dst_smem)), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tmem_relinquish1() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc1(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;"
                 ::"r"(taddr), "r"(ncols) : "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16, both operands by descriptor.
__device__ __forceinline__ void mma_f16_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                           uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive once on this CTA's mbarrier `bar` when every tcgen05 operation
// issued so far by this thread has completed.
__device__ __forceinline__ void commit1(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
                 ::"r"(smem_u32(bar)) : "memory");
}

// 2-D tiled TMA store of the box at (x, y) from shared memory, as one bulk
// group of this thread.
__device__ __forceinline__ void tma_store_2d(const void *map, int x, int y, const void *src) {
    asm volatile(
        "cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];"
        ::"l"(map), "r"(x), "r"(y), "r"(smem_u32(src)) : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

// Wait until none of this thread's bulk groups still reads shared memory.
__device__ __forceinline__ void store_wait_read0() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}

// Two int32 saturated to int16 and packed: `lo` in the low half.
__device__ __forceinline__ uint32_t pack2_sat_s16(int32_t lo, int32_t hi) {
    uint32_t d;
    asm("cvt.pack.sat.s16.s32 %0, %1, %2;" : "=r"(d) : "r"(hi), "r"(lo));
    return d;
}

// Four int32 saturated to int8 and packed, value i in byte i.
__device__ __forceinline__ uint32_t pack4_sat_s8(int32_t v0, int32_t v1, int32_t v2, int32_t v3) {
    uint32_t hi, d;
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(hi) : "r"(v3), "r"(v2), "r"(0u));
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(v1), "r"(v0), "r"(hi));
    return d;
}

// ------------------------------------------------------------------ kernel
struct Params {
    CUtensorMap tmap_x[PREFILL_MAX_PROBLEMS];  // int8 [M][ldx], box 64 B x 128, no swizzle
    CUtensorMap tmap_w[PREFILL_MAX_PROBLEMS];  // int8 [N][ldw], box 64 B x TN, no swizzle
    CUtensorMap tmap_y[PREFILL_MAX_PROBLEMS];  // y [M][ldy], box 64 (wide) / 32 channels x 32, swizzled
    Problem p[PREFILL_MAX_PROBLEMS];            // tile_begin; tiles_m: token tiles
    int tn[PREFILL_MAX_PROBLEMS];               // channels per tile: TNW or TNN
    int kpr[PREFILL_MAX_PROBLEMS];              // stages per exact run
    int vec[PREFILL_MAX_PROBLEMS];              // y (and residual) rows allow 16-byte accesses
    int tma_y[PREFILL_MAX_PROBLEMS];            // y written by TMA stores (vec, no residual)
    int part[PREFILL_MAX_PROBLEMS];             // y is int32 [M][ldy]: raw sums of a slice of K
    int wt[PREFILL_MAX_PROBLEMS];               // w stored [K][ldw] (narrow tiles); tmap_w: box
                                                // 64 channels x 64 k
    int count;
    int total_tiles;
    int *status;
    uint64_t wait_ns;
};

template <bool NARROW>
struct Smem {
    using C = Cfg<NARROW>;
    uint8_t opa[C::SF][OPA];  // 1024-byte aligned (the swizzle pattern follows address bits)
    uint8_t opb[C::SF][C::OPB];
    uint8_t out[C::EPI_WARPS][OUTB];  // per epilogue warp: a block of 32 tokens x 64 channels
    Problem prob[PREFILL_MAX_PROBLEMS];  // the problem table (parameter reads are slow)
    int tn[PREFILL_MAX_PROBLEMS], kpr[PREFILL_MAX_PROBLEMS], flags[PREFILL_MAX_PROBLEMS];
    uint8_t stx[C::S8][STX];
    uint8_t stw[C::S8][C::STW];
    uint64_t ld_full[C::S8];
    uint64_t ld_empty[C::S8];
    uint64_t op_full[C::SF];
    uint64_t op_empty[C::SF];
    uint64_t f_full[C::NF];
    uint64_t f_empty[C::NF];
    uint64_t done;
    uint32_t tmem_base;
    int abort;
};

template <bool NARROW>
constexpr size_t smem_bytes() {
    return sizeof(Smem<NARROW>) + 1024;  // + alignment slack
}

struct Tile {
    int pi, tt, ct, tn;
    int nkb, kpr;  // stages, stages per exact run
};

// The last problem whose first tile is <= tile.
template <class S>
__device__ __forceinline__ int problem_of(const S &s, int count, int tile) {
    int lo = 0, hi = count - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (s.prob[mid].tile_begin <= tile)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

template <class S>
__device__ __forceinline__ Tile tile_of(const S &s, int count, int tile) {
    Tile t;
    t.pi = problem_of(s, count, tile);
    const Problem &p = s.prob[t.pi];
    const int local = tile - p.tile_begin;
    t.tt = local % p.tiles_m;
    t.ct = local / p.tiles_m;
    t.tn = s.tn[t.pi];
    t.nkb = (p.K + KS - 1) / KS;
    t.kpr = s.kpr[t.pi];
    return t;
}

template <class S>
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, S &s, const Params &P) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0) ok = mq_wait_parity(bar, parity, &s.abort, P.status, P.wait_ns);
    return __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
}

// Byte offset of 16-byte chunk j (0..7) of row r in a 128-byte swizzled
// K-major tile: rows 128 bytes apart, chunk index xor (r mod 8).
__device__ __forceinline__ uint32_t sw128(int r, int j) {
    return (uint32_t)(r * 128 + ((j ^ (r & 7)) << 4));
}

// 16 int8 (one staged 16-byte chunk) -> 16 f16 (v - z, `off` from
// f16x2_i8_offset(z)) into chunks 2c and 2c + 1 of row r.  Elements from
// `live` on are written as 0 (k past K: TMA fills zeros there, whose v - z
// would not vanish).
__device__ __forceinline__ void widen_chunk(const uint8_t *src, uint8_t *dst, int r, int c,
                                            uint32_t off, int live = 16) {
    const uint4 v = *reinterpret_cast<const uint4 *>(src);
    uint32_t h[8];
    i8x4_to_f16x4(v.x, h[0], h[1], off);
    i8x4_to_f16x4(v.y, h[2], h[3], off);
    i8x4_to_f16x4(v.z, h[4], h[5], off);
    i8x4_to_f16x4(v.w, h[6], h[7], off);
    if (live < 16) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const uint32_t keep = (2 * e < live ? 0xFFFFu : 0u) | (2 * e + 1 < live ? 0xFFFF0000u : 0u);
            h[e] &= keep;
        }
    }
    *reinterpret_cast<uint4 *>(dst + sw128(r, 2 * c)) = make_uint4(h[0], h[1], h[2], h[3]);
    *reinterpret_cast<uint4 *>(dst + sw128(r, 2 * c + 1)) = make_uint4(h[4], h[5], h[6], h[7]);
}

// The weights' offsets of one staged [K][N] chunk (16 channels ch0 .. ch0 +
// 15, one k): off[e] holds channels ch0 + 2e (low half) and ch0 + 2e + 1
// (high half), 1152 + zw, or 1152 without a zero point or past N.
template <int NOFF>
__device__ __forceinline__ void wt_offsets(const Problem &p, int ch0, uint32_t (&off)[NOFF]) {
    static_assert(NOFF >= 8, "eight channel pairs");
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        uint32_t lo = 0x6480u, hi = 0x6480u;
        const int ch = ch0 + 2 * e;
        if (p.zw && ch < p.N) lo = (uint32_t)(0x6480 + __ldg(p.zw + ch));
        if (p.zw && ch + 1 < p.N) hi = (uint32_t)(0x6480 + __ldg(p.zw + ch + 1));
        off[e] = (hi << 16) | lo;
    }
}

// 16 int8 of one k (channels of one staged [K][N] chunk) -> 16 f16 (w - zw
// per channel, offsets from wt_offsets) into chunks 2c and 2c + 1 of row r of
// the N-major tile (the same 128-byte swizzle, rows now along k).
template <int NOFF>
__device__ __forceinline__ void widen_chunk_pairs(const uint8_t *src, uint8_t *dst, int r, int c,
                                                  const uint32_t (&off)[NOFF]) {
    const uint4 v = *reinterpret_cast<const uint4 *>(src);
    const uint32_t q[4] = {v.x, v.y, v.z, v.w};
    uint32_t h[8];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const uint32_t u = q[e] ^ 0x80808080u;
        h[2 * e] = hsub2(prmt(u, 0x64646464u, 0x4140u), off[2 * e]);
        h[2 * e + 1] = hsub2(prmt(u, 0x64646464u, 0x4342u), off[2 * e + 1]);
    }
    *reinterpret_cast<uint4 *>(dst + sw128(r, 2 * c)) = make_uint4(h[0], h[1], h[2], h[3]);
    *reinterpret_cast<uint4 *>(dst + sw128(r, 2 * c + 1)) = make_uint4(h[4], h[5], h[6], h[7]);
}

// Shared-memory descriptor of an N-major operand in 128-byte swizzle atoms
// (8 k-rows of 64 f16 channels, 1024 B): atoms along k 1024 B apart (the
// stride field); along N (the leading field) there is one atom in a 64-channel
// tile, given 1024 B as well.
__device__ __forceinline__ uint64_t smem_desc_sw128_nmajor(uint32_t saddr) {
    return (smem_desc_sw128(saddr) & ~(0x3FFFull << 16)) | ((uint64_t)(1024u >> 4) << 16);
}

// An f32 accumulator holding an integer v with |v| < 2^22 -> v: adding
// 1.5 * 2^23 puts v in the low mantissa bits exactly (one add and one integer
// subtract instead of a conversion instruction).
__device__ __forceinline__ int32_t f2i_exact(uint32_t f) {
    return __float_as_int(__fadd_rn(__uint_as_float(f), 12582912.0f)) - 0x4B400000;
}

// Requantize one token's 32 sums (this lane's row; channels ch0 .. ch0 + 31
// with M0 / shift in lane i of m0 / sh, all equal when `uniform`) into
// 16 (int16) or 8 (int8) packed words.
template <bool O16>
__device__ __forceinline__ void requant32(const int32_t (&a)[32], int32_t m0, int32_t sh,
                                          bool uniform, int32_t zy, uint32_t (&w)[16]) {
    const int32_t m00 = __shfl_sync(0xffffffffu, m0, 0);
    const int32_t sh0 = __shfl_sync(0xffffffffu, sh, 0);
    if (uniform && sh0 >= 33) {  // exact multiply-high form, saturating packs
        // floor((h + 2^(rs-1)) / 2^rs) + zy = floor((h + 2^(rs-1) + zy 2^rs) / 2^rs); the
        // single bias is used where it and |h| <= 2^30 cannot overflow
        const int32_t rs = sh0 - 32;
        const int64_t bias = ((int64_t)1 << (rs - 1)) + ((int64_t)zy << rs);
        const bool fold = bias > -((int64_t)1 << 30) && bias < ((int64_t)1 << 30);
        const int32_t b1 = fold ? (int32_t)bias : (1 << (rs - 1));
        const int32_t b2 = fold ? 0 : zy;
#pragma unroll
        for (int i = 0; i < 32; i += 4) {
            int32_t q[4];
            if (fold) {
#pragma unroll
                for (int e = 0; e < 4; ++e) q[e] = (__mulhi(a[i + e], m00) + b1) >> rs;
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e) q[e] = ((__mulhi(a[i + e], m00) + b1) >> rs) + b2;
            }
            if (O16) {
                w[i / 2] = pack2_sat_s16(q[0], q[1]);
                w[i / 2 + 1] = pack2_sat_s16(q[2], q[3]);
            } else {
                w[i / 4] = pack4_sat_s8(q[0], q[1], q[2], q[3]);
            }
        }
    } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            const int32_t m0i = __shfl_sync(0xffffffffu, m0, i);
            const int32_t shi = __shfl_sync(0xffffffffu, sh, i);
            if (O16) {
                const int32_t o = mq_requant16((int64_t)a[i], m0i, shi, zy);
                if (i & 1)
                    w[i >> 1] |= (uint32_t)(uint16_t)o << 16;
                else
                    w[i >> 1] = (uint32_t)(uint16_t)o;
            } else {
                const int32_t o = mq_requant(a[i], m0i, shi, zy);
                if ((i & 3) == 0) w[i >> 2] = 0u;
                w[i >> 2] |= (uint32_t)(uint8_t)o << (8 * (i & 3));
            }
        }
    }
}

// The warp's output block: 32 token rows x 32 or 64 channels of 1- or
// 2-byte codes, rows RB = 128, 64 or 32 bytes apart, laid out as the TMA
// store of that row width swizzles it (128-, 64- or 32-byte swizzle: 16-byte
// chunk j of row r at chunk j ^ (r mod 8), j ^ ((r / 2) mod 4), j ^ ((r / 4)
// mod 2)), which also keeps the row writes and chunk reads conflict-free.
__device__ __forceinline__ uint32_t out_off(int r, int j, int rb) {
    const int x = rb == 128 ? (r & 7) : (rb == 64 ? ((r >> 1) & 3) : ((r >> 2) & 1));
    return (uint32_t)(r * rb + ((j ^ x) << 4));
}

// Row `lane` of the block: the words of 32 channels at column group g (0 or 1).
template <bool O16, int RB>
__device__ __forceinline__ void stage32(uint8_t *blk, int g, int lane, const uint32_t (&w)[16]) {
    constexpr int NCH = O16 ? 4 : 2;  // 16-byte chunks of 32 codes
#pragma unroll
    for (int j = 0; j < NCH; ++j)
        *reinterpret_cast<uint4 *>(blk + out_off(lane, g * NCH + j, RB)) =
            make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
}

// Write the staged block (rows of RB bytes) to y: lanes take consecutive
// 16-byte chunks of consecutive rows (whole row segments per instruction),
// adding the residual (int8) chunk by chunk; rows past M are skipped, chunks
// that reach past N (or rows without 16-byte alignment) go element by element.
template <bool O16, int RB>
__device__ __forceinline__ void store_block(const uint8_t *blk, const Problem &p, int tok0,
                                            int ch0, bool vec, int lane) {
    constexpr int OSZ = O16 ? 2 : 1;
    constexpr int E = 16 / OSZ;     // codes per chunk
    constexpr int CPR = RB / 16;    // chunks per row
    constexpr int RPI = 32 / CPR;   // rows per pass of the warp
    const int j = lane % CPR;
    const int ch = ch0 + j * E;
    const bool full = vec && ch + E <= p.N;
    const size_t ldy = (size_t)p.ldy;
#pragma unroll
    for (int i = 0; i < 32 / RPI; ++i) {
        const int r = lane / CPR + RPI * i;
        const int tok = tok0 + r;
        if (tok >= p.M || ch >= p.N) continue;
        uint4 v = *reinterpret_cast<const uint4 *>(blk + out_off(r, j, RB));
        const size_t at = (size_t)tok * ldy + (size_t)ch;
        if (full) {
            if (!O16 && p.residual) {
                const uint4 q = __ldg(reinterpret_cast<const uint4 *>(p.residual + at));
                v.x = __vaddss4(v.x, q.x), v.y = __vaddss4(v.y, q.y);
                v.z = __vaddss4(v.z, q.z), v.w = __vaddss4(v.w, q.w);
            }
            *reinterpret_cast<uint4 *>(reinterpret_cast<uint8_t *>(p.y) + at * OSZ) = v;
        } else {
            const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int e = 0; e < E; ++e)
                if (ch + e < p.N) {
                    if (O16) {
                        reinterpret_cast<int16_t *>(p.y)[at + e] =
                            (int16_t)(wv[e >> 1] >> (16 * (e & 1)));
                    } else {
                        int32_t o = (int32_t)(int8_t)(wv[e >> 2] >> (8 * (e & 3)));
                        if (p.residual) o = min(127, max(-128, o + (int32_t)p.residual[at + e]));
                        p.y[at + e] = (int8_t)o;
                    }
                }
        }
    }
}

// The warp's staged block out to y: one TMA store (lane 0 issues it after
// every lane's writes are visible to the async proxy), or 16-byte stores.
template <bool O16, int RB>
__device__ __forceinline__ void flush_block(uint8_t *blk, const Problem &p, const void *tmap,
                                            int tok0, int ch0, bool vec, bool by_tma, int lane) {
    if (by_tma) {
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) tma_store_2d(tmap, ch0, tok0, blk);
    } else {
        __syncwarp();
        store_block<O16, RB>(blk, p, tok0, ch0, vec, lane);
        __syncwarp();
    }
}

// A slice of split K: this lane's token's 32 raw sums (channels ch0 .. ch0 +
// 31) into the int32 partial buffer y [M][ldy].
__device__ __forceinline__ void store_part32(const int32_t *a, const Problem &p, int tok, int ch0) {
    if (tok >= p.M) return;
    int32_t *y = reinterpret_cast<int32_t *>(p.y) + (size_t)tok * (size_t)p.ldy + ch0;
    const bool vec = (p.ldy & 3) == 0 && (reinterpret_cast<uintptr_t>(p.y) & 15) == 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        const int ch = ch0 + 4 * j;
        if (vec && ch + 4 <= p.N) {
            *reinterpret_cast<int4 *>(y + 4 * j) =
                make_int4(a[4 * j], a[4 * j + 1], a[4 * j + 2], a[4 * j + 3]);
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e)
                if (ch + e < p.N) y[4 * j + e] = a[4 * j + e];
        }
    }
}

// O16: every problem of the launch has an int16 output (else int8).  NARROW:
// the narrow tile shape (every problem of the launch has it).
template <bool O16, bool NARROW>
__global__ void __launch_bounds__(Cfg<NARROW>::THREADS, 1)
    tmajor_kernel(const __grid_constant__ Params P) {
    using C = Cfg<NARROW>;
    constexpr int S8 = C::S8, SF = C::SF, THREADS = C::THREADS;
    constexpr int EPI_WARP0 = C::EPI_WARP0, EPI_WARPS = C::EPI_WARPS;
    extern __shared__ uint8_t smem_raw[];
    Smem<NARROW> &s = *reinterpret_cast<Smem<NARROW> *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    for (int i = threadIdx.x; i < P.count; i += THREADS) {
        s.prob[i] = P.p[i];
        s.tn[i] = P.tn[i];
        s.kpr[i] = P.kpr[i];
        s.flags[i] = (P.vec[i] ? 1 : 0) | (P.tma_y[i] ? 2 : 0) | (P.part[i] ? 4 : 0) |
                     (NARROW && P.wt[i] ? 8 : 0);
    }
    if (threadIdx.x == 0) {
        for (int i = 0; i < S8; ++i) {
            mbar_init(&s.ld_full[i], 1);
            mbar_init(&s.ld_empty[i], GROUP_WARPS);
        }
        for (int i = 0; i < SF; ++i) {
            mbar_init(&s.op_full[i], GROUP_WARPS);
            mbar_init(&s.op_empty[i], 1);
        }
        for (int b = 0; b < C::NF; ++b) {
            mbar_init(&s.f_full[b], 1);
            mbar_init(&s.f_empty[b], EPI_WARPS);
        }
        mbar_init(&s.done, 32);  // one commit from every lane of the MMA warp
        s.abort = 0;
        fence_mbar_init();
    }
    if (warp == MMA_WARP) {
        tmem_alloc1(&s.tmem_base, TMEM_COLS);
        tmem_relinquish1();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (threadIdx.x == 0) griddep_launch_dependents();
    const uint32_t tmem = s.tmem_base;
    // this CTA's tiles: a contiguous, balanced range (neighbouring tiles share
    // their weight rows, so concurrent CTAs spread over the weight tiles)
    const int tile0 = (int)(((long long)P.total_tiles * blockIdx.x) / gridDim.x);
    const int tile1 = (int)(((long long)P.total_tiles * (blockIdx.x + 1)) / gridDim.x);

    if (warp == TMA_WARP) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            for (int i = 0; i < P.count; ++i) {
                prefetch_tensormap(&P.tmap_x[i]);
                prefetch_tensormap(&P.tmap_w[i]);
            }
            griddep_wait();  // x and w may be the previous kernel's outputs
            uint32_t it = 0;
            bool ok = true;
            for (int tile = tile0; ok && tile < tile1; ++tile) {
                const Tile t = tile_of(s, P.count, tile);
                const uint32_t bytes = (uint32_t)(STX + t.tn * KS);
                for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                    const int slot = it % S8;
                    if (!mq_wait_parity(&s.ld_empty[slot], ((it / S8) & 1) ^ 1, &s.abort,
                                        P.status, P.wait_ns)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&s.ld_full[slot], bytes);
                    tma_load_2d(s.stx[slot], &P.tmap_x[t.pi], kb * KS, t.tt * TMT,
                                &s.ld_full[slot]);
                    if (s.flags[t.pi] & 8)  // [K][N]: x = channel, y = k
                        tma_load_2d(s.stw[slot], &P.tmap_w[t.pi], t.ct * t.tn, kb * KS,
                                    &s.ld_full[slot]);
                    else
                        tma_load_2d(s.stw[slot], &P.tmap_w[t.pi], kb * KS, t.ct * t.tn,
                                    &s.ld_full[slot]);
                }
            }
            if (!ok) {
                // loads already issued land before the CTA may leave: only the
                // last S8 stages can still be in flight
                s.abort = 1;
                for (uint32_t i = it > (uint32_t)S8 ? it - S8 : 0u; i < it; ++i)
                    mq_wait_parity_drain(&s.ld_full[i % S8], (i / S8) & 1, P.status, P.wait_ns);
            }
        }
        __syncwarp();
    } else if (warp == MMA_WARP) {
        // ------------------------------------------------------ MMA issuer
        // the whole warp runs the loop (lane 0 waits, the verdict is
        // broadcast) and one elected lane issues and commits
        uint32_t it = 0, runs = 0;
        bool ok = true;
        for (int tile = tile0; ok && tile < tile1; ++tile) {
            const Tile t = tile_of(s, P.count, tile);
            const bool wt = (s.flags[t.pi] & 8) != 0;
            // an N-major B (transposed weights): the "transpose B" bit; its
            // 16-k steps are 16 rows of 128 bytes, 2048 B (+128 in addr >> 4)
            const uint32_t idesc = idesc_f16_f32(TMT, t.tn) | (wt ? 1u << 16 : 0u);
            const uint32_t bstep = wt ? 128u : 2u;
            int kr = 0;  // stage within the exact run
            for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                const bool run_start = kr == 0;
                const uint32_t b = runs % C::NF;
                if (run_start && !warp_wait(&s.f_empty[b], ((runs / C::NF) & 1) ^ 1, s, P)) {
                    ok = false;
                    break;
                }
                const int slot = it % SF;
                if (!warp_wait(&s.op_full[slot], (it / SF) & 1, s, P)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const bool run_end = ++kr == t.kpr || kb + 1 == t.nkb;
                if (elect_one()) {
                    const uint64_t ad = smem_desc_sw128(smem_u32(s.opa[slot]));
                    const uint64_t bd = wt ? smem_desc_sw128_nmajor(smem_u32(s.opb[slot]))
                                           : smem_desc_sw128(smem_u32(s.opb[slot]));
#pragma unroll
                    for (int j = 0; j < KS / 16; ++j)  // +32 B along K: +2 in the (addr >> 4) field
                        mma_f16_ss(tmem + (uint32_t)C::TN * b, ad + 2 * j, bd + bstep * j, idesc,
                                   (run_start && j == 0) ? 0u : 1u);
                    commit1(&s.op_empty[slot]);
                    if (run_end) commit1(&s.f_full[b]);
                }
                __syncwarp();
                if (run_end) {
                    ++runs;
                    kr = 0;
                }
            }
        }
        if (!ok && lane == 0) s.abort = 1;
        // every MMA issued above has completed once `done` fires (bounded,
        // ignoring the abort word): they read shared memory and write tensor
        // memory, both released after the final barrier
        commit1(&s.done);
        if (lane == 0) mq_wait_parity_drain(&s.done, 0, P.status, P.wait_ns);
        __syncwarp();
    } else if (warp < EPI_WARP0) {
        // ------------------------------------------------------ converters
        griddep_wait();  // before reading the weight zero points
        const int grp = (warp - CONV_WARP0) / GROUP_WARPS;  // stages it with it % GROUPS == grp
        const int ct = threadIdx.x - (CONV_WARP0 + GROUP_WARPS * grp) * 32;  // 0 .. 127
        uint32_t it = 0;
        bool ok = true;
        for (int tile = tile0; ok && tile < tile1; ++tile) {
            const Tile t = tile_of(s, P.count, tile);
            const Problem &p = s.prob[t.pi];
            const uint32_t xoff = f16x2_i8_offset(p.zx);
            // the weight rows this thread widens: r = ct / 4 + 32 u
            const int wchunks = t.tn * (KS / 16);  // 16-byte chunks of the staged w
            uint32_t woff[C::TN / 32 > 8 ? C::TN / 32 : 8];  // >= 8 for wt_offsets
            const bool wt = NARROW && (s.flags[t.pi] & 8) != 0;
            if (wt) {
                // [K][N] staging: this thread's chunks are channels 16 (ct % 4) ..
                // + 15 of every row; one offset per channel pair
                wt_offsets(p, t.ct * t.tn + 16 * (ct & 3), woff);
            } else {
#pragma unroll
                for (int u = 0; u < C::TN / 32; ++u) {
                    const int ch = t.ct * t.tn + (ct >> 2) + 32 * u;
                    woff[u] = F16X2_1152;
                    if (p.zw && 32 * u < t.tn && ch < p.N)
                        woff[u] = f16x2_i8_offset(__ldg(p.zw + ch));
                }
            }
            for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                if ((int)(it % C::GROUPS) != grp) continue;  // the other group's stage
                const int s8 = it % S8, sf = it % SF;
                if (!warp_wait(&s.ld_full[s8], (it / S8) & 1, s, P) ||
                    !warp_wait(&s.op_empty[sf], ((it / SF) & 1) ^ 1, s, P)) {
                    ok = false;
                    break;
                }
                // k past K contributes 0: x - zx is zeroed there (w - zw need not be)
                const int kleft = p.K - kb * KS;
#pragma unroll
                for (int u = 0; u < (TMT * KS / 16) / GROUP_THREADS; ++u) {
                    const int i = ct + GROUP_THREADS * u;
                    const int live = kleft - 16 * (i & 3);
                    widen_chunk(s.stx[s8] + 16 * i, s.opa[sf], i >> 2, i & 3, xoff,
                                live < 0 ? 0 : (live > 16 ? 16 : live));
                }
                if (wt) {
                    // row r of the staging = k r, chunk c = channels 16 c .. + 15: the
                    // f16 tile's row r, chunks 2c and 2c + 1 (N-major)
#pragma unroll
                    for (int u = 0; u < (C::TN * KS / 16) / GROUP_THREADS; ++u) {
                        const int i = ct + GROUP_THREADS * u;
                        widen_chunk_pairs(s.stw[s8] + 16 * i, s.opb[sf], i >> 2, i & 3, woff);
                    }
                } else {
#pragma unroll
                    for (int u = 0; u < (C::TN * KS / 16) / GROUP_THREADS; ++u) {
                        const int i = ct + GROUP_THREADS * u;
                        if (i < wchunks)
                            widen_chunk(s.stw[s8] + 16 * i, s.opb[sf], i >> 2, i & 3, woff[u]);
                    }
                }
                fence_proxy_async_smem();  // the f16 tiles, for the tensor core's reads
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&s.ld_empty[s8]);
                    mbar_arrive(&s.op_full[sf]);
                }
            }
        }
        if (!ok && lane == 0) s.abort = 1;
    } else {
        // ------------------------------------------------------ epilogue
        // Warp w drains TMEM lanes 32 (w % 4) .. + 31 (its tokens) and 64 of
        // the tile's columns (a quarter of a wide tile, all of a narrow one):
        // two 32-column groups, stored as one block of 32 tokens x 64 channels.
        griddep_wait();  // before the first global access (parameters, residual, y)
        const int ew = warp - EPI_WARP0;
        const int quad = warp & 3;  // TMEM lane quarter: tokens 32 quad .. + 31
        const int colq = ew >> 2;   // 64-column quarter of a wide tile (0 for narrow)
        uint8_t *blk = s.out[ew];
        uint32_t runs = 0;
        bool ok = true, pending = false;
        // this lane's channel's M0 / shift in each of the warp's two column
        // groups, loaded one tile ahead
        int32_t nm0[2], nsh[2];
        auto fetch = [&](int tile) {
            if (tile >= tile1) return;
            const Tile t = tile_of(s, P.count, tile);
            const Problem &p = s.prob[t.pi];
            const int chw = t.ct * C::TN + 64 * colq;
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int ch = chw + 32 * u + lane;
                const bool in = ch < p.N;
                nm0[u] = in ? __ldg(p.M0 + ch) : 0;
                nsh[u] = in ? __ldg(p.shift + ch) : 33;
            }
        };
        fetch(tile0);
        for (int tile = tile0; ok && tile < tile1; ++tile) {
            const Tile t = tile_of(s, P.count, tile);
            const Problem &p = s.prob[t.pi];
            const int chw = t.ct * C::TN + 64 * colq;  // first channel of this warp
            int32_t m0[2], sh[2];
            bool uni[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                m0[u] = nm0[u], sh[u] = nsh[u];
                const int32_t a0 = __shfl_sync(0xffffffffu, m0[u], 0);
                const int32_t s0 = __shfl_sync(0xffffffffu, sh[u], 0);
                // lanes past N hold (0, 33): uniform if every live lane agrees
                const bool live = chw + 32 * u + lane < p.N;
                uni[u] = __all_sync(0xffffffffu, !live || (m0[u] == a0 && sh[u] == s0));
            }
            fetch(tile + 1);  // the next tile's parameters, while this one runs
            const int tok0 = t.tt * TMT + quad * 32;
            const int32_t zy = p.zy;
            const bool vec = (s.flags[t.pi] & 1) != 0;
            const bool by_tma = (s.flags[t.pi] & 2) != 0;
            const bool part = (s.flags[t.pi] & 4) != 0;  // raw int32 sums of a slice of K
            const uint32_t t_lane = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(64 * colq);
            const int nruns = (t.nkb + t.kpr - 1) / t.kpr;
            const bool active = chw < p.N;  // any channel of this warp inside N
            if (active && pending) {  // the block's previous TMA store has read it
                if (lane == 0) store_wait_read0();
                __syncwarp();
            }
            if (!NARROW || nruns == 1) {
                const uint32_t b = runs % C::NF;
                if (!warp_wait(&s.f_full[b], (runs / C::NF) & 1, s, P)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                if (active) {
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        int32_t a[32];
                        {
                            uint32_t f[32];
                            tc_ld_32x32b_x32(t_lane + (uint32_t)C::TN * b + 32u * u, f);
                            tc_wait_ld();
#pragma unroll
                            for (int i = 0; i < 32; ++i)
                                a[i] = NARROW ? __float2int_rn(__uint_as_float(f[i])) : f2i_exact(f[i]);
                        }
                        if (part) {
                            store_part32(a, p, tok0 + lane, chw + 32 * u);
                            continue;
                        }
                        uint32_t w[16];
                        requant32<O16>(a, m0[u], sh[u], uni[u], zy, w);
                        stage32<O16, O16 ? 128 : 64>(blk, u, lane, w);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.f_empty[b]);  // F[b] read: the MMAs may go on
                ++runs;
            } else {
                // several runs (narrow tiles): 64 channels summed in int32
                int32_t acc[64];
#pragma unroll
                for (int i = 0; i < 64; ++i) acc[i] = 0;
                for (int r = 0; r < nruns; ++r, ++runs) {
                    const uint32_t b = runs % C::NF;
                    if (!warp_wait(&s.f_full[b], (runs / C::NF) & 1, s, P)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    if (active) {
#pragma unroll
                        for (int h = 0; h < 4; ++h) {  // four 16-column loads
                            uint32_t f[16];
                            tc_ld_32x32b_x16(t_lane + (uint32_t)C::TN * b + 16u * h, f);
                            tc_wait_ld();
#pragma unroll
                            for (int i = 0; i < 16; ++i)
                                acc[16 * h + i] += __float2int_rn(__uint_as_float(f[i]));
                        }
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&s.f_empty[b]);
                }
                if (!ok) break;
                if (active && part) {
                    store_part32(acc, p, tok0 + lane, chw);
                    store_part32(acc + 32, p, tok0 + lane, chw + 32);
                } else if (active) {
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        int32_t a[32];
#pragma unroll
                        for (int i = 0; i < 32; ++i) a[i] = acc[32 * u + i];
                        uint32_t w[16];
                        requant32<O16>(a, m0[u], sh[u], uni[u], zy, w);
                        stage32<O16, O16 ? 128 : 64>(blk, u, lane, w);
                    }
                }
            }
            if (active && !part) {
                flush_block<O16, O16 ? 128 : 64>(blk, p, &P.tmap_y[t.pi], tok0, chw, vec, by_tma, lane);
                pending = pending || by_tma;
            }
        }
        if (!ok && lane == 0) s.abort = 1;
        if (lane == 0) store_wait_read0();  // the block stays until its store has read it
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();  // MMAs done (waited above), TMEM reads done, loads landed
    if (warp == MMA_WARP) {
        tc_fence_after();
        tmem_dealloc1(tmem, TMEM_COLS);
    }
}

// 2-D tensor [rows][cols] of `esize`-byte elements (row pitch `pitch`
// bytes), box box_cols x box_rows.
bool encode(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows, uint64_t pitch,
            uint32_t box_cols, uint32_t box_rows, int esize, CUtensorMapSwizzle swz) {
    auto fn = prefill::encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {pitch};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    const auto type = esize == 2 ? CU_TENSOR_MAP_DATA_TYPE_UINT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8;
    return fn(map, type, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Stages per exact f32 run: the largest |x - zx| |w - zw| bounds every
// product (x in [-128, 127]; w - zw in [-255, 255] with a per-channel zero
// point, else w in [-128, 127]); the run keeps its partial sums below
// 2^run_bits: 2^22 inside the range of f2i_exact (wide tiles), 2^24 f32's
// exact integers (narrow tiles, converted by cvt).
int run_stages(const Problem &p, int run_bits) {
    const int64_t ax = p.zx >= 0 ? 128 + p.zx : 127 - p.zx;
    const int64_t aw = p.zw ? 255 : 128;
    int64_t len = (((int64_t)1 << run_bits) - 1) / (ax * aw);
    len = len / KS;
    return len < 1 ? 1 : (int)len;
}

}  // namespace tmajor

bool tmajor_suits(const Problem &p) {
    const auto a16 = [](const void *q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    return p.K > 0 && p.bits == 8 && !p.a16 && a16(p.x) && a16(p.w) && p.ldx % 16 == 0 &&
           p.ldw % 16 == 0 && !(p.o16 && p.residual);
}

namespace tmajor {

// One launch of up to PREFILL_MAX_PROBLEMS problems of one tile shape.
template <bool NARROW>
int launch_group(const Problem *const *probs, const bool *part, const bool *wt, int n, bool o16,
                 int sms, cudaStream_t stream) {
    const auto al16 = [](const void *v) { return (reinterpret_cast<uintptr_t>(v) & 15u) == 0; };
    const int osz = o16 ? 2 : 1;
    Params P{};
    long long tiles = 0;
    for (int i = 0; i < n; ++i) {
        Problem &q = P.p[i];
        q = *probs[i];
        P.kpr[i] = run_stages(q, Cfg<NARROW>::RUN_BITS);
        P.tn[i] = Cfg<NARROW>::TN;
        q.tiles_m = (q.M + TMT - 1) / TMT;
        q.tile_begin = (int)tiles;
        tiles += (long long)q.tiles_m * ((q.N + P.tn[i] - 1) / P.tn[i]);
        P.wt[i] = NARROW && wt[i] ? 1 : 0;
        if (!NARROW && wt[i]) return MQ_ERR_UNSUPPORTED_SHAPE;
        const bool wmap = P.wt[i] ? encode(&P.tmap_w[i], q.w, (uint64_t)q.N, (uint64_t)q.K,
                                           (uint64_t)q.ldw, (uint32_t)P.tn[i], KS, 1,
                                           CU_TENSOR_MAP_SWIZZLE_NONE)
                                  : encode(&P.tmap_w[i], q.w, (uint64_t)q.K, (uint64_t)q.N,
                                           (uint64_t)q.ldw, KS, (uint32_t)P.tn[i], 1,
                                           CU_TENSOR_MAP_SWIZZLE_NONE);
        if (!encode(&P.tmap_x[i], q.x, (uint64_t)q.K, (uint64_t)q.M, (uint64_t)q.ldx, KS, TMT, 1,
                    CU_TENSOR_MAP_SWIZZLE_NONE) ||
            !wmap)
            return MQ_ERR_CUDA;
        // 16-byte stores where y's rows (and the residual's) allow them;
        // without a residual, TMA stores of blocks of 32 tokens x 64 channels
        // (rows of 128 or 64 bytes, swizzled to match)
        P.vec[i] = al16(q.y) && ((size_t)q.ldy * osz) % 16 == 0 &&
                   (!q.residual || al16(q.residual));
        P.part[i] = part[i] ? 1 : 0;
        // a TMA store clips the box at the tensor's edge only in whole 16-byte
        // chunks of the inner dimension, so it serves rows of 16-byte multiples
        P.tma_y[i] = P.vec[i] && !q.residual && !part[i] && ((size_t)q.N * osz) % 16 == 0;
        if (P.tma_y[i] &&
            !encode(&P.tmap_y[i], q.y, (uint64_t)q.N, (uint64_t)q.M, (uint64_t)q.ldy * osz, 64, 32,
                    osz, o16 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B))
            return MQ_ERR_CUDA;
    }
    if (tiles == 0) return MQ_OK;
    if (tiles > 0x7fffffffLL) return MQ_ERR_UNSUPPORTED_SHAPE;
    P.count = n;
    P.total_tiles = (int)tiles;
    P.status = device_status_ptr();
    P.wait_ns = wait_limit_ns();
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3((unsigned)(tiles < sms ? tiles : sms), 1, 1);
    cfg.blockDim = dim3(Cfg<NARROW>::THREADS, 1, 1);
    cfg.dynamicSmemBytes = smem_bytes<NARROW>();
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = o16 ? cudaLaunchKernelEx(&cfg, tmajor_kernel<true, NARROW>, P)
                              : cudaLaunchKernelEx(&cfg, tmajor_kernel<false, NARROW>, P);
    return e == cudaSuccess ? MQ_OK : MQ_ERR_CUDA;
}

}  // namespace tmajor

int launch_tmajor(const Problem *probs, int count, void *stream, const uint8_t *part,
                  const uint8_t *wt) {
    using namespace tmajor;
    static std::atomic<uint64_t> attr_done{0};  // bit d: device d prepared
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return MQ_ERR_CUDA;
    if (!(attr_done.load(std::memory_order_acquire) & (1ull << dev))) {
        const auto attr = cudaFuncAttributeMaxDynamicSharedMemorySize;
        const int sw = (int)smem_bytes<false>(), sn = (int)smem_bytes<true>();
        if (cudaFuncSetAttribute(tmajor_kernel<false, false>, attr, sw) != cudaSuccess ||
            cudaFuncSetAttribute(tmajor_kernel<true, false>, attr, sw) != cudaSuccess ||
            cudaFuncSetAttribute(tmajor_kernel<false, true>, attr, sn) != cudaSuccess ||
            cudaFuncSetAttribute(tmajor_kernel<true, true>, attr, sn) != cudaSuccess)
            return MQ_ERR_CUDA;
        attr_done.fetch_or(1ull << dev, std::memory_order_release);
    }
    if (count <= 0) return MQ_OK;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MQ_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const bool o16 = probs[0].o16 != 0;
    // wide tiles where K fits one exact run and N > 64, narrow ones otherwise
    // (and for transposed weights)
    for (int narrow = 0; narrow < 2; ++narrow) {
        const Problem *list[PREFILL_MAX_PROBLEMS];
        bool lpart[PREFILL_MAX_PROBLEMS], lwt[PREFILL_MAX_PROBLEMS];
        int n = 0;
        for (int i = 0; i <= count; ++i) {
            if (i < count) {
                const Problem &q = probs[i];
                const bool t = wt && wt[i];
                const bool wide = !t && (q.K + KS - 1) / KS <= run_stages(q, 22) && q.N > TNN;
                if (wide == (narrow == 0)) {
                    lpart[n] = part && part[i];
                    lwt[n] = t;
                    list[n++] = &q;
                }
            }
            if (n == PREFILL_MAX_PROBLEMS || (i == count && n > 0)) {
                const int rc = narrow ? launch_group<true>(list, lpart, lwt, n, o16, sms, st)
                                      : launch_group<false>(list, lpart, lwt, n, o16, sms, st);
                if (rc != MQ_OK) return rc;
                n = 0;
            }
        }
    }
    return MQ_OK;
}

namespace tmajor {

constexpr int REDUCE_THREADS = 256;

struct ReduceParams {
    ReduceJob job[REDUCE_MAX_JOBS];
    int block_begin[REDUCE_MAX_JOBS + 1];
    int count;
};

// y = requant(sum over the S slices of the int32 partial sums) (+ residual):
// one thread per four consecutive outputs of a row.  The partial sums come
// from the previous kernel in the stream, so nothing is read before
// griddep_wait.
template <bool O16>
__global__ void __launch_bounds__(REDUCE_THREADS) reduce_kernel(const __grid_constant__ ReduceParams R) {
    griddep_wait();
    griddep_launch_dependents();
    int j = 0;
    while (j + 1 < R.count && (int)blockIdx.x >= R.block_begin[j + 1]) ++j;
    const ReduceJob &q = R.job[j];
    const int quads = (q.N + 3) >> 2;  // four-channel groups of a row
    const int64_t e = (int64_t)(blockIdx.x - R.block_begin[j]) * REDUCE_THREADS + threadIdx.x;
    if (e >= (int64_t)q.M * quads) return;
    const int m = (int)(e / quads), n0 = 4 * (int)(e % quads);
    const size_t slice = (size_t)q.M * (size_t)q.N;
    const int32_t *src = q.part + (size_t)m * (size_t)q.N + n0;
    int32_t acc[4] = {0, 0, 0, 0};
    const bool vec = (q.N & 3) == 0 && n0 + 4 <= q.N;
    for (int s = 0; s < q.S; ++s, src += slice) {
        if (vec) {
            const int4 v = __ldcg(reinterpret_cast<const int4 *>(src));
            acc[0] += v.x, acc[1] += v.y, acc[2] += v.z, acc[3] += v.w;
        } else {
            for (int c = 0; c < 4; ++c)
                if (n0 + c < q.N) acc[c] += __ldcg(src + c);
        }
    }
    const size_t row = (size_t)m * (size_t)q.ldy;
    for (int c = 0; c < 4; ++c) {
        const int n = n0 + c;
        if (n >= q.N) break;
        const int32_t m0 = __ldg(q.M0 + n), sh = __ldg(q.shift + n);
        if (O16) {
            reinterpret_cast<int16_t *>(q.y)[row + n] =
                (int16_t)mq_requant16((int64_t)acc[c], m0, sh, q.zy);
        } else {
            int32_t o = mq_requant(acc[c], m0, sh, q.zy);
            if (q.residual) o = min(127, max(-128, o + (int32_t)q.residual[row + n]));
            reinterpret_cast<int8_t *>(q.y)[row + n] = (int8_t)o;
        }
    }
}

}  // namespace tmajor

int launch_splitk_reduce(const ReduceJob *jobs, int count, void *stream) {
    using namespace tmajor;
    for (int base = 0; base < count; base += REDUCE_MAX_JOBS) {
        const int n = count - base < REDUCE_MAX_JOBS ? count - base : REDUCE_MAX_JOBS;
        for (int o = 0; o < 2; ++o) {  // int8, then int16 outputs
            ReduceParams R{};
            int64_t blocks = 0;
            int c = 0;
            for (int i = 0; i < n; ++i) {
                const ReduceJob &q = jobs[base + i];
                if ((q.o16 != 0) != (o == 1) || q.M <= 0 || q.N <= 0) continue;
                R.job[c] = q;
                R.block_begin[c] = (int)blocks;
                blocks += ((int64_t)q.M * ((q.N + 3) / 4) + REDUCE_THREADS - 1) / REDUCE_THREADS;
                ++c;
            }
            if (c == 0) continue;
            if (blocks > 0x7fffffffLL) return MQ_ERR_UNSUPPORTED_SHAPE;
            R.block_begin[c] = (int)blocks;
            R.count = c;
            cudaLaunchConfig_t cfg{};
            cfg.gridDim = dim3((unsigned)blocks, 1, 1);
            cfg.blockDim = dim3(REDUCE_THREADS, 1, 1);
            cfg.stream = static_cast<cudaStream_t>(stream);
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
            attr[0].val.programmaticStreamSerializationAllowed = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            const cudaError_t e = o ? cudaLaunchKernelEx(&cfg, reduce_kernel<true>, R)
                                    : cudaLaunchKernelEx(&cfg, reduce_kernel<false>, R);
            if (e != cudaSuccess) return MQ_ERR_CUDA;
        }
    }
    return MQ_OK;
}

}  // namespace mq
