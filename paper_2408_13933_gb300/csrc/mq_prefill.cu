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
// 2^10); after each chunk the epilogue warps convert the f32 chunk sum to
// int32 and add it to an int32 running sum kept in tensor memory.
//
// CTA = one SM, persistent over 128 x 256 output tiles of up to
// PREFILL_MAX_PROBLEMS independent linears.  Warp roles:
//   warps 0-7  : converters.  Load int8/int4 tiles from global memory into
//                registers (prefetching the next stage), widen to f16 and
//                store into a 4-stage ring of 128-byte-swizzled K-major tiles.
//   warp 8     : allocates tensor memory; lane 0 issues tcgen05.mma
//                (M=128, N=256, K=16, f16 x f16 -> f32) into the chunk
//                accumulator F (TMEM columns 0-255).
//   warps 9-16 : epilogue.  Per chunk: F -> int32, T += F (TMEM columns
//                256-511).  Per tile: acc = T - zx*colsum[n], fixed-point
//                requant (round half up), saturate, optional residual, store.
// All waits are bounded (mq_wait_parity).
#include <cuda_runtime.h>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {
namespace prefill {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;  // one 128-byte f16 row segment per stage
constexpr int STAGES = 4;
constexpr int CONV_WARPS = 8;
constexpr int MMA_WARP = 8;
constexpr int EPI_WARP0 = 9;
constexpr int EPI_WARPS = 8;
constexpr int NUM_WARPS = 17;
constexpr int THREADS = NUM_WARPS * 32;
constexpr int A_STAGE = BM * 128;
constexpr int B_STAGE = BN * 128;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t F_COL = 0;
constexpr uint32_t T_COL = 256;
constexpr int KB_PER_CHUNK_I8 = 1024 / BK;   // |partial| <= 1024 * 2^14 = 2^24
constexpr int KB_PER_CHUNK_I4 = 16384 / BK;  // |partial| <= 16384 * 2^10 = 2^24

struct Params {
    Problem p[PREFILL_MAX_PROBLEMS];
    int count;
    int total_tiles;
    int *status;
};

struct Smem {
    uint8_t a[STAGES][A_STAGE];
    uint8_t b[STAGES][B_STAGE];
    uint64_t full[STAGES];
    uint64_t empty[STAGES];
    uint64_t f_full;
    uint64_t f_empty;
    uint64_t done;
    uint32_t tmem_base;
    int abort;
};

constexpr size_t SMEM_BYTES = sizeof(Smem) + 1024;  // + alignment slack

struct Tile {
    const Problem *p;
    int mt, nt, nkb, kpc;
};

__device__ __forceinline__ Tile tile_at(const Params &P, int tile) {
    int pi = 0;
    while (pi + 1 < P.count && tile >= P.p[pi + 1].tile_begin) ++pi;
    Tile t;
    t.p = &P.p[pi];
    const int local = tile - t.p->tile_begin;
    t.mt = local % t.p->tiles_m;
    t.nt = local / t.p->tiles_m;
    t.nkb = (t.p->K + BK - 1) / BK;
    t.kpc = t.p->bits == 8 ? KB_PER_CHUNK_I8 : KB_PER_CHUNK_I4;
    return t;
}

// Warp-uniform bounded wait: lane 0 polls, the verdict is broadcast.
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, Smem &s, int *status) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0) ok = mq_wait_parity(bar, parity, &s.abort, status);
    return __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
}

// Byte offset of 16-byte chunk `c` (0..7) of row `r` in a 128B-swizzled tile.
__device__ __forceinline__ uint32_t swz(int r, int c) {
    return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4));
}

__device__ __forceinline__ uint4 ldg16(const void *p) {
    uint4 v;
    asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

__device__ __forceinline__ void sts16(uint8_t *base, uint32_t off, uint32_t a, uint32_t b,
                                      uint32_t c, uint32_t d) {
    *reinterpret_cast<uint4 *>(base + off) = make_uint4(a, b, c, d);
}

// Registers holding one stage's worth of this converter thread's loads.
struct StageRegs {
    uint4 a[2];
    uint4 b[4];
};

__device__ __forceinline__ void load_stage(const Tile &t, int kb, int ct, StageRegs &r) {
    const Problem &p = *t.p;
    const int k0 = kb * BK;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int g = ct + 256 * i;
        const int row = t.mt * BM + (g >> 2);
        const int k = k0 + (g & 3) * 16;
        r.a[i] = (row < p.M && k < p.K)
                     ? ldg16(p.x + (size_t)row * (size_t)p.ldx + (size_t)k)
                     : make_uint4(0, 0, 0, 0);
    }
    if (p.bits == 8) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int g = ct + 256 * i;
            const int n = t.nt * BN + (g >> 2);
            const int k = k0 + (g & 3) * 16;
            r.b[i] = (n < p.N && k < p.K) ? ldg16(p.w + (size_t)n * (size_t)p.K + (size_t)k)
                                          : make_uint4(0, 0, 0, 0);
        }
    } else {
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int g = ct + 256 * i;
            const int n = t.nt * BN + (g >> 1);
            const int k = k0 + (g & 1) * 32;
            r.b[i] = (n < p.N && k < p.K)
                         ? ldg16(p.w + (size_t)n * (size_t)(p.K / 2) + (size_t)(k / 2))
                         : make_uint4(0, 0, 0, 0);
        }
        r.b[2] = r.b[3] = make_uint4(0, 0, 0, 0);
    }
}

// 16 int8 (k = 16*kc .. 16*kc+15 of tile row `row`) -> two swizzled f16 chunks.
__device__ __forceinline__ void store_i8x16(uint8_t *tile, int row, int kc, const uint4 &v) {
    uint32_t h[8];
    i8x4_to_f16x4(v.x, h[0], h[1]);
    i8x4_to_f16x4(v.y, h[2], h[3]);
    i8x4_to_f16x4(v.z, h[4], h[5]);
    i8x4_to_f16x4(v.w, h[6], h[7]);
    sts16(tile, swz(row, 2 * kc), h[0], h[1], h[2], h[3]);
    sts16(tile, swz(row, 2 * kc + 1), h[4], h[5], h[6], h[7]);
}

// 32 int4 (k = 32*half .. 32*half+31) -> four swizzled f16 chunks.
__device__ __forceinline__ void store_i4x32(uint8_t *tile, int row, int half, const uint4 &v) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        uint32_t o[4];
        i4x8_to_f16x8(w[j], o);
        sts16(tile, swz(row, 4 * half + j), o[0], o[1], o[2], o[3]);
    }
}

__device__ __forceinline__ void convert_stage(const Tile &t, int ct, const StageRegs &r,
                                              uint8_t *a_tile, uint8_t *b_tile) {
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int g = ct + 256 * i;
        store_i8x16(a_tile, g >> 2, g & 3, r.a[i]);
    }
    if (t.p->bits == 8) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int g = ct + 256 * i;
            store_i8x16(b_tile, g >> 2, g & 3, r.b[i]);
        }
    } else {
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int g = ct + 256 * i;
            store_i4x32(b_tile, g >> 1, g & 1, r.b[i]);
        }
    }
}

// Advance (tile, kb) to the next stage position of this CTA.
__device__ __forceinline__ bool next_pos(const Params &P, int &tile, int &kb, Tile &t) {
    ++kb;
    while (tile < P.total_tiles) {
        if (kb < t.nkb) return true;
        tile += gridDim.x;
        kb = 0;
        if (tile < P.total_tiles) t = tile_at(P, tile);
    }
    return false;
}

__device__ __forceinline__ int8_t sat8(int64_t v) {
    return (int8_t)(v < -128 ? -128 : (v > 127 ? 127 : v));
}

// Requantize and store 32 consecutive outputs (columns n0 .. n0+31 of `row`).
__device__ __forceinline__ void requant_store32(const Problem &p, int row, int n0,
                                                const uint32_t (&acc)[32]) {
    if (row >= p.M) return;
    uint32_t packed[8];
    const int8_t *res = p.residual ? p.residual + (size_t)row * (size_t)p.ldy : nullptr;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        const int n = n0 + i;
        int8_t out = 0;
        if (n < p.N) {
            const int32_t cs = __ldg(p.colsum + n);
            const int32_t m0 = __ldg(p.M0 + n);
            const int32_t sh = __ldg(p.shift + n);
            // acc = sum(x w) - zx * colsum (two's-complement wrap is exact: the
            // true value fits in int32 for K <= MQ_MAX_K)
            const int32_t a = (int32_t)(acc[i] - (uint32_t)(p.zx * cs));
            const int64_t v = (int64_t)a * (int64_t)m0;
            const int64_t q = (v + ((int64_t)1 << (sh - 1))) >> sh;
            int64_t yv = (int64_t)p.zy + q;
            yv = yv < -128 ? -128 : (yv > 127 ? 127 : yv);
            if (res) yv = yv + (int64_t)res[n];
            out = sat8(yv);
        }
        const int sh8 = (i & 3) * 8;
        if ((i & 3) == 0) packed[i >> 2] = 0;
        packed[i >> 2] |= ((uint32_t)(uint8_t)out) << sh8;
    }
    int8_t *dst = p.y + (size_t)row * (size_t)p.ldy + n0;
    if (n0 + 32 <= p.N && ((reinterpret_cast<uintptr_t>(dst) & 15) == 0)) {
        reinterpret_cast<uint4 *>(dst)[0] = make_uint4(packed[0], packed[1], packed[2], packed[3]);
        reinterpret_cast<uint4 *>(dst)[1] = make_uint4(packed[4], packed[5], packed[6], packed[7]);
    } else {
#pragma unroll
        for (int i = 0; i < 32; ++i)
            if (n0 + i < p.N) dst[i] = (int8_t)((packed[i >> 2] >> ((i & 3) * 8)) & 0xFF);
    }
}

__global__ void __launch_bounds__(THREADS, 1) prefill_kernel(const __grid_constant__ Params P) {
    extern __shared__ uint8_t smem_raw[];
    Smem &s = *reinterpret_cast<Smem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(&s.full[i], CONV_WARPS);
            mbar_init(&s.empty[i], 1);
        }
        mbar_init(&s.f_full, 1);
        mbar_init(&s.f_empty, EPI_WARPS);
        mbar_init(&s.done, 1);
        s.abort = 0;
        fence_mbar_init();
    }
    if (warp == MMA_WARP) {
        tmem_alloc(&s.tmem_base, TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s.tmem_base;

    if (warp < CONV_WARPS) {
        // ------------------------------------------------------ converters
        const int ct = threadIdx.x;  // 0..255
        int tile = blockIdx.x, kb = -1;
        Tile t{};
        if (tile < P.total_tiles) t = tile_at(P, tile);
        bool have = next_pos(P, tile, kb, t);
        StageRegs cur, nxt;
        if (have) load_stage(t, kb, ct, nxt);
        uint32_t it = 0;
        while (have) {
            cur = nxt;
            const Tile tc = t;
            int ntile = tile, nkb = kb;
            Tile nt_ = t;
            const bool more = next_pos(P, ntile, nkb, nt_);
            if (more) load_stage(nt_, nkb, ct, nxt);  // prefetch the next stage
            const int stage = it % STAGES;
            if (!warp_wait(&s.empty[stage], ((it / STAGES) & 1) ^ 1, s, P.status)) break;
            convert_stage(tc, ct, cur, s.a[stage], s.b[stage]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.full[stage]);
            ++it;
            tile = ntile;
            kb = nkb;
            t = nt_;
            have = more;
        }
    } else if (warp == MMA_WARP) {
        // ------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_f16_f32(BM, BN);
            uint32_t it = 0, chunks = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < P.total_tiles; tile += gridDim.x) {
                const Tile t = tile_at(P, tile);
                for (int kb = 0; kb < t.nkb; ++kb) {
                    const bool chunk_start = (kb % t.kpc) == 0;
                    if (chunk_start) {
                        if (!mq_wait_parity(&s.f_empty, (chunks & 1) ^ 1, &s.abort, P.status)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                    }
                    const int stage = it % STAGES;
                    if (!mq_wait_parity(&s.full[stage], (it / STAGES) & 1, &s.abort, P.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t ad = smem_desc_sw128(smem_u32(s.a[stage]));
                    const uint64_t bd = smem_desc_sw128(smem_u32(s.b[stage]));
#pragma unroll
                    for (int j = 0; j < BK / 16; ++j) {
                        // +32 bytes along K per step: +2 in the (addr >> 4) field
                        tc_mma_f16(tmem + F_COL, ad + 2 * j, bd + 2 * j, idesc,
                                   (chunk_start && j == 0) ? 0u : 1u);
                    }
                    tc_commit(&s.empty[stage]);
                    ++it;
                    if (((kb + 1) % t.kpc) == 0 || kb + 1 == t.nkb) {
                        tc_commit(&s.f_full);
                        ++chunks;
                    }
                }
            }
            // every MMA issued above has completed once `done` fires
            tc_commit(&s.done);
            mq_wait_parity(&s.done, 0, &s.abort, P.status);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------ epilogue
        const int ew = warp - EPI_WARP0;     // 0..7
        const int quad = warp & 3;           // TMEM lane quadrant this warp may access
        const int col0 = (ew >> 2) * 128;    // column half of the tile
        const uint32_t t_lane = tmem + ((uint32_t)(quad * 32) << 16);
        uint32_t chunks = 0;
        bool ok = true;
        for (int tile = blockIdx.x; ok && tile < P.total_tiles; tile += gridDim.x) {
            const Tile t = tile_at(P, tile);
            const int nchunks = t.nkb ? (t.nkb + t.kpc - 1) / t.kpc : 0;
            for (int c = 0; c < nchunks; ++c) {
                if (!warp_wait(&s.f_full, chunks & 1, s, P.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
#pragma unroll 1
                for (int sl = 0; sl < 4; ++sl) {
                    const uint32_t col = (uint32_t)(col0 + sl * 32);
                    uint32_t f[32], acc[32];
                    tc_ld_32x32b_x32(t_lane + F_COL + col, f);
                    if (c > 0) tc_ld_32x32b_x32(t_lane + T_COL + col, acc);
                    tc_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const int32_t part = __float2int_rn(__uint_as_float(f[i]));
                        acc[i] = (c > 0 ? acc[i] : 0u) + (uint32_t)part;
                    }
                    tc_st_32x32b_x32(t_lane + T_COL + col, acc);
                }
                tc_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.f_empty);
                ++chunks;
            }
            if (!ok) break;
            const int row = t.mt * BM + quad * 32 + lane;
#pragma unroll 1
            for (int sl = 0; sl < 4; ++sl) {
                const uint32_t col = (uint32_t)(col0 + sl * 32);
                uint32_t acc[32];
                if (nchunks > 0) {
                    tc_ld_32x32b_x32(t_lane + T_COL + col, acc);
                    tc_wait_ld();
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) acc[i] = 0u;
                }
                requant_store32(*t.p, row, t.nt * BN + (int)col, acc);
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == MMA_WARP) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

}  // namespace prefill

int launch_prefill(const Problem *probs, int count, void *stream) {
    using namespace prefill;
    static int attr_done = -1;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return MQ_ERR_CUDA;
    if (attr_done != dev) {
        if (cudaFuncSetAttribute(prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)SMEM_BYTES) != cudaSuccess)
            return MQ_ERR_CUDA;
        attr_done = dev;
    }
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MQ_ERR_CUDA;
    for (int begin = 0; begin < count; begin += PREFILL_MAX_PROBLEMS) {
        const int n = count - begin < PREFILL_MAX_PROBLEMS ? count - begin : PREFILL_MAX_PROBLEMS;
        Params P{};
        int tiles = 0;
        for (int i = 0; i < n; ++i) {
            P.p[i] = probs[begin + i];
            P.p[i].tiles_m = (P.p[i].M + BM - 1) / BM;
            P.p[i].tile_begin = tiles;
            tiles += P.p[i].tiles_m * ((P.p[i].N + BN - 1) / BN);
        }
        P.count = n;
        P.total_tiles = tiles;
        P.status = device_status_ptr();
        if (tiles == 0) continue;
        const int grid = tiles < sms ? tiles : sms;
        prefill_kernel<<<grid, THREADS, SMEM_BYTES, static_cast<cudaStream_t>(stream)>>>(P);
        if (cudaGetLastError() != cudaSuccess) return MQ_ERR_CUDA;
    }
    return MQ_OK;
}

}  // namespace mq
