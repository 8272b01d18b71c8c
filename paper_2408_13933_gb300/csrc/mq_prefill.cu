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
// PREFILL_MAX_PROBLEMS independent linears (longest K first).  Data path:
//   HBM/L2 --TMA--> int8/int4 staging ring (3 stages, zero-filled outside the
//   tensors) --converter warps--> f16 operand ring (3 stages, 128-byte
//   swizzled, K-major) --tcgen05.mma--> f32 chunk accumulator F in TMEM.
// Warp roles:
//   warp 0     : TMA producer (one thread).
//   warp 1     : owns the TMEM allocation; one thread issues tcgen05.mma
//                (M=128, N=256, K=16, f16 x f16 -> f32) and the commits.
//   warps 2-9  : converters, int8/int4 staging -> exact f16 operand tiles;
//                every thread converts the same chunks of every stage, so
//                its shared-memory offsets are computed once.
//   warps 10-17: epilogue.  Per chunk: F -> int32, T += F (TMEM columns
//                256-511).  Per tile: acc = T - zx*colsum[n], fixed-point
//                requant (round half up) with per-column parameters staged in
//                shared memory, saturate, optional residual, store.
// All mbarrier waits are bounded (mq_wait_parity).
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {
namespace prefill {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;   // k per stage: one 128-byte f16 row segment
constexpr int S8 = 3;    // int8 staging stages
constexpr int SF = 3;    // f16 operand stages
constexpr int TMA_WARP = 0;
constexpr int MMA_WARP = 1;
constexpr int CONV_WARP0 = 2;
constexpr int CONV_WARPS = 8;
constexpr int CONV_THREADS = CONV_WARPS * 32;
constexpr int EPI_WARP0 = 10;
constexpr int EPI_WARPS = 8;
constexpr int NUM_WARPS = 18;
constexpr int THREADS = NUM_WARPS * 32;
constexpr int EPI_BARRIER = 1;  // named barrier among the epilogue warps
constexpr int OPA = BM * 128;   // f16 A tile bytes
constexpr int OPB = BN * 128;   // f16 B tile bytes
constexpr int STA = BM * BK;    // int8 A staging bytes
constexpr int STB = BN * BK;    // int8 B staging bytes (int4 uses half)
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t F_COL = 0;
constexpr uint32_t T_COL = 256;
constexpr int KB_PER_CHUNK_I8 = 1024 / BK;   // |partial| <= 1024 * 2^14 = 2^24
constexpr int KB_PER_CHUNK_I4 = 16384 / BK;  // |partial| <= 16384 * 2^10 = 2^24

struct Params {
    CUtensorMap tmap_x[PREFILL_MAX_PROBLEMS];  // int8 [M][ldx], box 64 x 128
    CUtensorMap tmap_w[PREFILL_MAX_PROBLEMS];  // int8 [N][K] box 64 x 256, or int4 bytes 32 x 256
    Problem p[PREFILL_MAX_PROBLEMS];
    int count;
    int total_tiles;
    int *status;
};

struct Smem {
    uint8_t opa[SF][OPA];
    uint8_t opb[SF][OPB];
    uint8_t sta[S8][STA];
    uint8_t stb[S8][STB];
    uint64_t ld_full[S8];
    uint64_t ld_empty[S8];
    uint64_t op_full[SF];
    uint64_t op_empty[SF];
    uint64_t f_full;
    uint64_t f_empty;
    uint64_t done;
    int32_t col_corr[BN];  // zx * colsum[n] of the epilogue's current tile
    int32_t col_m0[BN];
    int32_t col_shift[BN];
    uint32_t tmem_base;
    int abort;
};

constexpr size_t SMEM_BYTES = sizeof(Smem) + 1024;  // + alignment slack

struct Tile {
    int pi;
    int mt, nt, nkb, kpc;
};

__device__ __forceinline__ Tile tile_at(const Params &P, int tile) {
    Tile t;
    t.pi = 0;
    while (t.pi + 1 < P.count && tile >= P.p[t.pi + 1].tile_begin) ++t.pi;
    const Problem &p = P.p[t.pi];
    const int local = tile - p.tile_begin;
    t.mt = local % p.tiles_m;
    t.nt = local / p.tiles_m;
    t.nkb = (p.K + BK - 1) / BK;
    t.kpc = p.bits == 8 ? KB_PER_CHUNK_I8 : KB_PER_CHUNK_I4;
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

__device__ __forceinline__ void sts16(uint8_t *base, uint32_t off, uint32_t a, uint32_t b,
                                      uint32_t c, uint32_t d) {
    *reinterpret_cast<uint4 *>(base + off) = make_uint4(a, b, c, d);
}

__device__ __forceinline__ uint4 lds16(const uint8_t *p) {
    return *reinterpret_cast<const uint4 *>(p);
}

// 16 int8 -> two f16 chunks at precomputed swizzled offsets.
__device__ __forceinline__ void cvt_i8x16(uint8_t *tile, const uint32_t (&off)[2], const uint4 &v) {
    uint32_t h[8];
    i8x4_to_f16x4(v.x, h[0], h[1]);
    i8x4_to_f16x4(v.y, h[2], h[3]);
    i8x4_to_f16x4(v.z, h[4], h[5]);
    i8x4_to_f16x4(v.w, h[6], h[7]);
    sts16(tile, off[0], h[0], h[1], h[2], h[3]);
    sts16(tile, off[1], h[4], h[5], h[6], h[7]);
}

// 32 int4 -> four f16 chunks at precomputed swizzled offsets.
__device__ __forceinline__ void cvt_i4x32(uint8_t *tile, const uint32_t (&off)[4], const uint4 &v) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        uint32_t o[4];
        i4x8_to_f16x8(w[j], o);
        sts16(tile, off[j], o[0], o[1], o[2], o[3]);
    }
}

// What the epilogue needs of the current tile's problem, in registers (the
// problem table itself lives in the kernel parameters, where dynamically
// indexed reads are slow).
struct EpiArgs {
    int8_t *y;
    const int8_t *residual;
    int M, N, ldy, zy;
};

// Requantize and store 16 consecutive outputs (tile columns c0 .. c0+15 of
// `row`; global column = n0 + tile column).
__device__ __forceinline__ void requant_store16(const EpiArgs &e, const Smem &s, int row, int n0,
                                                int c0, const uint32_t (&acc)[16]) {
    if (row >= e.M) return;
    const int8_t *res = e.residual ? e.residual + (size_t)row * (size_t)e.ldy + n0 + c0 : nullptr;
    uint32_t packed[4];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const int c = c0 + i;
        int32_t out = mq_requant((int32_t)(acc[i] - (uint32_t)s.col_corr[c]), s.col_m0[c],
                                 s.col_shift[c], e.zy);
        if (res && n0 + c < e.N) out = min(127, max(-128, out + (int32_t)res[i]));
        if ((i & 3) == 0) packed[i >> 2] = 0;
        packed[i >> 2] |= ((uint32_t)(out & 0xFF)) << ((i & 3) * 8);
    }
    int8_t *dst = e.y + (size_t)row * (size_t)e.ldy + n0 + c0;
    if (n0 + c0 + 16 <= e.N && ((reinterpret_cast<uintptr_t>(dst) & 15) == 0)) {
        *reinterpret_cast<uint4 *>(dst) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
    } else {
#pragma unroll
        for (int i = 0; i < 16; ++i)
            if (n0 + c0 + i < e.N) dst[i] = (int8_t)((packed[i >> 2] >> ((i & 3) * 8)) & 0xFF);
    }
}

__device__ __forceinline__ void epi_sync() {
    asm volatile("bar.sync %0, %1;" ::"n"(EPI_BARRIER), "n"(EPI_WARPS * 32) : "memory");
}

__global__ void __launch_bounds__(THREADS, 1) prefill_kernel(const __grid_constant__ Params P) {
    extern __shared__ uint8_t smem_raw[];
    Smem &s = *reinterpret_cast<Smem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < S8; ++i) {
            mbar_init(&s.ld_full[i], 1);
            mbar_init(&s.ld_empty[i], CONV_WARPS);
        }
        for (int i = 0; i < SF; ++i) {
            mbar_init(&s.op_full[i], CONV_WARPS);
            mbar_init(&s.op_empty[i], 1);
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

    if (warp == TMA_WARP) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            for (int i = 0; i < P.count; ++i) {
                if (P.p[i].K == 0) continue;  // no map was encoded
                prefetch_tensormap(&P.tmap_x[i]);
                prefetch_tensormap(&P.tmap_w[i]);
            }
            uint32_t it = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < P.total_tiles; tile += gridDim.x) {
                const Tile t = tile_at(P, tile);
                const bool i4 = P.p[t.pi].bits == 4;
                const uint32_t bytes = STA + (i4 ? STB / 2 : STB);
                for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                    const int slot = it % S8;
                    if (!mq_wait_parity(&s.ld_empty[slot], ((it / S8) & 1) ^ 1, &s.abort,
                                        P.status)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&s.ld_full[slot], bytes);
                    tma_load_2d(s.sta[slot], &P.tmap_x[t.pi], kb * BK, t.mt * BM, &s.ld_full[slot]);
                    tma_load_2d(s.stb[slot], &P.tmap_w[t.pi], i4 ? kb * (BK / 2) : kb * BK,
                                t.nt * BN, &s.ld_full[slot]);
                }
            }
        }
        __syncwarp();
    } else if (warp == MMA_WARP) {
        // ------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_f16_f32(BM, BN);
            uint32_t it = 0, chunks = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < P.total_tiles; tile += gridDim.x) {
                const Tile t = tile_at(P, tile);
                for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                    const bool chunk_start = (kb % t.kpc) == 0;
                    if (chunk_start) {
                        if (!mq_wait_parity(&s.f_empty, (chunks & 1) ^ 1, &s.abort, P.status)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                    }
                    const int slot = it % SF;
                    if (!mq_wait_parity(&s.op_full[slot], (it / SF) & 1, &s.abort, P.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t ad = smem_desc_sw128(smem_u32(s.opa[slot]));
                    const uint64_t bd = smem_desc_sw128(smem_u32(s.opb[slot]));
#pragma unroll
                    for (int j = 0; j < BK / 16; ++j)  // +32 B along K: +2 in the (addr >> 4) field
                        tc_mma_f16(tmem + F_COL, ad + 2 * j, bd + 2 * j, idesc,
                                   (chunk_start && j == 0) ? 0u : 1u);
                    tc_commit(&s.op_empty[slot]);
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
    } else if (warp < EPI_WARP0) {
        // ------------------------------------------------------ converters
        // Thread ct converts, in every stage: A chunks ct and ct + 256 (128
        // rows x 4 chunks of 16 int8); B int8 chunks ct + 256 i, i < 4 (256
        // rows x 4), or B int4 chunks ct and ct + 256 (256 rows x 2 chunks of
        // 32 nibbles).  Chunk g of A / int8 B is row g >> 2, chunk g & 3;
        // of int4 B row g >> 1, half g & 1.
        const int ct = threadIdx.x - CONV_WARP0 * 32;  // 0..255
        uint32_t a_src[2], a_dst[2][2], b_src[4], b_dst[4][2], q_dst[2][4];
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int g = ct + 256 * i, row = g >> 2, kc = g & 3;
            a_src[i] = g * 16;
            a_dst[i][0] = swz(row, 2 * kc);
            a_dst[i][1] = swz(row, 2 * kc + 1);
            const int qrow = g >> 1, half = g & 1;
#pragma unroll
            for (int j = 0; j < 4; ++j) q_dst[i][j] = swz(qrow, 4 * half + j);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int g = ct + 256 * i, row = g >> 2, kc = g & 3;
            b_src[i] = g * 16;
            b_dst[i][0] = swz(row, 2 * kc);
            b_dst[i][1] = swz(row, 2 * kc + 1);
        }
        uint32_t it = 0;
        bool ok = true;
        for (int tile = blockIdx.x; ok && tile < P.total_tiles; tile += gridDim.x) {
            const Tile t = tile_at(P, tile);
            const bool i4 = P.p[t.pi].bits == 4;
            for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                const int s8 = it % S8, sf = it % SF;
                if (!warp_wait(&s.ld_full[s8], (it / S8) & 1, s, P.status) ||
                    !warp_wait(&s.op_empty[sf], ((it / SF) & 1) ^ 1, s, P.status)) {
                    ok = false;
                    break;
                }
                const uint8_t *sa = s.sta[s8];
                const uint8_t *sb = s.stb[s8];
                uint8_t *oa = s.opa[sf];
                uint8_t *ob = s.opb[sf];
                uint4 va[2], vb[4];
#pragma unroll
                for (int i = 0; i < 2; ++i) va[i] = lds16(sa + a_src[i]);
                if (!i4) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) vb[i] = lds16(sb + b_src[i]);
                } else {
#pragma unroll
                    for (int i = 0; i < 2; ++i) vb[i] = lds16(sb + a_src[i]);
                }
#pragma unroll
                for (int i = 0; i < 2; ++i) cvt_i8x16(oa, a_dst[i], va[i]);
                if (!i4) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) cvt_i8x16(ob, b_dst[i], vb[i]);
                } else {
#pragma unroll
                    for (int i = 0; i < 2; ++i) cvt_i4x32(ob, q_dst[i], vb[i]);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&s.op_full[sf]);
                    mbar_arrive(&s.ld_empty[s8]);
                }
            }
        }
    } else {
        // ------------------------------------------------------ epilogue
        const int et = threadIdx.x - EPI_WARP0 * 32;  // 0..255
        const int ew = warp - EPI_WARP0;              // 0..7
        const int quad = warp & 3;          // TMEM lane quadrant this warp may access
        const int col0 = (ew >> 2) * 128;   // column half of the tile
        const uint32_t t_lane = tmem + ((uint32_t)(quad * 32) << 16);
        uint32_t chunks = 0;
        // After a failed wait (ok == false) the warp keeps walking the tile
        // loop without touching TMEM, so that every epilogue warp reaches the
        // same named barriers.
        bool ok = true;
        for (int tile = blockIdx.x; tile < P.total_tiles; tile += gridDim.x) {
            const Tile t = tile_at(P, tile);
            const Problem &p = P.p[t.pi];
            const EpiArgs e{p.y, p.residual, p.M, p.N, p.ldy, p.zy};
            const int n0 = t.nt * BN;
            epi_sync();  // the previous tile's requant pass is done with the parameters
            {
                const int n = n0 + et;
                const bool in = n < e.N;
                s.col_corr[et] = in ? p.zx * __ldg(p.colsum + n) : 0;
                s.col_m0[et] = in ? __ldg(p.M0 + n) : 0;
                s.col_shift[et] = in ? __ldg(p.shift + n) : 33;
            }
            const int nchunks = t.nkb ? (t.nkb + t.kpc - 1) / t.kpc : 0;
            for (int c = 0; ok && c < nchunks; ++c) {
                if (!warp_wait(&s.f_full, chunks & 1, s, P.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                // drain F into T, one 16-column slice at a time; the TMEM
                // loads of slice sl+1 overlap the arithmetic of slice sl
                uint32_t f[2][16], acc[2][16];
                tc_ld_32x32b_x16(t_lane + F_COL + col0, f[0]);
                if (c > 0) tc_ld_32x32b_x16(t_lane + T_COL + col0, acc[0]);
                tc_wait_ld();
#pragma unroll
                for (int sl = 0; sl < 8; ++sl) {
                    const int b = sl & 1;
                    if (sl + 1 < 8) {
                        const uint32_t nc = (uint32_t)(col0 + (sl + 1) * 16);
                        tc_ld_32x32b_x16(t_lane + F_COL + nc, f[b ^ 1]);
                        if (c > 0) tc_ld_32x32b_x16(t_lane + T_COL + nc, acc[b ^ 1]);
                    }
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int32_t part = __float2int_rn(__uint_as_float(f[b][i]));
                        acc[b][i] = (c > 0 ? acc[b][i] : 0u) + (uint32_t)part;
                    }
                    tc_st_32x32b_x16(t_lane + T_COL + (uint32_t)(col0 + sl * 16), acc[b]);
                    if (sl + 1 < 8) tc_wait_ld();
                }
                tc_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.f_empty);
                ++chunks;
            }
            epi_sync();  // column parameters visible to every epilogue warp
            if (!ok) continue;
            const int row = t.mt * BM + quad * 32 + lane;
#pragma unroll 1
            for (int sl = 0; sl < 8; ++sl) {
                const int c0 = col0 + sl * 16;
                uint32_t acc[16];
                if (nchunks > 0) {
                    tc_ld_32x32b_x16(t_lane + T_COL + (uint32_t)c0, acc);
                    tc_wait_ld();
                } else {
#pragma unroll
                    for (int i = 0; i < 16; ++i) acc[i] = 0u;
                }
                requant_store16(e, s, row, n0, c0, acc);
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

// 2-D uint8 tensor [rows][cols] with row pitch `pitch` bytes, box box_cols x box_rows.
bool encode_2d(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows, uint64_t pitch,
               uint32_t box_cols, uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {pitch};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
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
        // longest K first: the longest tiles start in the first wave
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
            q.tiles_m = (q.M + BM - 1) / BM;
            q.tile_begin = tiles;
            tiles += q.tiles_m * ((q.N + BN - 1) / BN);
            if (q.K > 0) {
                const uint64_t wcols = q.bits == 8 ? (uint64_t)q.K : (uint64_t)q.K / 2;
                if (!encode_2d(&P.tmap_x[i], q.x, (uint64_t)q.K, (uint64_t)q.M, (uint64_t)q.ldx,
                               BK, BM) ||
                    !encode_2d(&P.tmap_w[i], q.w, wcols, (uint64_t)q.N, wcols,
                               q.bits == 8 ? BK : BK / 2, BN))
                    return MQ_ERR_CUDA;
            }
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
