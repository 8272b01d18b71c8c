// mq_gemv.cu -- weight-streaming kernel for the integer-only quantized linear
// layer at one or two tokens (autoregressive generation), bit-exact.
//
// At M <= 2 the layer reads every weight once and does one or two MACs with
// it: the time is the weight stream (the paper notes that autoregressive
// generation is memory-bound, Sec. 5.6 and Appendix A.2).  This kernel is
// built to stream HBM at its rate:
//
// Work.  Every problem's weight matrix is cut into row tiles of TR = 8 rows;
// a row tile is read in stages of at most CHUNK = 1024 bytes of each of its
// rows.  The row tiles of all problems of a launch form one sequence, and
// each CTA (one per SM) takes a contiguous run of it, cut by the host so that
// every CTA streams about the same number of bytes.  A row tile never spans
// two CTAs, so every output is finished by the CTA that streamed it: no
// split-K, no exchange between CTAs.
//
// Data path.  One producer warp copies each stage into a shared-memory ring
// with 1-D bulk copies (cp.async.bulk): one contiguous copy per weight row
// segment (each row lands 16 bytes past a 1024-byte pitch, which spreads the
// rows over the banks) and one per token of the matching slice of x; the
// row tile's requantization parameters ride along with its last stage as
// 4-byte cp.async copies whose completion the same mbarrier tracks.  Weight
// copies of the first ring stages are issued before waiting for the previous
// kernel in the stream (programmatic dependent launch): packed weights are
// constant inputs.
//
// Compute.  Eight consumer warps share every stage: warp w takes bytes
// [128 w, 128 w + 128) of the chunk, lane (r, p) = (lane / 4, lane % 4) the
// 32 bytes at offset 32 p of that slice of row r.  The eight lanes of a warp
// that read the same slice of x read the same addresses, which the shared
// memory broadcasts.  int4 weights: one LOP3 (and a shift for the high
// nibbles) forms u = w + 8 in [0, 15] per byte and two PRMT put the nibbles in
// k order, so that one dp4a multiplies four weights with four activation
// bytes as they are stored; int8 weights go to dp4a unchanged.  The int32
// sums are exact: |partial| <= 15 * 128 * 65536 < 2^31.
//
// Epilogue (per row tile).  Each lane's sum is reduced over its four pieces
// (two shuffles), the warps' sums over shared memory; then one thread per
// (row, token) removes the bias, sum(w x) = sum(u x) - 8 sum(x) (int4), and
// forms sum((x - zx)(w - zw)) = sum(w x) - zw sum(x) - zx (colsum - K zw),
// requantizes (round half up, saturate), adds the optional residual and
// stores.  sum(x) of each problem's tokens is accumulated while the CTA
// streams its first row tile of that problem, which covers every k.
// All mbarrier waits are bounded (mq_wait_parity).
#include <cuda_runtime.h>

#include <atomic>
#include <vector>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {
namespace gemv {

constexpr int CONS_WARPS = 8;
constexpr int CONS_THREADS = CONS_WARPS * 32;
constexpr int PROD_WARP = CONS_WARPS;
constexpr int THREADS = CONS_THREADS + 32;
constexpr int TR = 8;                     // weight rows per row tile
constexpr int CHUNK = 1024;               // weight bytes of a row per stage
constexpr int ROW_PITCH = CHUNK + 16;     // shared-memory row pitch
constexpr int W_BYTES = TR * ROW_PITCH;
constexpr int MAX_MT = 2;                 // tokens
constexpr int PARAM_BYTES = 128;          // colsum, M0, shift, zw of 8 rows
constexpr int CONS_BARRIER = 1;           // named barrier of the consumer warps
constexpr int MAX_GRID = 320;
constexpr int MAX_PROBLEMS = DECODE_MAX_PROBLEMS;
constexpr int MAX_STAGES = 24;

__host__ __device__ constexpr int x_bytes(int bits, int mt) { return mt * CHUNK * (8 / bits); }
__host__ __device__ constexpr int stage_bytes(int bits, int mt) {
    return (W_BYTES + x_bytes(bits, mt) + PARAM_BYTES + 127) / 128 * 128;
}

struct Params {
    Problem p[MAX_PROBLEMS];      // tile_begin = first global row tile, tiles_m = row tiles
    int count;
    int stages;                   // ring depth
    int pre_w;                    // 1: weights are read before griddep_wait
    int cta_begin[MAX_GRID + 1];  // each CTA's first row tile
    int *status;
    uint64_t wait_ns;
};

// What the kernel reads of a problem, kept in shared memory.
struct GProb {
    const uint8_t *w;
    const int8_t *x;
    const int32_t *colsum, *M0, *shift, *zw;
    const int8_t *residual;
    int8_t *y;
    int32_t M, N, K, ldx, ldy, ldw, zx, zy;
    int32_t tile_begin, tiles;
    int32_t L;        // weight bytes of a row
    int32_t nchunks;  // stages per row tile
};

template <int MT>
struct Tail {
    int32_t red[2][CONS_WARPS][TR][MT];  // the warps' row sums (row-tile parity)
    int32_t xsred[2][CONS_WARPS][MT];    // the warps' sum(x) pieces
    int32_t xsum[MT];                    // sum(x) of the current problem's tokens
    GProb prob[MAX_PROBLEMS];
    uint64_t full[MAX_STAGES];
    uint64_t empty[MAX_STAGES];
    int abort;
};

template <int BITS, int MT>
constexpr size_t smem_bytes(int stages) {
    return (size_t)stages * stage_bytes(BITS, MT) + sizeof(Tail<MT>) + 128;
}

__device__ __forceinline__ void cons_sync() {
    asm volatile("bar.sync %0, %1;" ::"n"(CONS_BARRIER), "n"(CONS_THREADS) : "memory");
}

__device__ __forceinline__ uint4 lds128(const uint8_t *p) {
    return *reinterpret_cast<const uint4 *>(p);
}

// The problem holding row tile `tile`, searching forward from `pi` (a CTA
// visits its tiles in increasing order, so the walk is amortized O(1)).
template <class S>
__device__ __forceinline__ int problem_from(const S &s, int count, int pi, int tile) {
    while (pi + 1 < count && tile >= s.prob[pi + 1].tile_begin) ++pi;
    return pi;
}

template <int BITS, int MT, bool O16>
__global__ void __launch_bounds__(THREADS, 2) gemv_kernel(const __grid_constant__ Params P) {
    constexpr int KPB = 8 / BITS;  // k per weight byte
    constexpr int SB = stage_bytes(BITS, MT);
    constexpr int XOFF = W_BYTES;
    constexpr int POFF = W_BYTES + x_bytes(BITS, MT);
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~static_cast<uintptr_t>(127));
    const int S = P.stages;
    Tail<MT> &s = *reinterpret_cast<Tail<MT> *>(ring + (size_t)S * SB);
    volatile int *abort_flag = &s.abort;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t_begin = P.cta_begin[blockIdx.x], t_end = P.cta_begin[blockIdx.x + 1];
    const int count = P.count;

    if (threadIdx.x == 0) {
        for (int i = 0; i < S; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], CONS_WARPS);
        }
        s.abort = 0;
        fence_mbar_init();
    }
    for (int i = threadIdx.x; i < count; i += THREADS) {
        const Problem &q = P.p[i];
        GProb g;
        g.w = q.w;
        g.x = q.x;
        g.colsum = q.colsum;
        g.M0 = q.M0;
        g.shift = q.shift;
        g.zw = q.zw;
        g.residual = q.residual;
        g.y = q.y;
        g.M = q.M;
        g.N = q.N;
        g.K = q.K;
        g.ldx = q.ldx;
        g.ldy = q.ldy;
        g.ldw = q.ldw;
        g.zx = q.zx;
        g.zy = q.zy;
        g.tile_begin = q.tile_begin;
        g.tiles = q.tiles_m;
        g.L = q.K / KPB;
        g.nchunks = (g.L + CHUNK - 1) / CHUNK;
        s.prob[i] = g;
    }
    __syncthreads();
    if (threadIdx.x == 0) griddep_launch_dependents();

    if (warp == PROD_WARP) {
        // ------------------------------------------------------ producer
        // Weight copies of the first ring stages go out before the wait for
        // the previous kernel (constant inputs unless pre_w == 0); x and the
        // parameters only after it.
        uint32_t npre = 0;
        if (lane == 0 && P.pre_w) {
            int pi = 0;
            for (int t = t_begin; t < t_end && npre < (uint32_t)S; ++t) {
                pi = problem_from(s, count, pi, t);
                const GProb &g = s.prob[pi];
                const int n0 = (t - g.tile_begin) * TR;
                const int rows = min(TR, g.N - n0);
                for (int c = 0; c < g.nchunks && npre < (uint32_t)S; ++c, ++npre) {
                    const int cb = min(CHUNK, g.L - c * CHUNK);
                    uint8_t *st = ring + (size_t)npre * SB;
                    mbar_expect_tx(&s.full[npre], (uint32_t)(rows * cb));
                    for (int r = 0; r < rows; ++r)
                        bulk_load(st + r * ROW_PITCH, g.w + (size_t)(n0 + r) * g.ldw + c * CHUNK,
                                  (uint32_t)cb, &s.full[npre]);
                }
            }
        }
        npre = __shfl_sync(0xffffffffu, npre, 0);
        griddep_wait();
        uint32_t it = 0;
        bool ok = true;
        int pi = 0;
        for (int t = t_begin; ok && t < t_end; ++t) {
            pi = problem_from(s, count, pi, t);
            const GProb &g = s.prob[pi];
            const int n0 = (t - g.tile_begin) * TR;
            const int rows = min(TR, g.N - n0);
            for (int c = 0; c < g.nchunks; ++c, ++it) {
                const int slot = it % S;
                bool got = true;
                if (lane == 0)
                    got = mq_wait_parity(&s.empty[slot], ((it / S) & 1) ^ 1, &s.abort, P.status,
                                         P.wait_ns);
                if (!__shfl_sync(0xffffffffu, got ? 1 : 0, 0)) {
                    ok = false;
                    break;
                }
                uint8_t *st = ring + (size_t)slot * SB;
                const int cb = min(CHUNK, g.L - c * CHUNK);
                if (c == g.nchunks - 1) {
                    // the row tile's parameters: lane = 8 array + row
                    const int arr = lane >> 3, r = lane & 7;
                    const int32_t *src = arr == 0 ? g.colsum : arr == 1 ? g.M0
                                       : arr == 2 ? g.shift : g.zw;
                    if (r < rows && src) cp_async4(st + POFF + lane * 4, src + n0 + r);
                    cp_async_arrive(&s.full[slot]);
                }
                __syncwarp();
                if (lane == 0) {
                    if (it >= npre) {
                        mbar_expect_tx(&s.full[slot], (uint32_t)(rows * cb));
                        for (int r = 0; r < rows; ++r)
                            bulk_load(st + r * ROW_PITCH,
                                      g.w + (size_t)(n0 + r) * g.ldw + c * CHUNK, (uint32_t)cb,
                                      &s.full[slot]);
                    }
                    mbar_arrive_expect_tx(&s.full[slot], (uint32_t)(g.M * cb * KPB));
                    for (int m = 0; m < g.M; ++m)
                        bulk_load(st + XOFF + m * CHUNK * KPB,
                                  g.x + (size_t)m * g.ldx + (size_t)c * CHUNK * KPB,
                                  (uint32_t)(cb * KPB), &s.full[slot]);
                }
            }
        }
        if (!ok && lane == 0) {
            // Given up: let the copies already issued land before the CTA can
            // leave (only the last S stages can still be in flight; stages
            // below `it` were issued whole).
            for (uint32_t i = it > (uint32_t)S ? it - S : 0u; i < it; ++i)
                mq_wait_parity_drain(&s.full[i % S], (i / S) & 1, P.status, P.wait_ns);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------ consumers
        griddep_wait();  // before the first global access (residual, y)
        const int r = lane >> 2, pc = lane & 3;
        const int off = warp * 128 + pc * 32;  // this lane's bytes within a chunk
        const int et = threadIdx.x;            // epilogue thread: row et % 8, token et / 8
        uint32_t it = 0;
        int pi = -1;
        int parity = 0;
        for (int t = t_begin; t < t_end; ++t) {
            const int npi = problem_from(s, count, pi < 0 ? 0 : pi, t);
            const bool first = npi != pi;  // first row tile of this problem in this CTA
            pi = npi;
            const GProb &g = s.prob[pi];
            const int n0 = (t - g.tile_begin) * TR;
            const int rows = min(TR, g.N - n0);
            // the residual of this thread's output, loaded now for the epilogue
            int32_t res = 0;
            if (et < TR * MT && g.residual && (et & 7) < rows && (et >> 3) < g.M)
                res = g.residual[(size_t)(et >> 3) * g.ldy + n0 + (et & 7)];
            int32_t acc[MT], xs[MT];
#pragma unroll
            for (int m = 0; m < MT; ++m) acc[m] = xs[m] = 0;
            for (int c = 0; c < g.nchunks; ++c, ++it) {
                const int slot = it % S;
                bool got = false;
                if (lane == 0)
                    got = !*abort_flag && mq_wait_parity(&s.full[slot], (it / S) & 1, &s.abort,
                                                         P.status, P.wait_ns);
                got = __shfl_sync(0xffffffffu, got ? 1 : 0, 0) != 0;
                const uint8_t *st = ring + (size_t)slot * SB;
                const int cb = min(CHUNK, g.L - c * CHUNK);
                if (got && off < cb) {
                    const uint8_t *xp = st + XOFF + off * KPB;
                    // A chunk ends on a 16-byte boundary, so the last lane's
                    // piece may hold only 16 valid bytes: the activations of
                    // the other half then read as zero (the stale weights
                    // beside them multiply nothing).
                    const bool h2 = off + 32 <= cb;
                    auto xld = [&](int m, int q) {
                        return (q < KPB || h2) ? lds128(xp + m * CHUNK * KPB + 16 * q)
                                               : make_uint4(0u, 0u, 0u, 0u);
                    };
                    if (first) {
                        // sum(x) of the slice (every k of the problem passes
                        // through the lanes of row 0 during its first tile)
#pragma unroll
                        for (int m = 0; m < MT; ++m)
#pragma unroll
                            for (int q = 0; q < 2 * KPB; ++q) {
                                const uint4 v = xld(m, q);
                                xs[m] = __dp4a((int)v.x, 0x01010101, xs[m]);
                                xs[m] = __dp4a((int)v.y, 0x01010101, xs[m]);
                                xs[m] = __dp4a((int)v.z, 0x01010101, xs[m]);
                                xs[m] = __dp4a((int)v.w, 0x01010101, xs[m]);
                            }
                    }
                    if (r < rows) {
                        const uint4 wa = lds128(st + r * ROW_PITCH + off);
                        const uint4 wb = lds128(st + r * ROW_PITCH + off + 16);
                        const uint32_t wv[8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
                        if constexpr (BITS == 4) {
                            // word j holds k = 8 j .. 8 j + 7 of the piece; lo / hi
                            // are k 8j..8j+3 / 8j+4..8j+7 as bytes u = w + 8
                            uint32_t lo[8], hi[8];
#pragma unroll
                            for (int j = 0; j < 8; ++j) {
                                const uint32_t e = (wv[j] & 0x0F0F0F0Fu) ^ 0x08080808u;
                                const uint32_t o = ((wv[j] >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
                                lo[j] = prmt(e, o, 0x5140u);
                                hi[j] = prmt(e, o, 0x7362u);
                            }
#pragma unroll
                            for (int m = 0; m < MT; ++m)
#pragma unroll
                                for (int q = 0; q < 4; ++q) {
                                    const uint4 v = xld(m, q);
                                    acc[m] = __dp4a((int)lo[2 * q], (int)v.x, acc[m]);
                                    acc[m] = __dp4a((int)hi[2 * q], (int)v.y, acc[m]);
                                    acc[m] = __dp4a((int)lo[2 * q + 1], (int)v.z, acc[m]);
                                    acc[m] = __dp4a((int)hi[2 * q + 1], (int)v.w, acc[m]);
                                }
                        } else {
#pragma unroll
                            for (int m = 0; m < MT; ++m)
#pragma unroll
                                for (int q = 0; q < 2; ++q) {
                                    const uint4 v = xld(m, q);
                                    acc[m] = __dp4a((int)wv[4 * q + 0], (int)v.x, acc[m]);
                                    acc[m] = __dp4a((int)wv[4 * q + 1], (int)v.y, acc[m]);
                                    acc[m] = __dp4a((int)wv[4 * q + 2], (int)v.z, acc[m]);
                                    acc[m] = __dp4a((int)wv[4 * q + 3], (int)v.w, acc[m]);
                                }
                        }
                    }
                }
                const bool last = c == g.nchunks - 1;
                // the last stage of a tile holds its parameters: warp 0 (the
                // epilogue's) releases it after the epilogue
                if (!(last && warp == 0)) {
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&s.empty[slot]);
                }
            }
            // ---- epilogue of the row tile
#pragma unroll
            for (int m = 0; m < MT; ++m) {
                acc[m] += __shfl_xor_sync(0xffffffffu, acc[m], 1);
                acc[m] += __shfl_xor_sync(0xffffffffu, acc[m], 2);
                if (first) {
                    xs[m] += __shfl_xor_sync(0xffffffffu, xs[m], 1);
                    xs[m] += __shfl_xor_sync(0xffffffffu, xs[m], 2);
                }
            }
            if (pc == 0) {
#pragma unroll
                for (int m = 0; m < MT; ++m) s.red[parity][warp][r][m] = acc[m];
            }
            if (first && lane == 0) {
#pragma unroll
                for (int m = 0; m < MT; ++m) s.xsred[parity][warp][m] = xs[m];
            }
            cons_sync();
            const uint32_t lslot = (it - 1) % S;  // the tile's last stage
            if (et < TR * MT) {
                const int er = et & 7, m = et >> 3;
                int32_t sum = 0, xsum;
#pragma unroll
                for (int w = 0; w < CONS_WARPS; ++w) sum += s.red[parity][w][er][m];
                if (first) {
                    xsum = 0;
#pragma unroll
                    for (int w = 0; w < CONS_WARPS; ++w) xsum += s.xsred[parity][w][m];
                } else {
                    xsum = s.xsum[m];
                }
                const int n = n0 + er;
                if (!*abort_flag && er < rows && m < g.M) {
                    const int32_t *prm =
                        reinterpret_cast<const int32_t *>(ring + (size_t)lslot * SB + POFF);
                    const int32_t colsum = prm[er], m0 = prm[8 + er], sh = prm[16 + er];
                    const int32_t zw = g.zw ? prm[24 + er] : 0;
                    // sum(w x) = sum(u x) - 8 sum(x) (int4); then the zero points:
                    // sum((x - zx)(w - zw)) = sum(w x) - zw sum(x) - zx (colsum - K zw)
                    // (two's-complement wrap is exact: the true value fits int32)
                    const uint32_t wx = (uint32_t)sum - (uint32_t)(BITS == 4 ? 8 * xsum : 0);
                    const int32_t a =
                        (int32_t)(wx - (uint32_t)zw * (uint32_t)xsum -
                                  (uint32_t)g.zx * ((uint32_t)colsum - (uint32_t)g.K * (uint32_t)zw));
                    if constexpr (O16) {
                        reinterpret_cast<int16_t *>(g.y)[(size_t)m * g.ldy + n] =
                            (int16_t)mq_requant16((int64_t)a, m0, sh, g.zy);
                    } else {
                        int32_t y = mq_requant(a, m0, sh, g.zy);
                        if (g.residual) y = min(127, max(-128, y + res));
                        g.y[(size_t)m * g.ldy + n] = (int8_t)y;
                    }
                }
                if (first && er == 0) s.xsum[m] = xsum;
            }
            if (warp == 0) {
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.empty[lslot]);
            }
            parity ^= 1;
        }
    }
    __syncthreads();
}

template <int BITS, int MT, bool O16>
int prepare_t(int dev, size_t smem) {
    static std::atomic<uint64_t> done{0};  // bit d: device d prepared
    if (dev < 0 || dev >= 64) return MQ_ERR_CUDA;
    const uint64_t bit = 1ull << dev;
    if (done.load(std::memory_order_acquire) & bit) return MQ_OK;
    if (cudaFuncSetAttribute(gemv_kernel<BITS, MT, O16>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
        return MQ_ERR_CUDA;
    done.fetch_or(bit, std::memory_order_release);
    return MQ_OK;
}

// Stages of the ring: as deep as fits beside a second CTA of the same size on
// the SM (the next launch's, which programmatic dependent launch starts while
// this one drains).
constexpr int SMEM_BUDGET = 110 * 1024;

template <int BITS, int MT>
int ring_stages() {
    int st = (int)((SMEM_BUDGET - sizeof(Tail<MT>) - 128) / stage_bytes(BITS, MT));
    return st > MAX_STAGES ? MAX_STAGES : st;
}

template <int BITS, int MT, bool O16>
int launch_t(const Problem *probs, int count, cudaStream_t stream) {
    constexpr int KPB = 8 / BITS;
    const int stages = ring_stages<BITS, MT>();
    const size_t smem = smem_bytes<BITS, MT>(stages);
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return MQ_ERR_CUDA;
    if (prepare_t<BITS, MT, O16>(dev, smem_bytes<BITS, MT>(ring_stages<BITS, MT>())) != MQ_OK)
        return MQ_ERR_CUDA;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MQ_ERR_CUDA;
    for (int begin = 0; begin < count; begin += MAX_PROBLEMS) {
        const int n = count - begin < MAX_PROBLEMS ? count - begin : MAX_PROBLEMS;
        Params P{};
        P.pre_w = 1;
        // row tiles of every problem, and the bytes each one streams (plus a
        // fixed share for its epilogue)
        std::vector<long long> cost;
        int tiles = 0;
        for (int i = 0; i < n; ++i) {
            Problem &q = P.p[i];
            q = probs[begin + i];
            if (q.wdynamic) P.pre_w = 0;
            q.tile_begin = tiles;
            q.tiles_m = (q.N + TR - 1) / TR;
            tiles += q.tiles_m;
            const long long L = q.K / KPB;
            for (int t = 0; t < q.tiles_m; ++t) {
                const int rows = q.N - t * TR < TR ? q.N - t * TR : TR;
                cost.push_back(rows * L + q.M * L * KPB / 8 + 2048);
            }
        }
        if (tiles == 0) continue;
        int grid = sms < MAX_GRID ? sms : MAX_GRID;
        if (grid > tiles) grid = tiles;
        // contiguous runs of row tiles of about equal cost
        long long total = 0;
        for (long long c : cost) total += c;
        P.cta_begin[0] = 0;
        long long acc = 0;
        int t = 0;
        for (int c = 1; c < grid; ++c) {
            const long long target = total * c / grid;
            while (t < tiles && acc + cost[t] / 2 <= target) acc += cost[t++];
            P.cta_begin[c] = t;
        }
        P.cta_begin[grid] = tiles;
        P.count = n;
        P.stages = stages;
        P.status = device_status_ptr();
        P.wait_ns = wait_limit_ns();
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)grid, 1, 1);
        cfg.blockDim = dim3(THREADS, 1, 1);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = stream;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaLaunchKernelEx(&cfg, gemv_kernel<BITS, MT, O16>, P) != cudaSuccess)
            return MQ_ERR_CUDA;
    }
    return MQ_OK;
}

}  // namespace gemv

// Whether a decode launch can take this kernel: 8-bit activations, at most
// two tokens, K > 0, and (unless forced) enough row tiles of small enough
// size that contiguous runs of them balance the SMs.
bool gemv_suits(const Problem *probs, int count, int sms, bool force) {
    using namespace gemv;
    if (count <= 0) return false;
    long long total = 0, max_tile = 0, tiles = 0;
    for (int i = 0; i < count; ++i) {
        const Problem &q = probs[i];
        if (q.a16 || q.M < 1 || q.M > MAX_MT || q.K <= 0 || q.N <= 0) return false;
        const long long L = (long long)q.K * q.bits / 8;
        const long long tile = TR * L;
        total += (long long)q.N * L;
        tiles += (q.N + TR - 1) / TR;
        if (tile > max_tile) max_tile = tile;
    }
    if (force) return true;
    // at least two row tiles per SM, and no tile above a quarter of an SM's share
    return tiles >= 2LL * sms && max_tile * 4 * sms <= total;
}

int launch_gemv(const Problem *probs, int count, void *stream) {
    using namespace gemv;
    int mt = 0;
    for (int i = 0; i < count; ++i) mt = probs[i].M > mt ? probs[i].M : mt;
    const bool i4 = probs[0].bits == 4, o16 = probs[0].o16;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
#define MQ_GEMV_CASE(B, T, O) \
    if ((B == 4) == i4 && mt == T && o16 == O) return launch_t<B, T, O>(probs, count, s);
    MQ_GEMV_CASE(4, 1, false)
    MQ_GEMV_CASE(4, 2, false)
    MQ_GEMV_CASE(8, 1, false)
    MQ_GEMV_CASE(8, 2, false)
    MQ_GEMV_CASE(4, 1, true)
    MQ_GEMV_CASE(4, 2, true)
    MQ_GEMV_CASE(8, 1, true)
    MQ_GEMV_CASE(8, 2, true)
#undef MQ_GEMV_CASE
    return MQ_ERR_INVALID_ARG;
}

}  // namespace mq
