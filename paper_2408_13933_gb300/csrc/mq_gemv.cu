// mq_gemv.cu -- weight-streaming kernel for the integer-only quantized linear
// layer at one or two tokens (autoregressive generation), bit-exact.
//
// At M <= 2 the layer reads every weight once and does one or two MACs with
// it: the time is the weight stream (the paper notes that autoregressive
// generation is memory-bound, Sec. 5.6 and Appendix A.2).  This kernel is
// built to stream HBM at its rate, with no shared memory and no barriers:
//
// Work.  Every problem's weight matrix is cut into row groups of R = 4 rows.
// The row groups of all problems of a launch form one sequence, weighed by
// the bytes they stream; each warp of the grid takes a contiguous run of
// about equal weight (the warps of a CTA take neighbouring runs, so every SM
// streams about the same number of bytes).  A row group never spans two
// warps, so every output is finished by the warp that streamed it.
//
// Data path.  A warp reads its rows 1 KB at a time: lane l loads the 16 bytes
// at 16 l and 512 + 16 l of each of the R rows (eight 16-byte loads in flight
// per lane, streaming past L1), and the matching activation bytes through the
// L1 cache, where x stays for the whole launch: every SM reads all of it again
// and again.  The loads of a warp's first step are issued before waiting for
// the previous kernel in the stream (programmatic dependent launch): packed
// weights are constant inputs.
//
// Compute.  int4 weights: one LOP3 (and a shift for the high nibbles) forms
// u = w + 8 in [0, 15] per byte and two PRMT put the nibbles in k order, so
// that one dp4a multiplies four weights with four activation bytes as they
// are stored; int8 weights go to dp4a unchanged.  The int32 sums are exact:
// |partial| <= 15 * 128 * 65536 < 2^31.  Bytes past the end of a row load as
// zero.
//
// Epilogue (per row group).  The R x M lane sums are reduced over the warp by
// a reduce-scatter (each shuffle halves the values a lane holds), leaving one
// (row, token) sum per group of lanes; its first lane removes the bias,
// sum(w x) = sum(u x) - 8 sum(x) (int4), forms sum((x - zx)(w - zw)) =
// sum(w x) - zw sum(x) - zx (colsum - K zw), requantizes (round half up,
// saturate), adds the optional residual and stores.  Its parameters were
// loaded when the group began, so their latency hides behind the weights'.
// sum(x) of each problem's tokens is accumulated while the warp streams its
// first row group of that problem, which covers every k.
#include <cuda_runtime.h>

#include <atomic>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {
namespace gemv {

constexpr int WARPS = 8;                 // per CTA
constexpr int THREADS = WARPS * 32;
constexpr int CTAS_PER_SM = 3;
constexpr int R = 4;                     // rows per group
constexpr int STEP = 1024;               // weight bytes of a row per step
constexpr int MAX_MT = 2;                // tokens
constexpr int MAX_PROBLEMS = DECODE_MAX_PROBLEMS;

struct Params {
    Problem p[MAX_PROBLEMS];  // tile_begin = first row group, tiles_m = row groups
    long long cost_begin[MAX_PROBLEMS + 1];  // weight of the problems before p
    int cost_group[MAX_PROBLEMS];            // weight of one row group of p
    int count;
    int pre_w;  // 1: weights are read before griddep_wait
};

__device__ __forceinline__ uint4 ldg_w(const uint8_t *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

// 16 bytes of x through the L1 cache (read-only for the kernel's lifetime:
// read only after the previous kernel in the stream has completed).
__device__ __forceinline__ uint4 ldg_x(const int8_t *p) {
    uint4 v;
    asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

__device__ __forceinline__ int dp4a4(uint4 w, uint4 x, int acc) {
    acc = __dp4a((int)w.x, (int)x.x, acc);
    acc = __dp4a((int)w.y, (int)x.y, acc);
    acc = __dp4a((int)w.z, (int)x.z, acc);
    return __dp4a((int)w.w, (int)x.w, acc);
}

__device__ __forceinline__ int sum4(uint4 x, int acc) {
    return dp4a4(make_uint4(0x01010101u, 0x01010101u, 0x01010101u, 0x01010101u), x, acc);
}

// acc += w . x over the 16 weight bytes of `w` (int4: 32 k, x in two vectors;
// int8: 16 k, x in one).
template <int BITS>
__device__ __forceinline__ int dot16(uint4 w, const uint4 *x, int acc) {
    if constexpr (BITS == 4) {
        // word i holds k = 8 i .. 8 i + 7; lo / hi are k 8i..8i+3 / 8i+4..8i+7
        // as bytes u = w + 8
        const uint32_t wi[4] = {w.x, w.y, w.z, w.w};
        uint32_t lo[4], hi[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint32_t e = (wi[i] & 0x0F0F0F0Fu) ^ 0x08080808u;
            const uint32_t o = ((wi[i] >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
            lo[i] = prmt(e, o, 0x5140u);
            hi[i] = prmt(e, o, 0x7362u);
        }
        acc = dp4a4(make_uint4(lo[0], hi[0], lo[1], hi[1]), x[0], acc);
        return dp4a4(make_uint4(lo[2], hi[2], lo[3], hi[3]), x[1], acc);
    } else {
        return dp4a4(w, x[0], acc);
    }
}

// One step's loads of a row group: 16 weight bytes of each row at two places
// (c0, c0 + 512) and the activations they meet.
template <int BITS, int MT>
struct Step {
    static constexpr int KPB = 8 / BITS;
    uint4 w[R][2];
    uint4 x[MT][2][KPB];
};

template <int BITS, int MT>
__device__ __forceinline__ void load_weights(Step<BITS, MT> &st, const Problem &p, int n0,
                                             int rows, int col) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = col + 512 * h;
        const bool in = c < p.K * BITS / 8;
#pragma unroll
        for (int r = 0; r < R; ++r)
            st.w[r][h] = (in && r < rows) ? ldg_w(p.w + (size_t)(n0 + r) * p.ldw + c)
                                          : make_uint4(0u, 0u, 0u, 0u);
    }
}

template <int BITS, int MT>
__device__ __forceinline__ void load_x(Step<BITS, MT> &st, const Problem &p, int col) {
    constexpr int KPB = 8 / BITS;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = col + 512 * h;
        const bool in = c < p.K * BITS / 8;
#pragma unroll
        for (int m = 0; m < MT; ++m)
#pragma unroll
            for (int i = 0; i < KPB; ++i)
                st.x[m][h][i] = (in && m < p.M)
                                    ? ldg_x(p.x + (size_t)m * p.ldx + (size_t)c * KPB + 16 * i)
                                    : make_uint4(0u, 0u, 0u, 0u);
    }
}

// Reduce-scatter over the warp: on entry each lane holds R x MT partial sums;
// on exit lane l holds in v[0] the total of value (l >> 3) (R x MT = 4: row
// l >> 3) or, for R x MT = 8, of value 2 (l >> 3) + ((l >> 2) & 1).
template <int NV>
__device__ __forceinline__ int reduce_scatter(int (&v)[NV], int lane) {
    static_assert(NV == 4 || NV == 8, "4 or 8 values");
    // halve the values held at each of the first log2(NV) steps
#pragma unroll
    for (int n = NV, bit = 16; n > 1; n >>= 1, bit >>= 1) {
        const bool upper = (lane & bit) != 0;
#pragma unroll
        for (int i = 0; i < n / 2; ++i) {
            const int keep = upper ? v[i + n / 2] : v[i];
            const int give = upper ? v[i] : v[i + n / 2];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, give, bit);
        }
    }
    // the remaining lanes of each group: full reduction
    constexpr int rest = NV == 4 ? 4 : 2;  // bits below the ones used above
#pragma unroll
    for (int bit = rest; bit >= 1; bit >>= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], bit);
    return v[0];
}

template <int BITS, int MT, bool O16>
__global__ void __launch_bounds__(THREADS, CTAS_PER_SM) gemv_kernel(const __grid_constant__ Params P) {
    constexpr int NV = R * MT;  // sums per lane
    const int lane = threadIdx.x & 31;
    const long long W = (long long)gridDim.x * WARPS;
    const long long gw = (long long)blockIdx.x * WARPS + (threadIdx.x >> 5);
    const long long C = P.cost_begin[P.count];
    const long long c_lo = C * gw / W, c_hi = C * (gw + 1) / W;
    if (threadIdx.x == 0) griddep_launch_dependents();

    // the warp's row groups: those whose starting weight lies in [c_lo, c_hi)
    int pi = 0;
    while (pi + 1 < P.count && P.cost_begin[pi + 1] <= c_lo) ++pi;
    auto first_group = [&](int q, long long c) -> long long {
        // first group j of problem q with cost_begin[q] + j cost_group[q] >= c
        const long long d = c - P.cost_begin[q];
        if (d <= 0) return 0;
        return (d + P.cost_group[q] - 1) / P.cost_group[q];
    };
    long long g = first_group(pi, c_lo);
    bool waited = !P.pre_w;
    if (waited) griddep_wait();
    int xsum[MT];
    int cur_pi = -1;
    for (; pi < P.count && P.cost_begin[pi] < c_hi; ++pi, g = 0) {
        const Problem &p = P.p[pi];
        const long long g_end = min((long long)p.tiles_m, first_group(pi, c_hi));
        const int L = p.K * BITS / 8;
        const int nsteps = (L + STEP - 1) / STEP;
        for (; g < g_end; ++g) {
            const int n0 = (int)g * R;
            const int rows = min(R, p.N - n0);
            Step<BITS, MT> st;
            load_weights(st, p, n0, rows, 16 * lane);
            if (!waited) {  // x, parameters and outputs only after the previous kernel
                griddep_wait();
                waited = true;
            }
            const bool first = pi != cur_pi;  // the warp's first group of this problem
            cur_pi = pi;
            // this lane's output, if any: value (lane >> 3) of the reduce-scatter
            const int vi = NV == 4 ? (lane >> 3) : 2 * (lane >> 3) + ((lane >> 2) & 1);
            const int er = MT == 1 ? vi : vi >> 1, em = MT == 1 ? 0 : vi & 1;
            const bool owner = (lane & (NV == 4 ? 7 : 3)) == 0 && er < rows && em < p.M;
            int32_t colsum = 0, m0 = 0, sh = 33, zw = 0, res = 0;
            if (owner) {
                const int n = n0 + er;
                colsum = __ldg(p.colsum + n);
                m0 = __ldg(p.M0 + n);
                sh = __ldg(p.shift + n);
                if (p.zw) zw = __ldg(p.zw + n);
                if (p.residual) res = p.residual[(size_t)em * p.ldy + n];
            }
            int acc[NV];
            int xs[MT];
#pragma unroll
            for (int i = 0; i < NV; ++i) acc[i] = 0;
#pragma unroll
            for (int m = 0; m < MT; ++m) xs[m] = 0;
            for (int s = 0; s < nsteps; ++s) {
                if (s > 0) load_weights(st, p, n0, rows, s * STEP + 16 * lane);
                load_x(st, p, s * STEP + 16 * lane);
                if (first) {
#pragma unroll
                    for (int m = 0; m < MT; ++m)
#pragma unroll
                        for (int h = 0; h < 2; ++h)
#pragma unroll
                            for (int i = 0; i < 8 / BITS; ++i) xs[m] = sum4(st.x[m][h][i], xs[m]);
                }
#pragma unroll
                for (int r = 0; r < R; ++r)
#pragma unroll
                    for (int m = 0; m < MT; ++m)
#pragma unroll
                        for (int h = 0; h < 2; ++h)
                            acc[r * MT + m] = dot16<BITS>(st.w[r][h], st.x[m][h], acc[r * MT + m]);
            }
            if (first) {
#pragma unroll
                for (int m = 0; m < MT; ++m) {
#pragma unroll
                    for (int bit = 16; bit >= 1; bit >>= 1)
                        xs[m] += __shfl_xor_sync(0xffffffffu, xs[m], bit);
                    xsum[m] = xs[m];
                }
            }
            const int sum = reduce_scatter<NV>(acc, lane);
            if (owner) {
                const int n = n0 + er;
                const int32_t xsm = MT == 1 ? xsum[0] : (em ? xsum[MT - 1] : xsum[0]);
                // sum(w x) = sum(u x) - 8 sum(x) (int4); then the zero points:
                // sum((x - zx)(w - zw)) = sum(w x) - zw sum(x) - zx (colsum - K zw)
                // (two's-complement wrap is exact: the true value fits int32)
                const uint32_t wx = (uint32_t)sum - (uint32_t)(BITS == 4 ? 8 * xsm : 0);
                const int32_t a =
                    (int32_t)(wx - (uint32_t)zw * (uint32_t)xsm -
                              (uint32_t)p.zx * ((uint32_t)colsum - (uint32_t)p.K * (uint32_t)zw));
                if constexpr (O16) {
                    reinterpret_cast<int16_t *>(p.y)[(size_t)em * p.ldy + n] =
                        (int16_t)mq_requant16((int64_t)a, m0, sh, p.zy);
                } else {
                    int32_t y = mq_requant(a, m0, sh, p.zy);
                    if (p.residual) y = min(127, max(-128, y + res));
                    p.y[(size_t)em * p.ldy + n] = (int8_t)y;
                }
            }
        }
    }
    if (!waited) griddep_wait();  // a warp without work still orders after its predecessor
}

template <int BITS, int MT, bool O16>
int launch_t(const Problem *probs, int count, cudaStream_t stream) {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MQ_ERR_CUDA;
    for (int begin = 0; begin < count; begin += MAX_PROBLEMS) {
        const int n = count - begin < MAX_PROBLEMS ? count - begin : MAX_PROBLEMS;
        Params P{};
        P.pre_w = 1;
        long long cost = 0, groups = 0;
        for (int i = 0; i < n; ++i) {
            Problem &q = P.p[i];
            q = probs[begin + i];
            if (q.wdynamic) P.pre_w = 0;
            q.tiles_m = (q.N + R - 1) / R;
            // a group's weight: its 1 KB steps and one more for its epilogue
            P.cost_group[i] = (q.K * q.bits / 8 + STEP - 1) / STEP + 1;
            P.cost_begin[i] = cost;
            cost += (long long)q.tiles_m * P.cost_group[i];
            groups += q.tiles_m;
        }
        P.cost_begin[n] = cost;
        P.count = n;
        if (groups == 0) continue;
        long long warps = (long long)CTAS_PER_SM * sms * WARPS;
        if (warps > groups) warps = groups;
        const int grid = (int)((warps + WARPS - 1) / WARPS);
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)grid, 1, 1);
        cfg.blockDim = dim3(THREADS, 1, 1);
        cfg.dynamicSmemBytes = 0;
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
// two tokens, K > 0, and (unless forced) at least one row group per warp of
// the grid, so that the launch's bytes spread over every SM.
bool gemv_suits(const Problem *probs, int count, int sms, bool force) {
    using namespace gemv;
    if (count <= 0) return false;
    long long groups = 0;
    for (int i = 0; i < count; ++i) {
        const Problem &q = probs[i];
        if (q.a16 || q.M < 1 || q.M > MAX_MT || q.K <= 0 || q.N <= 0) return false;
        groups += (q.N + R - 1) / R;
    }
    return force || groups >= (long long)CTAS_PER_SM * sms * WARPS;
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
