// mq_gemv.cu -- weight-streaming kernel for the integer-only quantized linear
// layer at one to four tokens (autoregressive generation), bit-exact.
//
// At M <= 4 the layer reads every weight once and does one to four MACs with
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
// and again.  Three CTAs of eight warps per SM (two for two tokens) keep about
// 96 KB of weights in flight per SM.  The weights of a warp's next group are
// requested before the current group's epilogue, and those of its first group
// before waiting for the previous kernel in the stream (programmatic
// dependent launch): packed weights are constant inputs.  Measured against a
// shared-memory ring fed by bulk or tensor-map copies, this path streams more:
// one CTA's copy engine stops near 3.9 TB/s over the GPU, and per-stage
// barriers cost more than the work of an 8 KB stage.
//
// Compute.  int4 weights: the low nibbles of a word give u = w + 8 in
// [0, 15] per byte with one LOP3, the high nibbles 16 u in [0, 240] in place
// with another; a signed and an unsigned-by-signed dp4a multiply them with the
// activations of the even and the odd k of the word, which two PRMT per word
// pair form once per step and token (shared by the R rows).  The sums of the
// high nibbles are multiples of 16 and are divided back exactly.  int8
// weights go to dp4a unchanged.  The int32 sums are exact: |partial| <=
// 240 * 128 * 32768 < 2^31.  Bytes past the end of a row load as zero.
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
constexpr int R = 4;                     // rows per group
constexpr int MAX_MT = 4;                // tokens
// Weight bytes of a row per step: 1 KB (two 16-byte loads per lane) for one
// or two tokens; 512 bytes for up to four, whose activations of a step would
// not fit the registers otherwise.
template <int MT>
__host__ __device__ constexpr int step_of() { return MT <= 2 ? 1024 : 512; }
constexpr int MAX_PROBLEMS = DECODE_MAX_PROBLEMS;
// CTAs per SM: three for one token (80 registers a thread); two for two or
// four tokens, whose activation vectors would not fit 80 registers without
// spills (measured, two tokens: 9.9 us against 10.5 us per TinyLlama-shaped
// block).
template <int MT>
constexpr int ctas_per_sm() { return MT == 1 ? 3 : 2; }

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

// acc + sum of the four unsigned bytes of a times the four signed bytes of b
__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int acc) {
    int d;
    asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(acc));
    return d;
}

// The activations of 32 consecutive k (two 16-byte vectors) regrouped for
// the int4 words that hold them: word i (k 8i .. 8i + 7, low nibbles the even
// k) meets e[i] = x of k 8i, 8i+2, 8i+4, 8i+6 and o[i] = x of the odd k.
struct XEO {
    uint32_t e[4], o[4];
};

__device__ __forceinline__ XEO x_even_odd(uint4 a, uint4 b) {
    const uint32_t v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
    XEO r;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        r.e[i] = prmt(v[2 * i], v[2 * i + 1], 0x6420u);
        r.o[i] = prmt(v[2 * i], v[2 * i + 1], 0x7531u);
    }
    return r;
}

// int4: lo += sum(u x) over the low nibbles (u = w + 8), hi += 16 sum(u x)
// over the high nibbles, for the 16 weight bytes of `w`.
__device__ __forceinline__ void dot16_i4(uint4 w, const XEO &x, int &lo, int &hi) {
    const uint32_t wi[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        lo = __dp4a((int)((wi[i] & 0x0F0F0F0Fu) ^ 0x08080808u), (int)x.e[i], lo);
        hi = dp4a_us((wi[i] & 0xF0F0F0F0u) ^ 0x80808080u, x.o[i], hi);
    }
}

// One step's loads of a row group: 16 weight bytes of each row at two places
// (c0, c0 + 512) and the activations they meet.
template <int BITS, int MT>
struct Step {
    static constexpr int KPB = 8 / BITS;
    static constexpr int H = step_of<MT>() / 512;  // 16-byte loads of a row per lane
    uint4 w[R][H];
    uint4 x[MT][H][KPB];
};

// The loads of one step: c0 is the step's first byte in a row (warp-uniform);
// lane l takes bytes c0 + 16 l and c0 + 512 + 16 l.  Full groups of full
// steps load without bounds checks; the others read zero past the matrix.
template <int BITS, int MT>
__device__ __forceinline__ void load_weights(Step<BITS, MT> &st, const Problem &p, int n0,
                                             int rows, int c0, int lane) {
    constexpr int H = Step<BITS, MT>::H;
    const int L = p.K * BITS / 8;
    const size_t ldw = (size_t)p.ldw;
    const uint8_t *b = p.w + (size_t)n0 * ldw + c0 + 16 * lane;
    if (rows == R && c0 + step_of<MT>() <= L) {
#pragma unroll
        for (int r = 0; r < R; ++r)
#pragma unroll
            for (int h = 0; h < H; ++h) st.w[r][h] = ldg_w(b + r * ldw + 512 * h);
        return;
    }
#pragma unroll
    for (int h = 0; h < H; ++h) {
        const bool in = c0 + 512 * h + 16 * lane < L;
#pragma unroll
        for (int r = 0; r < R; ++r)
            st.w[r][h] = (in && r < rows) ? ldg_w(b + r * ldw + 512 * h)
                                          : make_uint4(0u, 0u, 0u, 0u);
    }
}

template <int BITS, int MT>
__device__ __forceinline__ void load_x(Step<BITS, MT> &st, const Problem &p, int c0, int lane) {
    constexpr int KPB = 8 / BITS;
    constexpr int H = Step<BITS, MT>::H;
    const int L = p.K * BITS / 8;
    const int8_t *b = p.x + ((size_t)c0 + 16 * lane) * KPB;
    const size_t ldx = (size_t)p.ldx;
    if (p.M == MT && c0 + step_of<MT>() <= L) {
#pragma unroll
        for (int m = 0; m < MT; ++m)
#pragma unroll
            for (int h = 0; h < H; ++h)
#pragma unroll
                for (int i = 0; i < KPB; ++i) st.x[m][h][i] = ldg_x(b + m * ldx + 512 * KPB * h + 16 * i);
        return;
    }
#pragma unroll
    for (int h = 0; h < H; ++h) {
        const bool in = c0 + 512 * h + 16 * lane < L;
#pragma unroll
        for (int m = 0; m < MT; ++m)
#pragma unroll
            for (int i = 0; i < KPB; ++i)
                st.x[m][h][i] = (in && m < p.M) ? ldg_x(b + m * ldx + 512 * KPB * h + 16 * i)
                                                : make_uint4(0u, 0u, 0u, 0u);
    }
}

// Reduce-scatter over the warp: on entry each lane holds NV partial sums; on
// exit lane l holds in v[0] the total of value l / (32 / NV) over all lanes.
template <int NV>
__device__ __forceinline__ int reduce_scatter(int (&v)[NV], int lane) {
    static_assert(NV == 4 || NV == 8 || NV == 16, "4, 8 or 16 values");
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
#pragma unroll
    for (int bit = 16 / NV; bit >= 1; bit >>= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], bit);
    return v[0];
}

template <int BITS, int MT, bool O16>
__global__ void __launch_bounds__(THREADS, ctas_per_sm<MT>()) gemv_kernel(const __grid_constant__ Params P) {
    constexpr int NV = R * MT;  // sums per lane
    constexpr int STEP = step_of<MT>();
    constexpr int H = Step<BITS, MT>::H;
    const int lane = threadIdx.x & 31;
    const long long W = (long long)gridDim.x * WARPS;
    const long long gw = (long long)blockIdx.x * WARPS + (threadIdx.x >> 5);
    const long long C = P.cost_begin[P.count];
    // the range of weights this warp's groups start in
    const long long c_lo = C * gw / W, c_hi = C * (gw + 1) / W;
    if (threadIdx.x == 0) griddep_launch_dependents();

    // the warp's row groups: those whose starting weight lies in [c_lo, c_hi)
    auto first_group = [&](int q, long long c) -> long long {
        // first group j of problem q with cost_begin[q] + j cost_group[q] >= c
        const long long d = c - P.cost_begin[q];
        if (d <= 0) return 0;
        return (d + P.cost_group[q] - 1) / P.cost_group[q];
    };
    // (pi, g) advanced by k groups of the warp's sequence; false past its end
    auto advance = [&](int &q, long long &j, long long k) -> bool {
        j += k;
        while (q < P.count && P.cost_begin[q] < c_hi) {
            const long long last = min((long long)P.p[q].tiles_m, first_group(q, c_hi));
            if (j < last) return true;
            j -= last;  // the groups past this problem continue in the next one
            ++q;
        }
        return false;
    };
    int pi = 0;
    while (pi + 1 < P.count && P.cost_begin[pi + 1] <= c_lo) ++pi;
    long long g = first_group(pi, c_lo);
    bool have = advance(pi, g, 0);
    // The weights of a group's first step are loaded before the group begins
    // (the previous group's epilogue, or the wait for the previous kernel,
    // overlaps them).
    Step<BITS, MT> st;
    if (have && P.pre_w)
        load_weights(st, P.p[pi], (int)g * R, min(R, P.p[pi].N - (int)g * R), 0, lane);
    griddep_wait();  // x, parameters and outputs only after the previous kernel
    if (have && !P.pre_w)
        load_weights(st, P.p[pi], (int)g * R, min(R, P.p[pi].N - (int)g * R), 0, lane);
    int xsum[MT];
    int cur_pi = -1;
    while (have) {
        const Problem &p = P.p[pi];
        const int nsteps = (p.K * BITS / 8 + STEP - 1) / STEP;
        const int n0 = (int)g * R;
        const int rows = min(R, p.N - n0);
        const bool first = pi != cur_pi;  // the warp's first group of this problem
        cur_pi = pi;
        // this lane's output, if any: value lane / (32 / NV) of the reduce-scatter
        const int vi = lane / (32 / NV);
        const int er = vi / MT, em = vi % MT;
        const bool owner = lane % (32 / NV) == 0 && er < rows && em < p.M;
        int32_t colsum = 0, m0 = 0, sh = 33, zw = 0, res = 0;
        if (owner) {
            const int n = n0 + er;
            colsum = __ldg(p.colsum + n);
            m0 = __ldg(p.M0 + n);
            sh = __ldg(p.shift + n);
            if (p.zw) zw = __ldg(p.zw + n);
            if (p.residual) res = p.residual[(size_t)em * p.ldy + n];
        }
        int acc[NV], acc_hi[BITS == 4 ? NV : 1];
        int xs[MT];
#pragma unroll
        for (int i = 0; i < NV; ++i) acc[i] = 0;
#pragma unroll
        for (int i = 0; i < (BITS == 4 ? NV : 1); ++i) acc_hi[i] = 0;
#pragma unroll
        for (int m = 0; m < MT; ++m) xs[m] = 0;
        for (int s = 0; s < nsteps; ++s) {
            if (s > 0) load_weights(st, p, n0, rows, s * STEP, lane);
            load_x(st, p, s * STEP, lane);
            if (first) {
#pragma unroll
                for (int m = 0; m < MT; ++m)
#pragma unroll
                    for (int h = 0; h < H; ++h)
#pragma unroll
                        for (int i = 0; i < 8 / BITS; ++i) xs[m] = sum4(st.x[m][h][i], xs[m]);
            }
            if constexpr (BITS == 4) {
#pragma unroll
                for (int m = 0; m < MT; ++m)
#pragma unroll
                    for (int h = 0; h < H; ++h) {
                        const XEO x = x_even_odd(st.x[m][h][0], st.x[m][h][1]);
#pragma unroll
                        for (int r = 0; r < R; ++r)
                            dot16_i4(st.w[r][h], x, acc[r * MT + m], acc_hi[r * MT + m]);
                    }
            } else {
#pragma unroll
                for (int r = 0; r < R; ++r)
#pragma unroll
                    for (int m = 0; m < MT; ++m)
#pragma unroll
                        for (int h = 0; h < H; ++h)
                            acc[r * MT + m] = dp4a4(st.w[r][h], st.x[m][h][0], acc[r * MT + m]);
            }
        }
        if constexpr (BITS == 4) {
            // the high nibbles' sums are exact multiples of 16
#pragma unroll
            for (int i = 0; i < NV; ++i) acc[i] += acc_hi[i] >> 4;
        }
        // the next group's first weights go out before this group's epilogue
        int npi = pi;
        long long ng = g;
        have = advance(npi, ng, 1);
        if (have) load_weights(st, P.p[npi], (int)ng * R, min(R, P.p[npi].N - (int)ng * R), 0,
                               lane);
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
            int32_t xsm = xsum[0];  // sum(x) of this output's token
#pragma unroll
            for (int m = 1; m < MT; ++m)
                if (em == m) xsm = xsum[m];
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
        pi = npi;
        g = ng;
    }
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
            P.cost_group[i] = (q.K * q.bits / 8 + step_of<MT>() - 1) / step_of<MT>() + 1;
            P.cost_begin[i] = cost;
            cost += (long long)q.tiles_m * P.cost_group[i];
            groups += q.tiles_m;
        }
        P.cost_begin[n] = cost;
        P.count = n;
        if (groups == 0) continue;
        long long warps = (long long)ctas_per_sm<MT>() * sms * WARPS;
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
    int mt = 0;
    for (int i = 0; i < count; ++i) {
        const Problem &q = probs[i];
        if (q.a16 || q.M < 1 || q.M > MAX_MT || q.K <= 0 || q.N <= 0) return false;
        groups += (q.N + R - 1) / R;
        mt = q.M > mt ? q.M : mt;
    }
    const int occ = mt == 1 ? ctas_per_sm<1>() : ctas_per_sm<2>();
    return force || groups >= (long long)occ * sms * WARPS;
}

int launch_gemv(const Problem *probs, int count, void *stream) {
    using namespace gemv;
    int mt = 0;
    for (int i = 0; i < count; ++i) mt = probs[i].M > mt ? probs[i].M : mt;
    const bool i4 = probs[0].bits == 4, o16 = probs[0].o16;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
#define MQ_GEMV_CASE(B, T, O) \
    if ((B == 4) == i4 && mt == T && o16 == O) return launch_t<B, T, O>(probs, count, s);
    if (mt == 3) mt = 4;  // the four-token variant (tokens past M read as zero)
    MQ_GEMV_CASE(4, 1, false)
    MQ_GEMV_CASE(4, 2, false)
    MQ_GEMV_CASE(4, 4, false)
    MQ_GEMV_CASE(8, 1, false)
    MQ_GEMV_CASE(8, 2, false)
    MQ_GEMV_CASE(8, 4, false)
    MQ_GEMV_CASE(4, 1, true)
    MQ_GEMV_CASE(4, 2, true)
    MQ_GEMV_CASE(4, 4, true)
    MQ_GEMV_CASE(8, 1, true)
    MQ_GEMV_CASE(8, 2, true)
    MQ_GEMV_CASE(8, 4, true)
#undef MQ_GEMV_CASE
    return MQ_ERR_INVALID_ARG;
}

}  // namespace mq
