// mq_fold.cu -- the offline producer of the weights the integer layer
// consumes: the equivalent transform of eq. 1 folded into f32 weights, weight
// quantization (symmetric per channel, or asymmetric per channel / per tensor
// with the quantizer of eqs. 2-4, Sec. 5.1), packing and colsum, on the
// device.
//
// With weights stored [N out][K in], eq. 1's S W scales input channel k by
// s_in[k] and the S^-1 of the next transform (Figure 3) scales output
// channel n by 1 / s_out[n]:  w'[n][k] = (w[n][k] * s_in[k]) / s_out[n].
// Every floating-point step is one IEEE f32 operation rounded to nearest
// (the _rn intrinsics keep the compiler from contracting them), so the codes
// are the same on any correct implementation of the definition.
//
// Three launches over a whole batch of linears (one call for a model block):
// per-row minima / maxima of w', for the per-tensor scheme a one-CTA-per-
// tensor reduction of those to the tensor's, then quantization + packing +
// colsum, w' recomputed from w.  The last pass visits the rows in the reverse
// order of the first, so it starts on the rows the first pass read last,
// which are still in L2.  The later launches use programmatic dependent
// launch: they start while the previous pass drains and wait for it before
// reading its statistics.  The row kernels give each row one warp, so a CTA
// of eight warps has eight rows in flight and the reductions are warp
// shuffles.
// When K is a multiple of 4 and the rows are 16-byte aligned, a lane loads
// four weights (and four input scales) at a time, UNROLL such loads before
// using them, and writes their codes as one 4-byte (int8) or 2-byte (int4)
// store; the arithmetic per element is the scalar path's, and min, max and
// integer sums do not depend on the order.
#include <cuda_runtime.h>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {
namespace fold {

constexpr int THREADS = 256;
constexpr int ROWS = THREADS / 32;  // rows per CTA, one warp each
constexpr int UNROLL = 4;           // float4 loads a lane issues before using them

// w'[n][k]: multiply by s_in[k] first, then divide by s_out[n].
__device__ __forceinline__ float fold_one(float w, const float *s_in, int k, bool has_out,
                                          float s_out) {
    float v = w;
    if (s_in) v = __fmul_rn(v, __ldg(s_in + k));
    if (has_out) v = __fdiv_rn(v, s_out);
    return v;
}

// fold_one on four consecutive weights, with their four input scales s.
__device__ __forceinline__ void fold_four(float4 w, float4 s, bool has_in, bool has_out,
                                          float s_out, float v[4]) {
    v[0] = w.x, v[1] = w.y, v[2] = w.z, v[3] = w.w;
    if (has_in) {
        v[0] = __fmul_rn(v[0], s.x), v[1] = __fmul_rn(v[1], s.y);
        v[2] = __fmul_rn(v[2], s.z), v[3] = __fmul_rn(v[3], s.w);
    }
    if (has_out) {
#pragma unroll
        for (int e = 0; e < 4; ++e) v[e] = __fdiv_rn(v[e], s_out);
    }
}

// The code of one folded weight: clamp(rint(v / scale) + zero, cmin, qmax),
// with v / scale the correctly rounded f32 quotient.  Only its rint is used,
// so the quotient is first taken as q = v * (1 / scale), both correctly
// rounded: while 1 / scale and q are normal, |q - RN(v / scale)| is below
// 3.01 * 2^-24 * |q|.  If q is farther than 2^-21 * |q| from the half-integer
// floor(q) + 0.5 (the only rint boundary within 0.5 of it, for |q| < 2^21),
// both lie strictly between the same two half-integers and have the same
// rint; otherwise (near a tie, NaN, large q or scale) the quotient is taken
// by the exact division.  recip_ok says 1 / scale is normal (scale < 2^100).
__device__ __forceinline__ int32_t code_of(float v, float scale, float rscale, bool recip_ok,
                                           int32_t zero, int32_t cmin, int32_t qmax) {
    const float q = __fmul_rn(v, rscale);
    const float aq = fabsf(q);
    const float d = fabsf(__fsub_rn(q, __fadd_rn(floorf(q), 0.5f)));
    const float t = (recip_ok && aq < 0x1p21f && d > aq * 0x1p-21f) ? rintf(q)
                                                                     : rintf(__fdiv_rn(v, scale));
    return (int32_t)fminf(fmaxf(__fadd_rn(t, (float)zero), (float)cmin), (float)qmax);
}

__device__ float fmin_op(float a, float b) { return fminf(a, b); }
__device__ float fmax_op(float a, float b) { return fmaxf(a, b); }
__device__ int32_t iadd_op(int32_t a, int32_t b) { return a + b; }

template <class T>
__device__ __forceinline__ T warp_reduce(T v, T (*op)(T, T)) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Reduce v over the CTA with `op`; `identity` fills the lanes past the warp
// count in the second stage.
template <class T>
__device__ __forceinline__ T block_reduce(T v, T (*op)(T, T), T identity, T *smem) {
    v = warp_reduce(v, op);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) smem[warp] = v;
    __syncthreads();
    if (warp == 0) {
        v = warp_reduce(lane < THREADS / 32 ? smem[lane] : identity, op);
        if (lane == 0) smem[0] = v;
    }
    __syncthreads();
    return smem[0];
}

struct Args {
    const float *w;
    const float *s_in;
    const float *s_out;
    int N, K, bits, scheme;
    uint8_t *packed;
    int32_t *colsum;
    float *sw;
    int32_t *zw;
    float *stats;  // [2N]: row minimum, row maximum (both including 0)
    int vec;       // K % 4 == 0, w and s_in 16-byte aligned, packed rows 4-byte (int8) /
                   // 2-byte (int4) aligned
};

// One launch's linears: job j's rows are CTAs block_begin[j] ..
// block_begin[j + 1] - 1, ROWS rows each; tensor_jobs lists the per-tensor
// jobs (pass 2 gives each one CTA).
struct Batch {
    Args job[FOLD_MAX_JOBS];
    int block_begin[FOLD_MAX_JOBS + 1];
    int tensor_jobs[FOLD_MAX_JOBS];
    int count, ntensor;
};

// The job of row block `blk` and the first row of that block within the job.
__device__ __forceinline__ int job_of(const Batch &B, int blk, int &row0) {
    int j = 0;
    while (j + 1 < B.count && blk >= B.block_begin[j + 1]) ++j;
    row0 = (blk - B.block_begin[j]) * ROWS;
    return j;
}

// Calls f(q, v) for every group q of four folded weights of row `row4` that
// this lane owns (q = lane, lane + 32, ...), with the group's loads issued
// UNROLL groups at a time.
template <class F>
__device__ __forceinline__ void for_each_four(const float4 *row4, const float4 *s4, int K4,
                                              bool has_out, float so, int lane, F &&f) {
    const float4 zero4 = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    for (int q0 = lane; q0 < K4; q0 += UNROLL * 32) {
        float4 wv[UNROLL], sv[UNROLL];
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int q = q0 + 32 * u;
            wv[u] = q < K4 ? __ldg(row4 + q) : zero4;
            sv[u] = (s4 && q < K4) ? __ldg(s4 + q) : zero4;
        }
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int q = q0 + 32 * u;
            if (q < K4) {
                float v[4];
                fold_four(wv[u], sv[u], s4 != nullptr, has_out, so, v);
                f(q, v);
            }
        }
    }
}

// Pass 1: lo = min(min_k w'[n][k], 0), hi = max(max_k w'[n][k], 0) per row.
__device__ __forceinline__ void row_stats(const Args &a, int n, int lane) {
    const float *row = a.w + (size_t)n * (size_t)a.K;
    const bool has_out = a.s_out != nullptr;
    const float so = has_out ? __ldg(a.s_out + n) : 1.0f;
    float lo = 0.0f, hi = 0.0f;
    if (a.vec) {
        for_each_four(reinterpret_cast<const float4 *>(row),
                      reinterpret_cast<const float4 *>(a.s_in), a.K >> 2, has_out, so, lane,
                      [&](int, const float *v) {
#pragma unroll
                          for (int e = 0; e < 4; ++e) lo = fminf(lo, v[e]), hi = fmaxf(hi, v[e]);
                      });
    } else {
        for (int k = lane; k < a.K; k += 32) {
            const float v = fold_one(__ldg(row + k), a.s_in, k, has_out, so);
            lo = fminf(lo, v);
            hi = fmaxf(hi, v);
        }
    }
    lo = warp_reduce<float>(lo, fmin_op);
    hi = warp_reduce<float>(hi, fmax_op);
    if (lane == 0) {
        a.stats[2 * n] = lo;
        a.stats[2 * n + 1] = hi;
    }
}

__global__ void __launch_bounds__(THREADS) row_stats_kernel(const __grid_constant__ Batch B) {
    griddep_launch_dependents();  // pass 2 / 3 wait for this grid before reading
    int row0;
    const int j = job_of(B, blockIdx.x, row0);
    const Args a = B.job[j];
    const int n = row0 + (threadIdx.x >> 5);
    if (n < a.N) row_stats(a, n, threadIdx.x & 31);
}

// Pass 2 (per tensor): the tensor's lo / hi into stats[0], stats[1].
__global__ void __launch_bounds__(THREADS) tensor_stats_kernel(const __grid_constant__ Batch B) {
    __shared__ float red[THREADS / 32];
    griddep_launch_dependents();
    const Args a = B.job[B.tensor_jobs[blockIdx.x]];
    griddep_wait();  // the row statistics of pass 1
    float lo = 0.0f, hi = 0.0f;
    for (int n = threadIdx.x; n < a.N; n += THREADS) {
        lo = fminf(lo, a.stats[2 * n]);
        hi = fmaxf(hi, a.stats[2 * n + 1]);
    }
    lo = block_reduce<float>(lo, fmin_op, 0.0f, red);
    hi = block_reduce<float>(hi, fmax_op, 0.0f, red);
    if (threadIdx.x == 0) {
        a.stats[0] = lo;
        a.stats[1] = hi;
    }
}

// Pass 3: scale and zero point of the row (or tensor), codes, packing, colsum.
__device__ __forceinline__ void quantize_row(const Args &a, int n, int lane) {
    const float *row = a.w + (size_t)n * (size_t)a.K;
    const bool has_out = a.s_out != nullptr;
    const float so = has_out ? __ldg(a.s_out + n) : 1.0f;
    const int j = a.scheme == 2 ? 0 : n;
    const float lo = a.stats[2 * j], hi = a.stats[2 * j + 1];
    const int32_t qmin = a.bits == 8 ? -128 : -8, qmax = a.bits == 8 ? 127 : 7;
    float scale;
    int32_t zero = 0;
    if (a.scheme == 0) {
        float amax = -lo > hi ? -lo : hi;
        if (!(amax > 0.0f)) amax = 1e-8f;
        scale = __fdiv_rn(amax, (float)qmax);
    } else {
        float span = __fsub_rn(hi, lo);
        if (!(span > 0.0f)) span = 1e-8f;
        scale = __fdiv_rn(span, (float)(qmax - qmin));
        const float zf = rintf(__fsub_rn((float)qmin, __fdiv_rn(lo, scale)));
        zero = (int32_t)fminf(fmaxf(zf, (float)qmin), (float)qmax);
    }
    const int32_t cmin = (a.scheme == 0 && a.bits == 8) ? -qmax : qmin;
    const float rscale = __frcp_rn(scale);
    const bool recip_ok = scale < 0x1p100f;
    int32_t sum = 0;
    if (a.vec) {
        uint8_t *dst = a.packed + (size_t)n * (size_t)(a.bits == 8 ? a.K : a.K / 2);
        for_each_four(reinterpret_cast<const float4 *>(row),
                      reinterpret_cast<const float4 *>(a.s_in), a.K >> 2, has_out, so, lane,
                      [&](int q, const float *v) {
                          int32_t c[4];
#pragma unroll
                          for (int e = 0; e < 4; ++e) {
                              c[e] = code_of(v[e], scale, rscale, recip_ok, zero, cmin, qmax);
                              sum += c[e];
                          }
                          if (a.bits == 8) {
                              reinterpret_cast<uint32_t *>(dst)[q] =
                                  (uint32_t)(c[0] & 0xFF) | (uint32_t)(c[1] & 0xFF) << 8 |
                                  (uint32_t)(c[2] & 0xFF) << 16 | (uint32_t)(c[3] & 0xFF) << 24;
                          } else {  // bytes 2q, 2q + 1: low nibble = even k
                              reinterpret_cast<uint16_t *>(dst)[q] =
                                  (uint16_t)((c[0] & 0x0F) | (c[1] & 0x0F) << 4 |
                                             (c[2] & 0x0F) << 8 | (c[3] & 0x0F) << 12);
                          }
                      });
    } else if (a.bits == 8) {
        uint8_t *dst = a.packed + (size_t)n * (size_t)a.K;
        for (int k = lane; k < a.K; k += 32) {
            const int32_t c = code_of(fold_one(__ldg(row + k), a.s_in, k, has_out, so), scale,
                                      rscale, recip_ok, zero, cmin, qmax);
            dst[k] = (uint8_t)c;
            sum += c;
        }
    } else {
        uint8_t *dst = a.packed + (size_t)n * (size_t)(a.K / 2);
        for (int p = lane; p < a.K / 2; p += 32) {
            int32_t c[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int k = 2 * p + e;
                c[e] = code_of(fold_one(__ldg(row + k), a.s_in, k, has_out, so), scale, rscale,
                               recip_ok, zero, cmin, qmax);
            }
            dst[p] = (uint8_t)((c[0] & 0x0F) | ((c[1] & 0x0F) << 4));
            sum += c[0] + c[1];
        }
    }
    sum = warp_reduce<int32_t>(sum, iadd_op);
    if (lane == 0) {
        a.colsum[n] = sum;
        a.sw[n] = scale;
        if (a.zw) a.zw[n] = zero;
    }
}

// Row blocks in the reverse order of pass 1 (the last ones read are in L2).
__global__ void __launch_bounds__(THREADS) quantize_pack_kernel(const __grid_constant__ Batch B) {
    int row0;
    const int j = job_of(B, (int)(gridDim.x - 1 - blockIdx.x), row0);
    const Args a = B.job[j];
    const int n = row0 + (threadIdx.x >> 5);
    griddep_wait();  // the statistics of pass 1 (and 2)
    if (n < a.N) quantize_row(a, n, threadIdx.x & 31);
}

}  // namespace fold

// Arguments validated by mq_fold_quantize_pack(_batch) (mq_host.cpp).
int launch_fold(const FoldJob *jobs, int count, void *stream) {
    using namespace fold;
    if (count < 1 || count > FOLD_MAX_JOBS) return MQ_ERR_INVALID_ARG;
    const auto aligned = [](const void *p, uintptr_t b) {
        return (reinterpret_cast<uintptr_t>(p) & (b - 1)) == 0;
    };
    Batch B{};
    B.count = count;
    int blocks = 0;
    for (int j = 0; j < count; ++j) {
        const FoldJob &f = jobs[j];
        const int vec = f.K % 4 == 0 && aligned(f.w, 16) && aligned(f.s_in, 16) &&
                        aligned(f.packed, f.bits == 8 ? 4 : 2);
        B.job[j] = Args{f.w, f.s_in, f.s_out, f.N, f.K, f.bits, f.scheme,
                        static_cast<uint8_t *>(f.packed), f.colsum, f.sw, f.zw, f.stats, vec};
        B.block_begin[j] = blocks;
        blocks += f.N / ROWS + (f.N % ROWS != 0);
        if (f.scheme == 2 && f.N > 0) B.tensor_jobs[B.ntensor++] = j;
    }
    B.block_begin[count] = blocks;
    if (blocks == 0) return MQ_OK;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    auto launch = [&](void (*k)(Batch), int grid, bool pdl) {
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)grid, 1, 1);
        cfg.blockDim = dim3(THREADS, 1, 1);
        cfg.stream = s;
        cfg.attrs = pdl ? attr : nullptr;
        cfg.numAttrs = pdl ? 1 : 0;
        return cudaLaunchKernelEx(&cfg, k, B) == cudaSuccess;
    };
    // pass 1 in plain stream order (w may be the previous kernel's output)
    bool ok = launch(row_stats_kernel, blocks, false);
    if (ok && B.ntensor) ok = launch(tensor_stats_kernel, B.ntensor, true);
    if (ok) ok = launch(quantize_pack_kernel, blocks, true);
    return ok ? MQ_OK : MQ_ERR_CUDA;
}

}  // namespace mq
