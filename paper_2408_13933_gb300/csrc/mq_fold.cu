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
// Three kernels: per-row minima / maxima of w' (one CTA per row), for the
// per-tensor scheme a one-CTA reduction of those to the tensor's, then
// quantization + packing + colsum (one CTA per row; w' is recomputed from w,
// which the first pass left in L2 for rows that fit).
#include <cuda_runtime.h>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {
namespace fold {

constexpr int THREADS = 256;

// w'[n][k]: multiply by s_in[k] first, then divide by s_out[n].
__device__ __forceinline__ float fold_one(float w, const float *s_in, int k, bool has_out,
                                          float s_out) {
    float v = w;
    if (s_in) v = __fmul_rn(v, __ldg(s_in + k));
    if (has_out) v = __fdiv_rn(v, s_out);
    return v;
}

// Reduce v over the CTA with `op`; `identity` fills the lanes past the warp
// count in the second stage.
template <class T>
__device__ __forceinline__ T block_reduce(T v, T (*op)(T, T), T identity, T *smem) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, o));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) smem[warp] = v;
    __syncthreads();
    if (warp == 0) {
        v = lane < THREADS / 32 ? smem[lane] : identity;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, o));
        if (lane == 0) smem[0] = v;
    }
    __syncthreads();
    return smem[0];
}

__device__ float fmin_op(float a, float b) { return fminf(a, b); }
__device__ float fmax_op(float a, float b) { return fmaxf(a, b); }
__device__ int32_t iadd_op(int32_t a, int32_t b) { return a + b; }

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
};

// Pass 1: lo = min(min_k w'[n][k], 0), hi = max(max_k w'[n][k], 0) per row.
__global__ void __launch_bounds__(THREADS) row_stats_kernel(const Args a) {
    __shared__ float red[THREADS / 32];
    const int n = blockIdx.x;
    const float *row = a.w + (size_t)n * (size_t)a.K;
    const bool has_out = a.s_out != nullptr;
    const float so = has_out ? __ldg(a.s_out + n) : 1.0f;
    float lo = 0.0f, hi = 0.0f;
    for (int k = threadIdx.x; k < a.K; k += THREADS) {
        const float v = fold_one(__ldg(row + k), a.s_in, k, has_out, so);
        lo = fminf(lo, v);
        hi = fmaxf(hi, v);
    }
    lo = block_reduce<float>(lo, fmin_op, 0.0f, red);
    hi = block_reduce<float>(hi, fmax_op, 0.0f, red);
    if (threadIdx.x == 0) {
        a.stats[2 * n] = lo;
        a.stats[2 * n + 1] = hi;
    }
}

// Pass 2 (per tensor): the tensor's lo / hi into stats[0], stats[1].
__global__ void __launch_bounds__(THREADS) tensor_stats_kernel(const Args a) {
    __shared__ float red[THREADS / 32];
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
__global__ void __launch_bounds__(THREADS) quantize_pack_kernel(const Args a) {
    __shared__ int32_t red[THREADS / 32];
    const int n = blockIdx.x;
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
    int32_t sum = 0;
    if (a.bits == 8) {
        uint8_t *dst = a.packed + (size_t)n * (size_t)a.K;
        for (int k = threadIdx.x; k < a.K; k += THREADS) {
            const float t = rintf(__fdiv_rn(fold_one(__ldg(row + k), a.s_in, k, has_out, so), scale));
            const int32_t c = (int32_t)fminf(fmaxf(__fadd_rn(t, (float)zero), (float)cmin), (float)qmax);
            dst[k] = (uint8_t)c;
            sum += c;
        }
    } else {
        uint8_t *dst = a.packed + (size_t)n * (size_t)(a.K / 2);
        for (int p = threadIdx.x; p < a.K / 2; p += THREADS) {
            int32_t c[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int k = 2 * p + e;
                const float t =
                    rintf(__fdiv_rn(fold_one(__ldg(row + k), a.s_in, k, has_out, so), scale));
                c[e] = (int32_t)fminf(fmaxf(__fadd_rn(t, (float)zero), (float)cmin), (float)qmax);
            }
            dst[p] = (uint8_t)((c[0] & 0x0F) | ((c[1] & 0x0F) << 4));
            sum += c[0] + c[1];
        }
    }
    sum = block_reduce<int32_t>(sum, iadd_op, 0, red);
    if (threadIdx.x == 0) {
        a.colsum[n] = sum;
        a.sw[n] = scale;
        if (a.zw) a.zw[n] = zero;
    }
}

}  // namespace fold

// Arguments validated by mq_fold_quantize_pack (mq_host.cpp).
int launch_fold(const float *w, int N, int K, const float *s_in, const float *s_out, int bits,
                int scheme, void *packed, int32_t *colsum, float *sw, int32_t *zw, float *stats,
                void *stream) {
    using namespace fold;
    if (N == 0) return MQ_OK;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const Args a{w, s_in, s_out, N, K, bits, scheme, static_cast<uint8_t *>(packed),
                 colsum, sw, zw, stats};
    row_stats_kernel<<<N, THREADS, 0, s>>>(a);
    if (scheme == 2) tensor_stats_kernel<<<1, THREADS, 0, s>>>(a);
    quantize_pack_kernel<<<N, THREADS, 0, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? MQ_OK : MQ_ERR_CUDA;
}

}  // namespace mq
