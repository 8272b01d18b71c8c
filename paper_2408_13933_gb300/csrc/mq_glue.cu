// mq_glue.cu -- boundary quantizers between the float, int16 and int8
// domains of an integer block: the static per-tensor activation quantizer
// (eqs. 2-4 forward, Sec. 4.2), its inverse, and fixed-point requantization
// between int8 and int16 codes (the 8-bit linears' activations meet the
// 16-bit activations kept around non-linear operators, Sec. 4.1).
//
// All three are elementwise and bound by HBM bandwidth: each thread takes 16
// elements per step with 16-byte loads and stores (a scalar path serves
// unaligned pointers and the tail), in a grid-stride loop over a grid of a
// few CTAs per SM.  Launches use programmatic dependent launch: the input may
// be the previous kernel's output, so nothing is read before griddep_wait.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "mq_internal.h"
#include "mq_ptx.cuh"

namespace mq {
namespace glue {

constexpr int THREADS = 256;
constexpr int VEC = 16;  // elements per thread per step

enum Kind { QUANTIZE = 0, DEQUANTIZE = 1, REQUANTIZE = 2 };

struct Args {
    const void *in;
    void *out;
    int64_t n;
    float alpha;  // quantize / dequantize
    int32_t zin;  // zero point of the input codes (dequantize, requantize)
    int32_t zout; // zero point of the output codes (quantize, requantize)
    int32_t m0, shift;  // requantize
    int32_t lo, hi;     // output code range
};

// Element loads (widened to f32 or int32) and stores.
template <int T>
__device__ __forceinline__ float load_f(const void *p, int64_t i);
template <>
__device__ __forceinline__ float load_f<MQ_TYPE_F32>(const void *p, int64_t i) {
    return static_cast<const float *>(p)[i];
}
template <>
__device__ __forceinline__ float load_f<MQ_TYPE_F16>(const void *p, int64_t i) {
    return __half2float(static_cast<const __half *>(p)[i]);
}
template <>
__device__ __forceinline__ float load_f<MQ_TYPE_BF16>(const void *p, int64_t i) {
    return __bfloat162float(static_cast<const __nv_bfloat16 *>(p)[i]);
}
template <int T>
__device__ __forceinline__ int32_t load_i(const void *p, int64_t i) {
    return T == MQ_TYPE_I8 ? (int32_t) static_cast<const int8_t *>(p)[i]
                           : (int32_t) static_cast<const int16_t *>(p)[i];
}
template <int T>
__device__ __forceinline__ void store_i(void *p, int64_t i, int32_t v) {
    if (T == MQ_TYPE_I8)
        static_cast<int8_t *>(p)[i] = (int8_t)v;
    else
        static_cast<int16_t *>(p)[i] = (int16_t)v;
}

__host__ __device__ constexpr int size_of(int t) {
    return t == MQ_TYPE_F32 ? 4 : (t == MQ_TYPE_I8 ? 1 : 2);
}

// One element.  Quantize: rint of the correctly rounded f32 quotient (ties
// to even), plus the zero point, saturated; NaN gives the zero point.
// Dequantize: (q - z) is exact in f32, the product is rounded once.
// Requantize: floor(((q - zx) M0 + 2^(s-1)) / 2^s) in int64 (|.| < 2^62).
template <int KIND>
__device__ __forceinline__ int32_t code_of(float xf, int32_t xi, const Args &a) {
    if (KIND == QUANTIZE) {
        const float q = __fdiv_rn(xf, a.alpha);
        if (q != q) return a.zout;
        const float t = rintf(q) + (float)a.zout;
        return (int32_t)fminf(fmaxf(t, (float)a.lo), (float)a.hi);
    }
    // |q - zx| < 2^17.  With v = (q - zx) M0 = hi 2^32 + lo (lo unsigned): for
    // shift >= 33 the quotient is (hi + 2^(shift-33)) >> (shift-32) exactly
    // (lo < 2^32 cannot carry across a multiple of 2^(shift-32)); for 32 it is
    // hi + (lo >> 31); smaller shifts take int64 (|v| < 2^48).
    const int32_t c = xi - a.zin;
    int32_t r;
    if (a.shift >= 33) {
        r = (__mulhi(c, a.m0) + (1 << (a.shift - 33))) >> (a.shift - 32);
    } else if (a.shift == 32) {
        r = __mulhi(c, a.m0) + (int32_t)(((uint32_t)c * (uint32_t)a.m0) >> 31);
    } else {
        const int64_t v = ((int64_t)c * (int64_t)a.m0 + ((int64_t)1 << (a.shift - 1))) >> a.shift;
        r = (int32_t)max((int64_t)-(1 << 20), min((int64_t)(1 << 20), v));
    }
    return max(a.lo, min(a.hi, a.zout + r));
}

template <int KIND, int TIN, int TOUT>
__device__ __forceinline__ void one(const Args &a, int64_t i) {
    if (KIND == QUANTIZE) {
        store_i<TOUT>(a.out, i, code_of<QUANTIZE>(load_f<TIN>(a.in, i), 0, a));
    } else if (KIND == DEQUANTIZE) {
        static_cast<float *>(a.out)[i] = __fmul_rn((float)(load_i<TIN>(a.in, i) - a.zin), a.alpha);
    } else {
        store_i<TOUT>(a.out, i, code_of<REQUANTIZE>(0.f, load_i<TIN>(a.in, i), a));
    }
}

// Element e of a vector of 32-bit words, widened.
template <int T>
__device__ __forceinline__ float word_f(const uint32_t *w, int e) {
    if (T == MQ_TYPE_F32) return __uint_as_float(w[e]);
    const uint32_t h = (w[e >> 1] >> (16 * (e & 1))) & 0xFFFFu;
    if (T == MQ_TYPE_BF16) return __uint_as_float(h << 16);
    return __half2float(__ushort_as_half((unsigned short)h));
}
template <int T>
__device__ __forceinline__ int32_t word_i(const uint32_t *w, int e) {
    if (T == MQ_TYPE_I8) return (int32_t)(int8_t)(w[e >> 2] >> (8 * (e & 3)));
    return (int32_t)(int16_t)(w[e >> 1] >> (16 * (e & 1)));
}

// 16 elements from 16-byte aligned vectors: the input as VEC * size / 16
// uint4 loads (streaming), the output packed into words and stored likewise.
template <int KIND, int TIN, int TOUT>
__device__ __forceinline__ void vec16(const Args &a, int64_t i0) {
    constexpr int IN_W = VEC * size_of(TIN) / 4, OUT_W = VEC * size_of(TOUT) / 4;
    uint32_t in[IN_W];
    const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const uint8_t *>(a.in) +
                                                       i0 * size_of(TIN));
#pragma unroll
    for (int w = 0; w < IN_W / 4; ++w) {
        const uint4 v = __ldcs(src + w);
        in[4 * w] = v.x;
        in[4 * w + 1] = v.y;
        in[4 * w + 2] = v.z;
        in[4 * w + 3] = v.w;
    }
    uint32_t out[OUT_W];
#pragma unroll
    for (int w = 0; w < OUT_W; ++w) out[w] = 0u;
#pragma unroll
    for (int e = 0; e < VEC; ++e) {
        if (KIND == DEQUANTIZE) {
            out[e] = __float_as_uint(__fmul_rn((float)(word_i<TIN>(in, e) - a.zin), a.alpha));
        } else {
            const int32_t c = KIND == QUANTIZE ? code_of<QUANTIZE>(word_f<TIN>(in, e), 0, a)
                                               : code_of<REQUANTIZE>(0.f, word_i<TIN>(in, e), a);
            if (TOUT == MQ_TYPE_I8)
                out[e >> 2] |= ((uint32_t)c & 0xFFu) << (8 * (e & 3));
            else
                out[e >> 1] |= ((uint32_t)c & 0xFFFFu) << (16 * (e & 1));
        }
    }
    uint4 *dst = reinterpret_cast<uint4 *>(static_cast<uint8_t *>(a.out) + i0 * size_of(TOUT));
#pragma unroll
    for (int w = 0; w < OUT_W / 4; ++w)
        __stcs(dst + w, make_uint4(out[4 * w], out[4 * w + 1], out[4 * w + 2], out[4 * w + 3]));
}

template <int KIND, int TIN, int TOUT, bool VECTOR>
__global__ void __launch_bounds__(THREADS) glue_kernel(const Args a) {
    griddep_wait();
    griddep_launch_dependents();
    const int64_t stride = (int64_t)gridDim.x * THREADS;
    const int64_t tid = (int64_t)blockIdx.x * THREADS + threadIdx.x;
    if (VECTOR) {
        const int64_t nvec = a.n / VEC;
        for (int64_t v = tid; v < nvec; v += stride) vec16<KIND, TIN, TOUT>(a, v * VEC);
        for (int64_t i = nvec * VEC + tid; i < a.n; i += stride) one<KIND, TIN, TOUT>(a, i);
    } else {
        for (int64_t i = tid; i < a.n; i += stride) one<KIND, TIN, TOUT>(a, i);
    }
}

template <int KIND, int TIN, int TOUT>
int launch_t(const Args &a, bool vector, cudaStream_t stream) {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MQ_ERR_CUDA;
    const int64_t per_block = (int64_t)THREADS * (vector ? VEC : 1);
    int64_t blocks = (a.n + per_block - 1) / per_block;
    const int64_t cap = (int64_t)sms * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3((unsigned)blocks, 1, 1);
    cfg.blockDim = dim3(THREADS, 1, 1);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = vector ? cudaLaunchKernelEx(&cfg, glue_kernel<KIND, TIN, TOUT, true>, a)
                                 : cudaLaunchKernelEx(&cfg, glue_kernel<KIND, TIN, TOUT, false>, a);
    return e == cudaSuccess ? MQ_OK : MQ_ERR_CUDA;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }


// dst[c][r] = src[r][c] through a 32 x 32 byte tile in shared memory (rows
// padded to 33 bytes): coalesced reads along src rows, coalesced writes along
// dst rows.  Launched with programmatic dependent launch (src is read after
// griddep_wait).
__global__ void __launch_bounds__(256) transpose_i8_kernel(const int8_t *__restrict__ src, int rows,
                                                           int cols, int lds,
                                                           int8_t *__restrict__ dst, int ldd) {
    __shared__ int8_t tile[32][33];
    griddep_wait();
    griddep_launch_dependents();
    const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 32 x 8 threads
#pragma unroll
    for (int i = 0; i < 32; i += 8) {
        const int r = r0 + ty + i, c = c0 + tx;
        if (r < rows && c < cols) tile[ty + i][tx] = src[(size_t)r * (size_t)lds + c];
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < 32; i += 8) {
        const int c = c0 + ty + i, r = r0 + tx;
        if (r < rows && c < cols) dst[(size_t)c * (size_t)ldd + r] = tile[tx][ty + i];
    }
}

}  // namespace glue

int launch_transpose_i8(const int8_t *src, int rows, int cols, int lds, int8_t *dst, int ldd,
                        void *stream) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3((unsigned)((cols + 31) / 32), (unsigned)((rows + 31) / 32), 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cfg.gridDim.y > 65535) return MQ_ERR_UNSUPPORTED_SHAPE;
    return cudaLaunchKernelEx(&cfg, glue::transpose_i8_kernel, src, rows, cols, lds, dst, ldd) ==
                   cudaSuccess
               ? MQ_OK
               : MQ_ERR_CUDA;
}

// Arguments are validated by the host entry points (mq_host.cpp).
int launch_glue(int kind, int in_type, int out_type, const void *in, void *out, int64_t n,
                float alpha, int32_t zin, int32_t zout, int32_t m0, int32_t shift, int32_t lo,
                int32_t hi, void *stream) {
    using namespace glue;
    if (n == 0) return MQ_OK;
    Args a{in, out, n, alpha, zin, zout, m0, shift, lo, hi};
    const bool vec = aligned16(in) && aligned16(out);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
#define MQ_GLUE_CASE(K, TI, TO) \
    if (kind == K && in_type == TI && out_type == TO) return launch_t<K, TI, TO>(a, vec, s);
    MQ_GLUE_CASE(QUANTIZE, MQ_TYPE_F32, MQ_TYPE_I8)
    MQ_GLUE_CASE(QUANTIZE, MQ_TYPE_F32, MQ_TYPE_I16)
    MQ_GLUE_CASE(QUANTIZE, MQ_TYPE_F16, MQ_TYPE_I8)
    MQ_GLUE_CASE(QUANTIZE, MQ_TYPE_F16, MQ_TYPE_I16)
    MQ_GLUE_CASE(QUANTIZE, MQ_TYPE_BF16, MQ_TYPE_I8)
    MQ_GLUE_CASE(QUANTIZE, MQ_TYPE_BF16, MQ_TYPE_I16)
    MQ_GLUE_CASE(DEQUANTIZE, MQ_TYPE_I8, MQ_TYPE_F32)
    MQ_GLUE_CASE(DEQUANTIZE, MQ_TYPE_I16, MQ_TYPE_F32)
    MQ_GLUE_CASE(REQUANTIZE, MQ_TYPE_I8, MQ_TYPE_I8)
    MQ_GLUE_CASE(REQUANTIZE, MQ_TYPE_I8, MQ_TYPE_I16)
    MQ_GLUE_CASE(REQUANTIZE, MQ_TYPE_I16, MQ_TYPE_I8)
    MQ_GLUE_CASE(REQUANTIZE, MQ_TYPE_I16, MQ_TYPE_I16)
#undef MQ_GLUE_CASE
    return MQ_ERR_INVALID_ARG;
}

}  // namespace mq
