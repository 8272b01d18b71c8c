// mq_pack.cu -- device-side weight packing and colsum, plus the library's
// device status word.
//
// colsum[n] = sum_k w[n][k] is the per-channel term of the zero-point
// correction sum((x - zx) w) = sum(x w) - zx * colsum (the offset of eq. 4
// applied to the layer input).  int4 packing: byte j of row n holds k = 2j in
// bits 0-3 and k = 2j+1 in bits 4-7, two's complement.
#include <cuda_runtime.h>

#include "mq_internal.h"

namespace mq {

__device__ int g_device_status = 0;
__device__ int g_pack_status = 0;

namespace {
constexpr int MAX_DEVICES = 64;

// Host code cannot use the symbol itself as an address: resolve it once per
// device, with that device current.
int *symbol_ptr(int which) {
    static int *cached[2][MAX_DEVICES] = {{nullptr}};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= MAX_DEVICES) return nullptr;
    if (!cached[which][dev]) {
        void *p = nullptr;
        const cudaError_t e = which == 0 ? cudaGetSymbolAddress(&p, g_device_status)
                                         : cudaGetSymbolAddress(&p, g_pack_status);
        if (e != cudaSuccess) return nullptr;
        cached[which][dev] = static_cast<int *>(p);
    }
    return cached[which][dev];
}
}  // namespace

int *device_status_ptr() { return symbol_ptr(0); }
int *pack_status_ptr() { return symbol_ptr(1); }

namespace pack {

constexpr int THREADS = 256;

// One CTA per weight row.
__global__ void __launch_bounds__(THREADS) pack_kernel(const int8_t *__restrict__ w, int N, int K,
                                                       int bits, uint8_t *__restrict__ packed,
                                                       int32_t *__restrict__ colsum,
                                                       int *status) {
    __shared__ int32_t part[THREADS / 32];
    const int n = blockIdx.x;
    const int8_t *row = w + (size_t)n * (size_t)K;
    int32_t sum = 0;
    bool bad = false;
    if (bits == 8) {
        uint8_t *dst = packed + (size_t)n * (size_t)K;
        for (int k = threadIdx.x; k < K; k += THREADS) {
            const int8_t v = row[k];
            dst[k] = (uint8_t)v;
            sum += v;
        }
    } else {
        uint8_t *dst = packed + (size_t)n * (size_t)(K / 2);
        for (int j = threadIdx.x; j < K / 2; j += THREADS) {
            const int lo = row[2 * j], hi = row[2 * j + 1];
            bad |= lo < -8 || lo > 7 || hi < -8 || hi > 7;
            dst[j] = (uint8_t)((lo & 0x0F) | ((hi & 0x0F) << 4));
            sum += lo + hi;
        }
    }
    if (bad) atomicOr(status, MQ_DEVICE_STATUS_PACK_RANGE);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = sum;
    __syncthreads();
    if (threadIdx.x == 0) {
        int32_t s = 0;
        for (int i = 0; i < THREADS / 32; ++i) s += part[i];
        colsum[n] = s;
    }
}

}  // namespace pack

int launch_pack(const int8_t *w, int N, int K, int bits, void *packed, int32_t *colsum,
                int *status, void *stream) {
    if (N == 0) return MQ_OK;
    pack::pack_kernel<<<N, pack::THREADS, 0, static_cast<cudaStream_t>(stream)>>>(
        w, N, K, bits, static_cast<uint8_t *>(packed), colsum, status);
    return cudaGetLastError() == cudaSuccess ? MQ_OK : MQ_ERR_CUDA;
}

namespace rowsum {

constexpr int ROWS_PER_BLOCK = 8;  // one warp per row

// rowsum[m] = sum_k x[m][k]; K and ldx are multiples of 16 and x is 16-byte
// aligned (the library's validation), so every load is a whole uint4.
__global__ void __launch_bounds__(ROWS_PER_BLOCK * 32)
    rowsum_kernel(const int8_t *__restrict__ x, int M, int K, int ldx, int32_t *__restrict__ out) {
    const int row = blockIdx.x * ROWS_PER_BLOCK + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= M) return;
    const int8_t *r = x + (size_t)row * (size_t)ldx;
    int acc = 0;
    for (int k = lane * 16; k < K; k += 32 * 16) {
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(r + k));
        acc = __dp4a((int)v.x, 0x01010101, acc);
        acc = __dp4a((int)v.y, 0x01010101, acc);
        acc = __dp4a((int)v.z, 0x01010101, acc);
        acc = __dp4a((int)v.w, 0x01010101, acc);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) out[row] = acc;
}

}  // namespace rowsum

int launch_rowsum(const Problem *probs, int count, void *stream) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    for (int i = 0; i < count; ++i) {
        const Problem &p = probs[i];
        if (!p.rowsum || p.M <= 0) continue;
        const int blocks = (p.M + rowsum::ROWS_PER_BLOCK - 1) / rowsum::ROWS_PER_BLOCK;
        rowsum::rowsum_kernel<<<blocks, rowsum::ROWS_PER_BLOCK * 32, 0, s>>>(
            p.x, p.M, p.K, p.ldx, const_cast<int32_t *>(p.rowsum));
        if (cudaGetLastError() != cudaSuccess) return MQ_ERR_CUDA;
    }
    return MQ_OK;
}

}  // namespace mq
