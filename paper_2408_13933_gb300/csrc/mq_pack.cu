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

}  // namespace mq
