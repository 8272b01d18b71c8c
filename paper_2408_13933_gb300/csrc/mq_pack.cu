// mq_pack.cu -- device-side weight packing and colsum, plus the library's
// device status word.
//
// colsum[n] = sum_k w[n][k] is the per-channel term of the zero-point
// correction sum((x - zx) w) = sum(x w) - zx * colsum (the offset of eq. 4
// applied to the layer input).  int4 packing: byte j of row n holds k = 2j in
// bits 0-3 and k = 2j+1 in bits 4-7, two's complement.
#include <cuda_runtime.h>

#include "mq_internal.h"
#include "mq_ptx.cuh"

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
constexpr int LOADS = 8;           // 16-byte loads in flight per lane

struct Params {
    RowsumJob job[ROWSUM_MAX_JOBS];
    int32_t block_begin[ROWSUM_MAX_JOBS + 1];  // first block of each job, then the total
    int32_t count;
};

// out[m] = sum_k x[m][k] for every job; K and ldx are multiples of 16 and x
// is 16-byte aligned (the library's validation), so every load is a whole
// uint4.  Launched with programmatic stream serialization: x may be the output
// of the previous kernel in the stream, so nothing is read before
// griddep_wait; a library kernel that follows reads `out` (a colsum) only
// after its own griddep_wait, i.e. after this grid has completed.
__global__ void __launch_bounds__(ROWS_PER_BLOCK * 32) rowsum_kernel(const __grid_constant__ Params P) {
    griddep_wait();
    griddep_launch_dependents();
    int j = 0;
    while (j + 1 < P.count && (int)blockIdx.x >= P.block_begin[j + 1]) ++j;
    const RowsumJob &q = P.job[j];
    const int row = ((int)blockIdx.x - P.block_begin[j]) * ROWS_PER_BLOCK + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= q.M) return;
    const uint4 *r = reinterpret_cast<const uint4 *>(q.x + (size_t)row * (size_t)q.ldx);
    const int n16 = q.K >> 4;  // 16-byte chunks of the row
    int acc = 0;
    // LOADS chunks per lane in flight per round: a row of K <= 4096 takes one
    // round of memory latency
    for (int base = lane; base < n16; base += 32 * LOADS) {
        uint4 v[LOADS];
#pragma unroll
        for (int u = 0; u < LOADS; ++u) {
            const int i = base + 32 * u;
            v[u] = i < n16 ? __ldg(r + i) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < LOADS; ++u) {
            acc = __dp4a((int)v[u].x, 0x01010101, acc);
            acc = __dp4a((int)v[u].y, 0x01010101, acc);
            acc = __dp4a((int)v[u].z, 0x01010101, acc);
            acc = __dp4a((int)v[u].w, 0x01010101, acc);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) q.out[row] = acc;
}

}  // namespace rowsum

int launch_rowsum(const RowsumJob *jobs, int count, void *stream) {
    for (int base = 0; base < count; base += ROWSUM_MAX_JOBS) {
        rowsum::Params P{};
        const int n = count - base < ROWSUM_MAX_JOBS ? count - base : ROWSUM_MAX_JOBS;
        int64_t blocks = 0;
        for (int i = 0; i < n; ++i) {
            P.job[i] = jobs[base + i];
            P.block_begin[i] = (int32_t)blocks;
            blocks += (jobs[base + i].M + rowsum::ROWS_PER_BLOCK - 1) / rowsum::ROWS_PER_BLOCK;
        }
        if (blocks == 0) continue;
        if (blocks > 0x7fffffffLL) return MQ_ERR_UNSUPPORTED_SHAPE;
        P.block_begin[n] = (int32_t)blocks;
        P.count = n;
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)blocks, 1, 1);
        cfg.blockDim = dim3(rowsum::ROWS_PER_BLOCK * 32, 1, 1);
        cfg.dynamicSmemBytes = 0;
        cfg.stream = static_cast<cudaStream_t>(stream);
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaLaunchKernelEx(&cfg, rowsum::rowsum_kernel, P) != cudaSuccess) return MQ_ERR_CUDA;
    }
    return MQ_OK;
}

namespace split16 {

constexpr int THREADS = 256;

struct Params {
    SplitJob job[SPLIT_MAX_JOBS];
    int64_t block_begin[SPLIT_MAX_JOBS + 1];  // first block of each job, then the total
    int32_t count;
};

// The two int8 planes of 16-bit activation codes: with hi the signed high
// byte and lo the unsigned low byte, x = 256 hi + (lo - 128) + 128, so row 2m
// of `out` gets the hi bytes of x row m and row 2m + 1 the bytes lo ^ 0x80
// (= lo - 128 as a signed byte).  One thread per 16 codes of a row (two
// 16-byte loads, two 16-byte stores); K is a multiple of 16, ldx of 8, and x
// and out are 16-byte aligned (the library's validation).  Launched with
// programmatic stream serialization: x is read only after griddep_wait.
__global__ void __launch_bounds__(THREADS) split16_kernel(const __grid_constant__ Params P) {
    griddep_wait();
    griddep_launch_dependents();
    int j = 0;
    while (j + 1 < P.count && (int64_t)blockIdx.x >= P.block_begin[j + 1]) ++j;
    const SplitJob &q = P.job[j];
    const int64_t g = ((int64_t)blockIdx.x - P.block_begin[j]) * THREADS + threadIdx.x;
    const int per_row = q.K >> 4;
    const int64_t row = g / per_row;
    if (row >= q.M) return;
    const int c = (int)(g - row * per_row);
    const uint4 *src = reinterpret_cast<const uint4 *>(q.x + (size_t)row * (size_t)q.ldx + 16 * c);
    const uint4 a = __ldg(src), b = __ldg(src + 1);
    // bytes 1, 3 of each 32-bit word are the high bytes of its two codes,
    // bytes 0, 2 the low bytes
    uint4 hi, lo;
    hi.x = __byte_perm(a.x, a.y, 0x7531);
    hi.y = __byte_perm(a.z, a.w, 0x7531);
    hi.z = __byte_perm(b.x, b.y, 0x7531);
    hi.w = __byte_perm(b.z, b.w, 0x7531);
    lo.x = __byte_perm(a.x, a.y, 0x6420) ^ 0x80808080u;
    lo.y = __byte_perm(a.z, a.w, 0x6420) ^ 0x80808080u;
    lo.z = __byte_perm(b.x, b.y, 0x6420) ^ 0x80808080u;
    lo.w = __byte_perm(b.z, b.w, 0x6420) ^ 0x80808080u;
    int8_t *dst = q.out + (size_t)(2 * row) * (size_t)q.K + 16 * c;
    *reinterpret_cast<uint4 *>(dst) = hi;
    *reinterpret_cast<uint4 *>(dst + q.K) = lo;
}

}  // namespace split16

int launch_split16(const SplitJob *jobs, int count, void *stream) {
    for (int base = 0; base < count; base += SPLIT_MAX_JOBS) {
        split16::Params P{};
        const int n = count - base < SPLIT_MAX_JOBS ? count - base : SPLIT_MAX_JOBS;
        int64_t blocks = 0;
        for (int i = 0; i < n; ++i) {
            P.job[i] = jobs[base + i];
            P.block_begin[i] = blocks;
            const int64_t groups = (int64_t)jobs[base + i].M * (jobs[base + i].K / 16);
            blocks += (groups + split16::THREADS - 1) / split16::THREADS;
        }
        if (blocks == 0) continue;
        if (blocks > 0x7fffffffLL) return MQ_ERR_UNSUPPORTED_SHAPE;
        P.block_begin[n] = blocks;
        P.count = n;
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)blocks, 1, 1);
        cfg.blockDim = dim3(split16::THREADS, 1, 1);
        cfg.dynamicSmemBytes = 0;
        cfg.stream = static_cast<cudaStream_t>(stream);
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaLaunchKernelEx(&cfg, split16::split16_kernel, P) != cudaSuccess)
            return MQ_ERR_CUDA;
    }
    return MQ_OK;
}

}  // namespace mq
