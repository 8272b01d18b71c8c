// mq_noalloc.cu -- mq_linear_w4a8_noalloc: the W4A8 decode layer (1 <= M <= 16)
// with its split-K combine scratch held in a static device array of this
// library instead of a workspace the caller provides.
//
// Some callers cannot hand over device memory for a decode step: a C host
// program without a device allocator of its own, or a serving loop whose
// memory pool is sized and frozen after warm-up and must not grow (or be
// drained by a caching allocator) in the middle of token generation.  This
// entry point gives them the same result as mq_linear_w4a8 without asking for
// a workspace and without allocating one.
//
// The scratch is one fixed-size array per device (DECODE_WS_BYTES, 2.5 MB:
// per CTA of the decode grid one slot of 64 x 16 {partial sum, launch epoch}
// entries), so every call on a device shares it.
// Calls on that device must therefore not overlap: two calls on different
// streams, or from different host threads, race on the scratch and give
// wrong results.  Calls issued one after another on one stream are fine.
//
// The scratch is never cleared by a call.  It starts zeroed (a static device
// array), and the decode kernel only needs that no entry carries the current
// launch's epoch before a contributor writes it: every launch has its own
// epoch, the finishing CTA polls each entry until it carries that epoch, and
// entries left behind by an earlier launch (also one that timed out) carry an
// older one.  So nothing but the kernel itself sits between two consecutive
// decode launches, and programmatic dependent launch can overlap them.
#include <cuda_runtime.h>

#include <atomic>

#include "mq_internal.h"

namespace mq {

// The decode kernel's combine scratch: per CTA of the decode grid one slot of
// 64 x 16 {partial sum, launch epoch} entries, left zero by the kernel.
static __device__ __align__(256) int32_t g_noalloc_scratch[DECODE_WS_BYTES / sizeof(int32_t)];

namespace {

constexpr int MAX_DEVICES = 64;
std::atomic<void *> g_scratch_addr[MAX_DEVICES];

// The scratch's device address, looked up once per device with that device
// current (on the first call made on it) and cached afterwards; the same
// first call prepares both variants of the decode kernel this entry point
// launches, so that later calls do no set-up at all (e.g. inside a capture).
void *scratch_ptr() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= MAX_DEVICES) return nullptr;
    void *p = g_scratch_addr[dev].load(std::memory_order_acquire);
    if (!p) {
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
        if (prepare_decode_w4a8() != MQ_OK) return nullptr;
        g_scratch_addr[dev].store(p, std::memory_order_release);
    }
    return p;
}

bool aligned16(const void *ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

}  // namespace
}  // namespace mq

extern "C" int mq_linear_w4a8_noalloc(const int8_t *x, int M, int K, int ldx, int32_t zx,
                                      const void *packed, const int32_t *colsum, int N,
                                      const int32_t *M0, const int32_t *shift, int32_t zy,
                                      int8_t *y, int ldy, void *stream) {
    // the same argument rules as mq_linear_w4a8, then the scratch's limit
    if (M < 0 || N < 0 || K < 0) return MQ_ERR_INVALID_ARG;
    if (zx < -128 || zx > 127 || zy < -128 || zy > 127) return MQ_ERR_INVALID_ARG;
    if (K > MQ_MAX_K) return MQ_ERR_K_OVERFLOW;
    if (M > mq::DECODE_MAX_M) return MQ_ERR_UNSUPPORTED_SHAPE;  // scratch holds 16 tokens
    if (M == 0 || N == 0) return MQ_OK;                         // nothing to compute or write
    if (!colsum || !M0 || !shift || !y || ldy < N) return MQ_ERR_INVALID_ARG;
    if (K > 0) {
        if (!x || !packed || ldx < K) return MQ_ERR_INVALID_ARG;
        if (K % 32 != 0 || ldx % 16 != 0) return MQ_ERR_ALIGNMENT;
        if (!mq::aligned16(x) || !mq::aligned16(packed)) return MQ_ERR_ALIGNMENT;
    }

    void *scratch = mq::scratch_ptr();
    if (!scratch) return MQ_ERR_CUDA;

    mq::Problem p{};
    p.x = x;
    p.w = static_cast<const uint8_t *>(packed);
    p.colsum = colsum;
    p.M0 = M0;
    p.shift = shift;
    p.residual = nullptr;
    p.y = y;
    p.M = M;
    p.N = N;
    p.K = K;
    p.ldx = ldx;
    p.ldy = ldy;
    p.zx = zx;
    p.zy = zy;
    p.bits = 4;
    p.ldw = K / 2;
    return mq::launch_decode(&p, 1, scratch, stream);
}
