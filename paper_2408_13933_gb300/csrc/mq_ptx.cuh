// mq_ptx.cuh -- inline-PTX building blocks for the sm_103a kernels of libmq:
// shared-memory mbarriers, tcgen05 (TMEM allocation, MMA, commit, loads and
// stores), proxy fences and bounded waits.  Every wait in this library gives
// up after a time limit that the launcher passes in the kernel parameters
// (mq_set_wait_limit_ns, 1 second by default).
#pragma once

#include <cstdint>

#include "mq_internal.h"

namespace mq {

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}"
                 ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// As mbar_try_wait, but the thread may be suspended in hardware (not
// spinning) for up to `hint_ns` nanoseconds while the phase is incomplete; it
// resumes as soon as the phase completes.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *bar, uint32_t parity,
                                                    uint32_t hint_ns) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
        : "memory");
    return ok != 0;
}

// Wait until the phase with the given parity of `bar` has completed.  Gives up
// (returns false) when `abort` becomes non-zero or after `limit_ns`; in the
// latter case it raises `abort` and records the timeout in `status`.  The
// waiting thread sleeps in hardware between checks instead of spinning, so it
// takes no issue slots from the warps doing work.
__device__ __forceinline__ bool mq_wait_parity(uint64_t *bar, uint32_t parity,
                                               volatile int *abort, int *status,
                                               uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
        if (*abort) return false;
        if (global_timer_ns() - t0 > limit_ns) {
            *abort = 1;
            atomicOr(status, MQ_DEVICE_STATUS_TIMEOUT);
            return false;
        }
    }
}

// A bounded wait that ignores `abort`: for phases that are bound to complete
// even after the kernel gave up on its work (tensor-core operations already
// issued), which must be waited for before their operands' memory is
// released.  Gives up after `limit_ns` and records a timeout then.
__device__ __forceinline__ bool mq_wait_parity_drain(uint64_t *bar, uint32_t parity, int *status,
                                                     uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
        if (global_timer_ns() - t0 > limit_ns) {
            atomicOr(status, MQ_DEVICE_STATUS_TIMEOUT);
            return false;
        }
    }
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("{\n\t.reg .b64 st;\n\t"
                 "mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}"
                 ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}

// 2-D tiled TMA load of the box at (x, y) (x = innermost, in elements) of the
// tensor described by `map` into shared memory at `dst`; completion is
// signalled on `bar` as transaction bytes.  Elements outside the tensor are
// filled with zeros.
__device__ __forceinline__ void tma_load_2d(void *dst, const void *map, int x, int y,
                                            uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3}], [%4];"
        ::"r"(smem_u32(dst)), "l"(map), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}

// 1-D bulk copy of `bytes` (a multiple of 16; both addresses 16-byte
// aligned) from global memory into this CTA's shared memory; completion is
// signalled on `bar` as transaction bytes.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes,
                                          uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// Raise the transaction bytes the current phase of `bar` waits for, without
// arriving.
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;"
                 ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}

// Asynchronous 4-byte copy global -> shared (both 4-byte aligned).
__device__ __forceinline__ void cp_async4(void *dst, const void *src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src)
                 : "memory");
}

// The current phase of `bar` also waits for every cp.async this thread has
// issued so far (one pending arrival, taken back when they complete).
__device__ __forceinline__ void cp_async_arrive(uint64_t *bar) {
    asm volatile("cp.async.mbarrier.arrive.shared::cta.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const void *map) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(map) : "memory");
}

// Generic-proxy shared-memory writes -> visible to the async proxy (tcgen05).
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ------------------------------------------ programmatic dependent launch
// Wait until the grids this one depends on (the previous kernel in the
// stream, when launched with programmatic stream serialization) have
// completed and their memory is visible; a no-op otherwise.
__device__ __forceinline__ void griddep_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// Let the next kernel in the stream be scheduled once every CTA of this grid
// has signalled (it still waits for this grid's completion before reading).
__device__ __forceinline__ void griddep_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// One lane of the (converged, full) warp is elected: true in that lane only.
__device__ __forceinline__ bool elect_one() {
    uint32_t pred = 0;
    asm volatile(
        "{\n\t.reg .pred P;\n\t.reg .b32 r;\n\t"
        "elect.sync r|P, 0xffffffff;\n\t"
        "selp.u32 %0, 1, 0, P;\n\t}"
        : "=r"(pred));
    return pred != 0;
}

// ----------------------------------------------------------------- clusters
__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// All threads of every CTA of the cluster (release / acquire at cluster scope).
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Shared-memory address of the same variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t cluster_addr(const void *p, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
    return r;
}

// Arrive (release, cluster scope) on an mbarrier given by its cluster address.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_bar) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];"
                 ::"r"(cluster_bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// mq_wait_parity for phases completed by arrivals from other CTAs of the
// cluster (remote arrives, multicast commits): acquire at cluster scope.
__device__ __forceinline__ bool mq_wait_parity_cluster(uint64_t *bar, uint32_t parity,
                                                       volatile int *abort, int *status,
                                                       uint64_t limit_ns) {
    const uint64_t t0 = global_timer_ns();
    for (uint32_t n = 0;; ++n) {
        if (mbar_try_wait_cluster(bar, parity)) return true;
        if ((n & 15) == 15) {
            if (*abort) return false;
            if (global_timer_ns() - t0 > limit_ns) {
                *abort = 1;
                atomicOr(status, MQ_DEVICE_STATUS_TIMEOUT);
                return false;
            }
        }
    }
}

// Non-blocking 4-byte store into another CTA's shared memory that signals the
// mbarrier next to it (complete_tx of 4 bytes, release at cluster scope): a
// cheap cross-CTA "data ready" signal.  Both addresses are cluster addresses
// in the same CTA.
__device__ __forceinline__ void st_async_signal(uint32_t cluster_dst, uint32_t value,
                                                uint32_t cluster_bar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];"
                 ::"r"(cluster_dst), "r"(value), "r"(cluster_bar) : "memory");
}

// ------------------------------------------------- tcgen05, CTA-pair mode
// Every tcgen05 instruction of a kernel uses the same CTA group; libmq's
// tensor-core kernel runs on CTA pairs (cta_group::2).  Allocation and
// deallocation are collective over one warp of each CTA of the pair; the
// pair's MMAs are issued by one thread of the even CTA.
__device__ __forceinline__ void tmem_alloc2(uint32_t *dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(dst_smem)), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tmem_relinquish2() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc2(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;"
                 ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Pair MMA, kind::f16: D[tmem] (+)= A[tmem] * B[smem]^T.  A (M = 256) is split
// by rows over the pair (128 TMEM lanes in each CTA at the same address), B
// by rows (N / 2 in each CTA's shared memory at the same address), D by rows
// like A.
__device__ __forceinline__ void tc_mma2_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                               uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], [%1], %2, %3, p;\n\t}"
        ::"r"(d_tmem), "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive once on the mbarrier at `bar`'s offset in every CTA of `cta_mask`
// when every tcgen05 operation issued so far by this thread has completed.
__device__ __forceinline__ void tc_commit2_mc(uint64_t *bar, uint16_t cta_mask) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
        " [%0], %1;"
        ::"r"(smem_u32(bar)), "h"(cta_mask) : "memory");
}

__device__ __forceinline__ void tc_wait_ld() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tc_wait_st() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 32 lanes x 32 consecutive 32-bit columns: thread i of the warp receives
// lane (base lane + i), columns [col, col + 32).
__device__ __forceinline__ void tc_ld_32x32b_x32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
          "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
          "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]),
          "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]),
          "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}

__device__ __forceinline__ void tc_st_32x32b_x32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};"
        ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]),
          "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]),
          "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]),
          "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]),
          "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

__device__ __forceinline__ void tc_ld_32x32b_x16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
          "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
          "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

__device__ __forceinline__ void tc_st_32x32b_x16(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
        ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]),
          "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]),
          "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile stored with the
// 128-byte swizzle: rows of 128 bytes, 8-row groups 1024 bytes apart, tile
// base 1024-byte aligned.  Advancing along K inside the 128-byte row is done
// by adding the byte offset to the start address.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);   // start address >> 4
    d |= (uint64_t)1u << 16;                    // leading byte offset (unused here)
    d |= (uint64_t)(1024u >> 4) << 32;          // stride byte offset: 8 rows x 128 B
    d |= (uint64_t)1u << 46;                    // descriptor version for tcgen05
    d |= (uint64_t)2u << 61;                    // layout: 128-byte swizzle
    return d;
}

// Instruction descriptor, kind::f16: A and B f16, D f32, both K-major.
__host__ __device__ constexpr uint32_t idesc_f16_f32(int m, int n) {
    return (1u << 4)                          // D format: f32
           | (0u << 7) | (0u << 10)           // A, B format: f16
           | (0u << 15) | (0u << 16)          // A, B K-major
           | ((uint32_t)(n >> 3) << 17)       // N / 8
           | ((uint32_t)(m >> 4) << 24);      // M / 16
}

// ------------------------------------------------- int8 / int4 -> fp16 pairs
// Signed int8 -> f16 exactly: bias each byte to u = x + 128 (xor 0x80), build
// the f16 1024 + u with the byte as mantissa, subtract 1152.
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t r;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
    return r;
}

__device__ __forceinline__ uint32_t hsub2(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

__device__ __forceinline__ uint32_t hfma2(uint32_t a, uint32_t b, uint32_t c) {
    uint32_t r;
    asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(c));
    return r;
}

// out = mask ? (a ^ bits) : bits, bit by bit (one LOP3).
__device__ __forceinline__ uint32_t lop3_sel_xor(uint32_t a, uint32_t mask, uint32_t bits) {
    uint32_t r;
    // truth table for f(a, b=mask, c=bits) = b ? (a ^ c) : c  -> 0x6A
    asm("lop3.b32 %0, %1, %2, %3, 0x6A;" : "=r"(r) : "r"(a), "r"(mask), "r"(bits));
    return r;
}

constexpr uint32_t F16X2_1152 = 0x64806480u;  // (1152, 1152)

// Four int8 (one 32-bit word, byte i = element i) -> two f16x2 words
// (elements 0,1) and (2,3).
__device__ __forceinline__ void i8x4_to_f16x4(uint32_t w, uint32_t &lo, uint32_t &hi,
                                              uint32_t off = F16X2_1152) {
    const uint32_t u = w ^ 0x80808080u;
    lo = hsub2(prmt(u, 0x64646464u, 0x4140u), off);
    hi = hsub2(prmt(u, 0x64646464u, 0x4342u), off);
}

// The offset of i8x4_to_f16x4 that also subtracts a weight zero point z in
// [-128, 127]: (1152 + z) in both halves, f16 bits 0x6480 + z (1024 <= 1152 +
// z < 2048, where f16 steps by 1).  (1024 + u) - (1152 + z) = w - z is exact:
// both operands and the result (|w - z| <= 255) are f16 integers.
__device__ __forceinline__ uint32_t f16x2_i8_offset(int32_t z) {
    const uint32_t c = (uint32_t)(0x6480 + z);
    return (c << 16) | c;
}

// Eight int4 (one word, nibble p = element p, two's complement) -> four f16x2
// words in natural order (0,1) (2,3) (4,5) (6,7).  Byte i is copied to bytes
// 0 and 2; the low nibble of byte 0 becomes 1024 + (e + 8) in the low half,
// the high nibble of byte 2 becomes 1024 + 16 (e + 8) in the high half; one
// f16x2 FMA with per-half scale (1, 1/16) and offset (-1032, -72) gives e.
__device__ __forceinline__ void i4x8_to_f16x8(uint32_t w, uint32_t (&o)[4],
                                              uint32_t offset = 0xD480E408u /* (-1032, -72) */) {
    const uint32_t scale = 0x2C003C00u;   // (1.0, 1/16)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t t = prmt(w, 0u, 0x1111u * (uint32_t)i);
        o[i] = hfma2(lop3_sel_xor(t, 0x00F0000Fu, 0x64806408u), scale, offset);
    }
}

// The offset of i4x8_to_f16x8 that also subtracts a weight zero point z in
// [-8, 7]: (-1032 - z, -72 - z); f16 bits 0xE408 + z (1024 < 1032 + z < 2048,
// step 1) and 0xD480 + 16 z (64 <= 72 + z < 128, step 1/16).  Each half is one
// FMA whose exact value e - z (|e - z| <= 15) is an f16 integer.
__device__ __forceinline__ uint32_t f16x2_i4_offset(int32_t z) {
    return (((uint32_t)(0xD480 + 16 * z) & 0xFFFFu) << 16) | ((uint32_t)(0xE408 + z) & 0xFFFFu);
}

// Requantize one accumulator (acc = sum(x w) - zx colsum, int32):
// clamp(zy + floor((acc * M0 + 2^(s-1)) / 2^s), -128, 127).  With
// v = acc * M0 = hi * 2^32 + lo (lo unsigned): for s >= 33 the result is
// (hi + 2^(s-33)) >> (s-32) exactly (the low word cannot carry across a
// multiple of 2^(s-32)); for s == 32 it is hi + (lo >> 31); smaller shifts
// take the 64-bit path.  `s` is uniform across the warp (one column).
__device__ __forceinline__ int32_t mq_requant(int32_t acc, int32_t m0, int32_t sh, int32_t zy) {
    int32_t q;
    if (sh >= 33) {
        q = (__mulhi(acc, m0) + (1 << (sh - 33))) >> (sh - 32);
    } else if (sh == 32) {
        q = __mulhi(acc, m0) + (int32_t)(((uint32_t)acc * (uint32_t)m0) >> 31);
    } else {
        const int64_t v = ((int64_t)acc * (int64_t)m0 + ((int64_t)1 << (sh - 1))) >> sh;
        q = (int32_t)(v < -1024 ? -1024 : (v > 1024 ? 1024 : v));
    }
    return min(127, max(-128, q + zy));
}

// The 16-bit output: clamp(zy + floor((acc m0 + 2^(sh-1)) / 2^sh), -32768,
// 32767) for |acc| < 2^41, 0 <= m0 < 2^31, 1 <= sh <= 62, in int64.  For
// sh >= 16, with m0 = mh 2^16 + ml (0 <= ml < 2^16) and
// Y = acc ml + 2^(sh-1):  acc m0 + 2^(sh-1) = 2^16 (acc mh + floor(Y / 2^16))
// + (Y mod 2^16), so the quotient is (acc mh + (Y >> 16)) >> (sh - 16) (the
// dropped remainder is below 2^16 <= 2^sh; arithmetic shifts floor); every
// term stays below 2^62.  For sh < 16 the multiplier is at least 2^15, so
// |acc| >= 2^32 saturates and smaller accumulators fit a plain int64 product.
__device__ __forceinline__ int32_t mq_requant16(int64_t acc, int32_t m0, int32_t sh, int32_t zy) {
    int64_t q;
    if (sh >= 16) {
        const int64_t y = acc * (int64_t)(m0 & 0xFFFF) + ((int64_t)1 << (sh - 1));
        q = (acc * (int64_t)(m0 >> 16) + (y >> 16)) >> (sh - 16);
    } else if (acc >= ((int64_t)1 << 32) || acc <= -((int64_t)1 << 32)) {
        q = acc > 0 ? (m0 ? 131072 : 0) : (m0 ? -131072 : 0);
    } else {
        q = (acc * (int64_t)m0 + ((int64_t)1 << (sh - 1))) >> sh;
    }
    const int32_t qc = (int32_t)(q < -131072 ? -131072 : (q > 131072 ? 131072 : q));
    return min(32767, max(-32768, qc + zy));
}

}  // namespace mq
