// mq_host.cpp -- host half of the libmq C ABI: argument validation,
// fixed-point requantization parameters, host-side packing, dispatch of
// linear problems to the prefill (tensor-core) and decode (weight-streaming)
// kernels, and device status reporting.
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstring>
#include <vector>

#include "mq_internal.h"
#include "mq_tmajor.h"

namespace mq {

namespace {
constexpr uint64_t DEFAULT_WAIT_NS = 1000000000ull;  // 1 second
std::atomic<uint64_t> g_wait_ns{DEFAULT_WAIT_NS};
std::atomic<int> g_skip_cta{-1};
std::atomic<int> g_decode_kernel{0};
std::atomic<int> g_prefill_kernel{0};
std::atomic<int> g_tmajor_kernel{0};
}  // namespace

uint64_t wait_limit_ns() { return g_wait_ns.load(std::memory_order_relaxed); }
int test_skip_cta() { return g_skip_cta.load(std::memory_order_relaxed); }
int test_decode_kernel() { return g_decode_kernel.load(std::memory_order_relaxed); }
int test_prefill_kernel() { return g_prefill_kernel.load(std::memory_order_relaxed); }
int test_tmajor_kernel() { return g_tmajor_kernel.load(std::memory_order_relaxed); }

}  // namespace mq

namespace {

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int abits_of(const mq_linear_desc &d) { return d.abits == 0 ? 8 : d.abits; }
int obits_of(const mq_linear_desc &d) { return d.obits == 0 ? abits_of(d) : d.obits; }

// Validate one linear problem; on success fill the kernel-side Problem (for
// 16-bit activations, x is filled in later with the planes' address).
int check_desc(const mq_linear_desc &d, mq::Problem &out) {
    const int ab = abits_of(d), ob = obits_of(d);
    if (d.bits != 8 && d.bits != 4) return MQ_ERR_INVALID_ARG;
    // activation / output widths: 8 / 8, 16 / 16, or 8 / 16
    if (!((ab == 8 && ob == 8) || (ab == 16 && ob == 16) || (ab == 8 && ob == 16)))
        return MQ_ERR_INVALID_ARG;
    if (d.M < 0 || d.N < 0 || d.K < 0) return MQ_ERR_INVALID_ARG;
    const int32_t zlo = ab == 8 ? -128 : -32768, zhi = ab == 8 ? 127 : 32767;
    const int32_t ylo = ob == 8 ? -128 : -32768, yhi = ob == 8 ? 127 : 32767;
    if (d.zx < zlo || d.zx > zhi || d.zy < ylo || d.zy > yhi) return MQ_ERR_INVALID_ARG;
    if (ab == 16 && d.residual) return MQ_ERR_INVALID_ARG;
    if (ob == 16 && d.residual) return MQ_ERR_INVALID_ARG;
    // transposed weights: int8 [K][N] beside 8-bit activations
    if (d.wt && (d.bits != 8 || ab != 8)) return MQ_ERR_INVALID_ARG;
    // packed bytes of one weight row (of one k-row when transposed)
    const int64_t wrow = d.wt ? (int64_t)d.N : (int64_t)d.K * d.bits / 8;
    if (d.ldw < 0 || (d.ldw > 0 && d.ldw < wrow)) return MQ_ERR_INVALID_ARG;
    if (d.ldw % 16 != 0) return MQ_ERR_ALIGNMENT;
    if (d.K > MQ_MAX_K) return MQ_ERR_K_OVERFLOW;
    // f16 copies of chained layers: only 8-bit activations and outputs
    if ((d.y16 != nullptr) != (d.ysq != nullptr) || (d.x16 != nullptr) != (d.xsq != nullptr))
        return MQ_ERR_INVALID_ARG;
    if ((d.y16 || d.x16) && (ab != 8 || ob != 8)) return MQ_ERR_INVALID_ARG;
    if (d.x16 && !aligned16(d.x16)) return MQ_ERR_ALIGNMENT;
    if (d.y16 && (d.N % 16 != 0 || d.ldy % 16 != 0 || !aligned16(d.y16) || !aligned16(d.y)))
        return MQ_ERR_ALIGNMENT;
    // int32 accumulators of 8-bit activations with int8 weights and a zero point
    // (16-bit activations accumulate in int64; their int8 planes stay below
    // 128 * 255 * 65536 < 2^31)
    if (d.zw && ab == 8 && d.bits == 8 && d.K > MQ_MAX_K_ASYM8) return MQ_ERR_K_OVERFLOW;
    if (d.M > 0 && d.N > 0) {
        // colsum may be omitted with int8 weights: the call derives it (see
        // batch_plan) or its kernel needs none
        if ((!d.colsum && d.bits != 8) || !d.M0 || !d.shift || !d.y || d.ldy < d.N)
            return MQ_ERR_INVALID_ARG;
        if (d.K > 0) {  // with K == 0 neither x nor the weights are read
            if (!d.x || !d.packed || d.ldx < d.K) return MQ_ERR_INVALID_ARG;
            const int kq = d.bits == 8 ? 16 : 32;  // k per 16-byte weight segment
            const int lq = ab == 8 ? 16 : 8;       // x elements per 16 bytes
            if (d.K % kq != 0 || d.ldx % lq != 0) return MQ_ERR_ALIGNMENT;
            if (!aligned16(d.x) || !aligned16(d.packed)) return MQ_ERR_ALIGNMENT;
        }
    }
    out.x = ab == 8 ? static_cast<const int8_t *>(d.x) : nullptr;
    out.w = static_cast<const uint8_t *>(d.packed);
    out.colsum = d.colsum;
    out.M0 = d.M0;
    out.shift = d.shift;
    out.residual = d.residual;
    out.zw = d.zw;
    out.wsq = d.wsq;
    out.y = static_cast<int8_t *>(d.y);
    out.M = ab == 8 ? d.M : 2 * d.M;  // 16 bits: rows of the plane matrix
    out.N = d.N;
    out.K = d.K;
    out.ldx = ab == 8 ? d.ldx : d.K;
    out.ldy = d.ldy;
    out.zx = d.zx;
    out.zy = d.zy;
    out.bits = d.bits;
    out.a16 = ab == 16;
    out.o16 = ab == 8 && ob == 16;
    out.ldw = d.ldw > 0 ? d.ldw : (int32_t)wrow;
    out.wdynamic = d.wdynamic != 0;
    out.tile_begin = 0;
    out.tiles_m = 0;
    return MQ_OK;
}

size_t align16(size_t v) { return (v + 15) & ~static_cast<size_t>(15); }

size_t align128(size_t v) { return (v + 127) & ~static_cast<size_t>(127); }

size_t align1024(size_t v) { return (v + 1023) & ~static_cast<size_t>(1023); }

// A decode shape: at most DECODE_MAX_M rows of the (plane) matrix.
bool is_decode(const mq_linear_desc &d) {
    const int64_t rows = abits_of(d) == 16 ? 2LL * d.M : d.M;
    return rows > 0 && rows <= mq::DECODE_MAX_M;
}

// Smallest M and N that take the 256-token prefill kernel by default: below
// 256 tokens the 128-token kernel's tiles fill the GPU better, and below 256
// output channels its 256-channel tiles would be mostly empty while the
// widening of x (2 M K bytes written per call) weighs more against the
// 2 M N K operations (the attention's P V products, N = 64).
constexpr int WIDE_MIN_M = 256;
constexpr int WIDE_MIN_N = 256;

// A problem served by the 256-token prefill kernel (mq_prefill2.cu) when the
// workspace has room for its widened input: a tensor-core shape with 8-bit
// activations and output.
bool wide_eligible(const mq_linear_desc &d) {
    if (d.M <= 0 || d.N <= 0 || d.K <= 0 || is_decode(d) || d.wt) return false;
    if (abits_of(d) != 8 || obits_of(d) != 8) return false;
    const int which = mq::test_prefill_kernel();
    if (which == 2) return false;
    return which == 1 || (d.M >= WIDE_MIN_M && d.N >= WIDE_MIN_N);
}

// Workspace layout of one batch: the decode region first (if any decode
// shape), then one [2M][K] int8 plane matrix per distinct input (x, M, K,
// ldx) of the 16-bit tensor-core descriptors, in order of first use, with
// offsets relative to the end of the decode region.  These make the required
// size.  Then, optionally, from the first 1024-byte boundary after both the
// required part and the decode region's size (so that it never overlaps the
// decode region of another call sharing the workspace), the f16 copy [M][K]
// and the row sums of squares [M] of every distinct input of the problems the
// 256-token prefill kernel serves: with room for them the batch takes that
// kernel, without it the 128-token one.  That region is scratch.
struct Plan {
    bool any_decode = false;
    std::vector<mq::SplitJob> split;
    std::vector<size_t> split_off;
    std::vector<mq::RowsumJob> csum;  // weight row sums of descriptors without colsum
    std::vector<size_t> csum_off;
    int ksplit = 0;                   // slices of K of the split problems (0: none)
    std::vector<int> ks_idx;          // descriptors split over K
    std::vector<size_t> ks_off;       // their int32 partial sums, from ks_at (1024-aligned)
    size_t ks_at = 0;
    size_t bytes_wide = 0;            // end of the widened inputs (or of the required part)
    std::vector<mq::Widen16Job> wide;
    std::vector<size_t> wide_off;  // f16 copy at wide_off, row sums at + align1024(2 M K)
    size_t required = 0;           // decode region + planes
    size_t bytes = 0;              // required + the widened inputs (if any)
};

template <class J>
int find_job(const std::vector<J> &jobs, const void *x, int M, int K, int ldx) {
    for (size_t i = 0; i < jobs.size(); ++i)
        if (jobs[i].x == x && jobs[i].M == M && jobs[i].K == K && jobs[i].ldx == ldx) return (int)i;
    return -1;
}

// Where the widened inputs may start (before rounding up to 1024 bytes).
size_t wide_at(const Plan &pl) {
    return pl.required > mq::DECODE_WS_BYTES ? pl.required : mq::DECODE_WS_BYTES;
}

// The pre-pass job that writes a problem's output y as f16 into y16 and its
// row sums of squares into ysq.
mq::Widen16Job output_copy_job(const mq_linear_desc &d) {
    mq::Widen16Job j{};
    j.x = static_cast<const int8_t *>(d.y);
    j.out = static_cast<uint16_t *>(d.y16);
    j.rowsq = d.ysq;
    j.M = d.M;
    j.K = d.N;
    j.ldx = d.ldy;
    return j;
}

// Whether a prefill problem takes the token-major kernel (mq_tmajor.cu): short
// K or few channels (8-bit weights and activations; the attention matmuls:
// Q K^T at head dimension K, P V with head dimension N).
bool routes_tmajor(const mq_linear_desc &d, const mq::Problem &p) {
    if (is_decode(d)) return false;
    const int mode = mq::test_tmajor_kernel();
    if (mode == 2 || !mq::tmajor_suits(p)) return false;
    if (d.wt) return true;  // transposed weights: this kernel alone reads them
    // a forced 256-token kernel (test hook) comes before the automatic choice
    if (mode == 0 && mq::test_prefill_kernel() == 1) return false;
    return mode == 1 || p.K <= 128 || p.N <= 64;
}

// A descriptor without colsum whose kernel needs one: the call computes the
// weights' row sums first (the token-major kernel folds both zero points into
// its operands and reads no colsum).
bool needs_row_sums(const mq_linear_desc &d) {
    if (d.colsum || d.M <= 0 || d.N <= 0) return false;
    mq::Problem p{};
    if (check_desc(d, p) != MQ_OK) return false;
    return !routes_tmajor(d, p);
}

// SMs of the current device (cached per device; 0 if the query fails).
int device_sms() {
    static std::atomic<int> cached[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    int n = cached[dev].load(std::memory_order_relaxed);
    if (n == 0 && cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess)
        cached[dev].store(n, std::memory_order_relaxed);
    return n;
}

// A prefill problem that may be split over K: one that the 128-token kernel
// would serve with few tiles (M < 256 or N < 256), 8-bit activations and
// weights, long enough K, and a shape the token-major kernel can take.
bool split_candidate(const mq_linear_desc &d) {
    if (d.M <= 0 || d.N <= 0 || d.K < 512 || is_decode(d) || d.y16 || d.wt) return false;
    if (abits_of(d) != 8 || d.bits != 8 || (d.M >= WIDE_MIN_M && d.N >= WIDE_MIN_N)) return false;
    mq::Problem p{};
    if (check_desc(d, p) != MQ_OK) return false;
    return !routes_tmajor(d, p) && mq::tmajor_suits(p);
}

Plan batch_plan(const mq_linear_desc *descs, int count) {
    Plan pl;
    size_t off = 0;
    for (int i = 0; i < count; ++i) {
        const mq_linear_desc &d = descs[i];
        if (d.M <= 0 || d.N <= 0) continue;
        if (is_decode(d)) pl.any_decode = true;
    }
    for (int i = 0; i < count; ++i) {
        const mq_linear_desc &d = descs[i];
        // the decode kernel reads 16-bit codes itself; only tensor-core shapes
        // take the plane matrix
        if (d.M <= 0 || d.N <= 0 || d.K <= 0 || abits_of(d) != 16 || is_decode(d)) continue;
        if (find_job(pl.split, d.x, d.M, d.K, d.ldx) >= 0) continue;
        off = align128(off);
        mq::SplitJob j{};
        j.x = static_cast<const int16_t *>(d.x);
        j.M = d.M;
        j.K = d.K;
        j.ldx = d.ldx;
        pl.split.push_back(j);
        pl.split_off.push_back(off);
        off += align128(2 * (size_t)d.M * (size_t)d.K);
    }
    for (int i = 0; i < count; ++i) {
        const mq_linear_desc &d = descs[i];
        if (!needs_row_sums(d)) continue;
        const int ldw = d.ldw > 0 ? d.ldw : d.K;
        if (find_job(pl.csum, d.packed, d.N, d.K, ldw) >= 0) continue;
        off = align128(off);
        mq::RowsumJob j{};
        j.x = static_cast<const int8_t *>(d.packed);
        j.M = d.N;
        j.K = d.K;
        j.ldx = ldw;
        pl.csum.push_back(j);
        pl.csum_off.push_back(off);
        off += align128(4 * (size_t)d.N);
    }
    pl.required = (pl.any_decode ? mq::DECODE_WS_BYTES : 0) + off;
    size_t woff = 0;
    for (int i = 0; i < count; ++i) {
        const mq_linear_desc &d = descs[i];
        if (!wide_eligible(d) || d.x16) continue;  // a given f16 copy needs no pre-pass
        const int8_t *x = static_cast<const int8_t *>(d.x);
        bool seen = false;
        for (const auto &j : pl.wide)
            seen = seen || (j.x == x && j.M == d.M && j.K == d.K && j.ldx == d.ldx);
        if (seen) continue;
        mq::Widen16Job j{};
        j.x = x;
        j.M = d.M;
        j.K = d.K;
        j.ldx = d.ldx;
        pl.wide.push_back(j);
        pl.wide_off.push_back(woff);
        woff += align1024(2 * (size_t)d.M * (size_t)d.K) + align1024(4 * (size_t)d.M);
    }
    // + 1024: the region starts at the first 1024-byte boundary after wide_at()
    pl.bytes = pl.wide.empty() ? pl.required : wide_at(pl) + woff + 1024;
    pl.bytes_wide = pl.bytes;
    // Split K: a call made only of prefill problems whose tiles would leave
    // most SMs idle (one M = 128 linear makes 8 pair tiles for 76 pairs) runs
    // them as S slices of K on the token-major kernel, each writing its raw
    // int32 sums, then one combine launch requantizes.  S = SMs / (the
    // token-major tiles of the call), at most 8, each slice at least 256 k;
    // only with the choice of prefill kernel left automatic, and only when the
    // workspace has room (optional, like the widened inputs).
    if (mq::test_prefill_kernel() == 0) {
        long long tiles = 0;
        int kmin = 1 << 30;
        bool all = true;  // only calls made of such problems alone
        for (int i = 0; i < count; ++i) {
            const mq_linear_desc &d = descs[i];
            if (d.M <= 0 || d.N <= 0) continue;
            if (!split_candidate(d)) {
                all = false;
                continue;
            }
            tiles += (long long)((d.M + 127) / 128) * ((d.N + 63) / 64);
            kmin = d.K < kmin ? d.K : kmin;
            pl.ks_idx.push_back(i);
        }
        const int sms = all ? device_sms() : 0;
        long long S = tiles > 0 ? sms / tiles : 0;
        if (S > 8) S = 8;
        if (S > kmin / 256) S = kmin / 256;
        if (S >= 2) {
            pl.ksplit = (int)S;
            pl.ks_at = pl.bytes > wide_at(pl) ? pl.bytes : wide_at(pl);
            size_t o = 0;
            for (int i : pl.ks_idx) {
                pl.ks_off.push_back(o);
                o += align1024((size_t)S * (size_t)descs[i].M * (size_t)descs[i].N * 4);
            }
            pl.bytes = pl.ks_at + o + 1024;
        } else {
            pl.ks_idx.clear();
        }
    }
    return pl;
}

int run_batch(const mq_linear_desc *descs, int count, void *workspace, size_t ws_bytes,
              void *stream) {
    if (!descs || count < 1 || count > MQ_MAX_BATCH) return MQ_ERR_INVALID_ARG;
    std::vector<mq::Problem> probs(count);
    for (int i = 0; i < count; ++i) {
        const int rc = check_desc(descs[i], probs[i]);
        if (rc != MQ_OK) return rc;
        // transposed weights are read by the token-major kernel alone
        const mq_linear_desc &d = descs[i];
        if (d.wt && d.M > 0 && d.N > 0 && d.K > 0 && !routes_tmajor(d, probs[i]))
            return MQ_ERR_UNSUPPORTED_SHAPE;
    }
    // the decode kernel combines split 64-row units in the workspace, 16-bit
    // tensor-core descriptors read their int8 planes from there
    Plan pl = batch_plan(descs, count);
    if (pl.required > 0 && (!workspace || ws_bytes < pl.required || !aligned16(workspace)))
        return MQ_ERR_WORKSPACE;
    uint8_t *region = static_cast<uint8_t *>(workspace) + (pl.any_decode ? mq::DECODE_WS_BYTES : 0);
    for (size_t i = 0; i < pl.split.size(); ++i)
        pl.split[i].out = reinterpret_cast<int8_t *>(region + pl.split_off[i]);
    for (size_t i = 0; i < pl.csum.size(); ++i)
        pl.csum[i].out = reinterpret_cast<int32_t *>(region + pl.csum_off[i]);
    // the 256-token kernel for problems whose f16 copy is given, and for the
    // others when the workspace has room for the widened inputs
    const bool room = !pl.wide.empty() && workspace && ws_bytes >= pl.bytes_wide;
    const bool room_split = pl.ksplit > 0 && workspace && ws_bytes >= pl.bytes;
    std::vector<mq::Problem> ksub;     // the slices of the split problems
    std::vector<uint8_t> ksub_part;
    std::vector<mq::ReduceJob> kred;   // their combines
    bool ready = false, ready_known = false;
    auto takes_wide = [&](const mq_linear_desc &d) {
        if (!wide_eligible(d) || !(d.x16 || room)) return false;
        if (!ready_known) {
            ready = mq::prefill2_ready();
            ready_known = true;
        }
        return ready;
    };
    if (room) {
        const uintptr_t base =
            (reinterpret_cast<uintptr_t>(workspace) + wide_at(pl) + 1023) & ~(uintptr_t)1023;
        for (size_t i = 0; i < pl.wide.size(); ++i) {
            uint8_t *at = reinterpret_cast<uint8_t *>(base + pl.wide_off[i]);
            pl.wide[i].out = reinterpret_cast<uint16_t *>(at);
            pl.wide[i].rowsq = reinterpret_cast<int32_t *>(
                at + align1024(2 * (size_t)pl.wide[i].M * (size_t)pl.wide[i].K));
        }
    }
    std::vector<mq::Problem> tmaj[2];  // by o16
    std::vector<uint8_t> tmaj_wt[2];   // their transposed-weights flags
    std::vector<mq::Problem> pre2;
    std::vector<const uint16_t *> pre2_x16;
    std::vector<const int32_t *> pre2_rowsq;
    std::vector<uint16_t *> pre2_y16;
    std::vector<int32_t *> pre2_ysq;
    std::vector<mq::Widen16Job> after;  // f16 copies of outputs the epilogues do not write
    // kernel families: prefill by activation / output width, decode by weight
    // bits and activation / output width (0: 8 / 8, 1: 16 / 16, 2: 8 / 16)
    std::vector<mq::Problem> pre[3], dec[2][3];
    for (int i = 0; i < count; ++i) {
        mq::Problem &p = probs[i];
        const mq_linear_desc &d = descs[i];
        if (p.M == 0 || p.N == 0) continue;  // nothing to compute or write
        if (p.K > 0 && p.a16) {
            if (is_decode(d)) {  // int16 codes, read by the decode kernel's TMA as they are
                p.x = static_cast<const int8_t *>(d.x);
                p.ldx = d.ldx;
            } else {
                p.x = pl.split[find_job(pl.split, d.x, d.M, d.K, d.ldx)].out;
            }
        }
        if (room_split) {
            int j = -1;
            for (size_t u = 0; u < pl.ks_idx.size(); ++u)
                if (pl.ks_idx[u] == i) j = (int)u;
            if (j >= 0) {  // S slices of K, raw int32 sums into the workspace, then a combine
                const uintptr_t base =
                    (reinterpret_cast<uintptr_t>(workspace) + pl.ks_at + 1023) & ~(uintptr_t)1023;
                int32_t *part = reinterpret_cast<int32_t *>(base + pl.ks_off[j]);
                const size_t slice = (size_t)p.M * (size_t)p.N;
                const int kl = ((p.K + pl.ksplit - 1) / pl.ksplit + 63) / 64 * 64;
                int nslices = 0;
                for (int k0 = 0; k0 < p.K; k0 += kl, ++nslices) {
                    mq::Problem q = p;
                    q.x = p.x + k0;
                    q.w = p.w + k0;
                    q.K = p.K - k0 < kl ? p.K - k0 : kl;
                    q.y = reinterpret_cast<int8_t *>(part + (size_t)nslices * slice);
                    q.ldy = p.N;
                    q.residual = nullptr;
                    q.o16 = 0;
                    q.wsq = nullptr;
                    ksub.push_back(q);
                    ksub_part.push_back(1);
                }
                mq::ReduceJob r{};
                r.part = part;
                r.S = nslices;
                r.M = p.M;
                r.N = p.N;
                r.M0 = p.M0;
                r.shift = p.shift;
                r.zy = p.zy;
                r.residual = p.residual;
                r.y = p.y;
                r.ldy = p.ldy;
                r.o16 = p.o16;
                kred.push_back(r);
                continue;
            }
        }
        if (!p.colsum && needs_row_sums(d)) {  // the row sums computed first
            const int ldw = d.ldw > 0 ? d.ldw : d.K;
            p.colsum = pl.csum[find_job(pl.csum, d.packed, d.N, d.K, ldw)].out;
        }
        const int mode = p.a16 ? 1 : (p.o16 ? 2 : 0);
        if (is_decode(d)) {
            dec[p.bits == 8][mode].push_back(p);
        } else if (routes_tmajor(d, p)) {
            tmaj[p.o16 ? 1 : 0].push_back(p);
            tmaj_wt[p.o16 ? 1 : 0].push_back(d.wt ? 1 : 0);
            if (d.y16) after.push_back(output_copy_job(d));
        } else if (takes_wide(d)) {
            pre2.push_back(p);
            if (d.x16) {
                pre2_x16.push_back(static_cast<const uint16_t *>(d.x16));
                pre2_rowsq.push_back(d.xsq);
            } else {
                const mq::Widen16Job *job = nullptr;
                for (const auto &j : pl.wide)
                    if (j.x == p.x && j.M == d.M && j.K == d.K && j.ldx == d.ldx) job = &j;
                pre2_x16.push_back(job->out);
                pre2_rowsq.push_back(job->rowsq);
            }
            // the epilogue writes the f16 copy of y where its 4-byte stores apply
            const bool fused = d.y16 && (reinterpret_cast<uintptr_t>(d.residual) & 3) == 0;
            pre2_y16.push_back(fused ? static_cast<uint16_t *>(d.y16) : nullptr);
            pre2_ysq.push_back(fused ? d.ysq : nullptr);
            if (d.y16 && !fused) after.push_back(output_copy_job(d));
        } else {
            pre[mode].push_back(p);
            if (d.y16) after.push_back(output_copy_job(d));
        }
    }
    int rc = MQ_OK;
    if (!pl.csum.empty()) rc = mq::launch_rowsum(pl.csum.data(), (int)pl.csum.size(), stream);
    if (rc == MQ_OK && !pl.split.empty())
        rc = mq::launch_split16(pl.split.data(), (int)pl.split.size(), stream);
    if (rc == MQ_OK && !pre2.empty()) {
        if (room) rc = mq::launch_widen16(pl.wide.data(), (int)pl.wide.size(), stream);
        if (rc == MQ_OK)
            rc = mq::launch_prefill2(pre2.data(), pre2_x16.data(), pre2_rowsq.data(),
                                     pre2_y16.data(), pre2_ysq.data(), (int)pre2.size(), stream);
    }
    for (int o = 0; o < 2; ++o)
        if (rc == MQ_OK && !tmaj[o].empty())
            rc = mq::launch_tmajor(tmaj[o].data(), (int)tmaj[o].size(), stream, nullptr,
                                   tmaj_wt[o].data());
    if (rc == MQ_OK && !ksub.empty()) {
        rc = mq::launch_tmajor(ksub.data(), (int)ksub.size(), stream, ksub_part.data());
        if (rc == MQ_OK) rc = mq::launch_splitk_reduce(kred.data(), (int)kred.size(), stream);
    }
    for (int mode = 0; mode < 3; ++mode)
        if (rc == MQ_OK && !pre[mode].empty())
            rc = mq::launch_prefill(pre[mode].data(), (int)pre[mode].size(), stream);
    for (int b = 1; b >= 0; --b)
        for (int a = 0; a < 3; ++a)
            if (rc == MQ_OK && !dec[b][a].empty())
                rc = mq::launch_decode(dec[b][a].data(), (int)dec[b][a].size(), workspace, stream);
    // f16 copies of outputs no epilogue wrote: the pre-pass on y, after everything
    // that writes y (its row sums overwrite the caller's zeros)
    if (rc == MQ_OK && !after.empty())
        rc = mq::launch_widen16(after.data(), (int)after.size(), stream);
    return rc;
}

int single(int bits, const int8_t *x, int M, int K, int ldx, int32_t zx, const void *packed,
           const int32_t *colsum, int N, const int32_t *M0, const int32_t *shift, int32_t zy,
           int8_t *y, int ldy, void *workspace, size_t ws_bytes, void *stream) {
    if (!colsum && M > 0 && N > 0) return MQ_ERR_INVALID_ARG;  // required by the single calls
    mq_linear_desc d{};
    d.x = x;
    d.packed = packed;
    d.colsum = colsum;
    d.M0 = M0;
    d.shift = shift;
    d.residual = nullptr;
    d.zw = nullptr;
    d.y = y;
    d.M = M;
    d.N = N;
    d.K = K;
    d.ldx = ldx;
    d.ldy = ldy;
    d.zx = zx;
    d.zy = zy;
    d.bits = bits;
    d.abits = 8;
    return run_batch(&d, 1, workspace, ws_bytes, stream);
}

int single_a16(int bits, const int16_t *x, int M, int K, int ldx, int32_t zx, const void *packed,
               const int32_t *colsum, int N, const int32_t *M0, const int32_t *shift, int32_t zy,
               int16_t *y, int ldy, void *workspace, size_t ws_bytes, void *stream) {
    if (!colsum && M > 0 && N > 0) return MQ_ERR_INVALID_ARG;  // required by the single calls
    mq_linear_desc d{};
    d.x = x;
    d.packed = packed;
    d.colsum = colsum;
    d.M0 = M0;
    d.shift = shift;
    d.y = y;
    d.M = M;
    d.N = N;
    d.K = K;
    d.ldx = ldx;
    d.ldy = ldy;
    d.zx = zx;
    d.zy = zy;
    d.bits = bits;
    d.abits = 16;
    return run_batch(&d, 1, workspace, ws_bytes, stream);
}

// Fixed-point form of one positive normal double m: m0 * 2^-s.
int fixed_point(double m, int32_t &m0_out, int32_t &s_out) {
    uint64_t bits;
    std::memcpy(&bits, &m, sizeof bits);
    const int biased = (int)((bits >> 52) & 0x7FF);
    if (biased == 0) {  // subnormal: far below 2^-32, product with any int32 rounds to 0
        m0_out = 0;
        s_out = 1;
        return MQ_OK;
    }
    // m = sig * 2^(biased - 1075), sig in [2^52, 2^53); as f * 2^e with
    // f = sig / 2^53 in [0.5, 1): e = biased - 1022.
    const uint64_t sig = (bits & ((1ull << 52) - 1)) | (1ull << 52);
    int e = biased - 1022;
    uint64_t m0 = (sig + (1ull << 21)) >> 22;  // round(f * 2^31), ties away from zero
    if (m0 == (1ull << 31)) {
        m0 = 1ull << 30;
        e += 1;
    }
    const int s = 31 - e;
    if (s > 62) {
        m0_out = 0;
        s_out = 1;
        return MQ_OK;
    }
    if (s < 1) return MQ_ERR_INVALID_ARG;
    m0_out = (int32_t)m0;
    s_out = s;
    return MQ_OK;
}

bool good_scale(float v) { return std::isfinite(v) && v > 0.0f; }

}  // namespace

extern "C" {

const char *mq_status_string(int status) {
    switch (status) {
        case MQ_OK: return "MQ_OK";
        case MQ_ERR_INVALID_ARG: return "MQ_ERR_INVALID_ARG";
        case MQ_ERR_UNSUPPORTED_SHAPE: return "MQ_ERR_UNSUPPORTED_SHAPE";
        case MQ_ERR_K_OVERFLOW: return "MQ_ERR_K_OVERFLOW";
        case MQ_ERR_ALIGNMENT: return "MQ_ERR_ALIGNMENT";
        case MQ_ERR_CUDA: return "MQ_ERR_CUDA";
        case MQ_ERR_DEVICE_TIMEOUT: return "MQ_ERR_DEVICE_TIMEOUT";
        case MQ_ERR_WORKSPACE: return "MQ_ERR_WORKSPACE";
        default: return "MQ_ERR_UNKNOWN";
    }
}

int mq_requant_params(const float *sw, int N, float sx, float sy, int32_t *M0, int32_t *shift) {
    if (N < 0 || (N > 0 && (!sw || !M0 || !shift))) return MQ_ERR_INVALID_ARG;
    if (!good_scale(sx) || !good_scale(sy)) return MQ_ERR_INVALID_ARG;
    for (int n = 0; n < N; ++n) {
        if (!good_scale(sw[n])) return MQ_ERR_INVALID_ARG;
        const double m = ((double)sx * (double)sw[n]) / (double)sy;
        const int rc = fixed_point(m, M0[n], shift[n]);
        if (rc != MQ_OK) return rc;
    }
    return MQ_OK;
}

int mq_packed_size(int N, int K, int bits, size_t *bytes) {
    if (!bytes || N < 0 || K < 0 || (bits != 8 && bits != 4)) return MQ_ERR_INVALID_ARG;
    if (bits == 4 && (K & 1)) return MQ_ERR_INVALID_ARG;
    *bytes = bits == 8 ? (size_t)N * (size_t)K : (size_t)N * (size_t)(K / 2);
    return MQ_OK;
}

int mq_pack_weights(const int8_t *w, int N, int K, int bits, void *packed, int32_t *colsum,
                    int on_device, void *stream) {
    if (N < 0 || K < 0 || (bits != 8 && bits != 4)) return MQ_ERR_INVALID_ARG;
    if (bits == 4 && (K & 1)) return MQ_ERR_INVALID_ARG;
    if (N == 0) return MQ_OK;
    if (!colsum || (K > 0 && (!w || !packed))) return MQ_ERR_INVALID_ARG;
    if (!on_device) {
        uint8_t *dst = static_cast<uint8_t *>(packed);
        for (int n = 0; n < N; ++n) {
            const int8_t *row = w + (size_t)n * (size_t)K;
            int64_t sum = 0;
            if (bits == 8) {
                for (int k = 0; k < K; ++k) sum += row[k];
                if (K) std::memcpy(dst + (size_t)n * (size_t)K, row, (size_t)K);
            } else {
                uint8_t *out = dst + (size_t)n * (size_t)(K / 2);
                for (int j = 0; j < K / 2; ++j) {
                    const int lo = row[2 * j], hi = row[2 * j + 1];
                    if (lo < -8 || lo > 7 || hi < -8 || hi > 7) return MQ_ERR_INVALID_ARG;
                    out[j] = (uint8_t)((unsigned)(lo & 0x0F) | ((unsigned)(hi & 0x0F) << 4));
                    sum += lo + hi;
                }
            }
            colsum[n] = (int32_t)sum;
        }
        return MQ_OK;
    }
    // Device path: the kernel flags out-of-range int4 values in the pack
    // status word; packing is an offline step, so the call waits for it.
    int *status = mq::pack_status_ptr();
    if (!status) return MQ_ERR_CUDA;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(status, 0, sizeof(int), s) != cudaSuccess) return MQ_ERR_CUDA;
    int rc = mq::launch_pack(w, N, K, bits, packed, colsum, status, stream);
    if (rc != MQ_OK) return rc;
    int flags = 0;
    if (cudaMemcpyAsync(&flags, status, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return MQ_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return MQ_ERR_CUDA;
    return flags ? MQ_ERR_INVALID_ARG : MQ_OK;
}

int mq_workspace_size(int M, int N, int K, int bits, size_t *bytes) {
    if (!bytes || M < 0 || N < 0 || K < 0 || (bits != 8 && bits != 4)) return MQ_ERR_INVALID_ARG;
    mq_linear_desc d{};
    d.x = reinterpret_cast<const void *>(16);  // placeholder addresses: only sizes are planned
    d.colsum = reinterpret_cast<const int32_t *>(16);
    d.M = M;
    d.N = N;
    d.K = K;
    d.ldx = K;
    d.bits = bits;
    *bytes = batch_plan(&d, 1).bytes;
    return MQ_OK;
}

int mq_linear_w8a8(const int8_t *x, int M, int K, int ldx, int32_t zx, const void *packed,
                   const int32_t *colsum, int N, const int32_t *M0, const int32_t *shift,
                   int32_t zy, int8_t *y, int ldy, void *workspace, size_t ws_bytes,
                   void *stream) {
    return single(8, x, M, K, ldx, zx, packed, colsum, N, M0, shift, zy, y, ldy, workspace,
                  ws_bytes, stream);
}

int mq_linear_w4a8(const int8_t *x, int M, int K, int ldx, int32_t zx, const void *packed,
                   const int32_t *colsum, int N, const int32_t *M0, const int32_t *shift,
                   int32_t zy, int8_t *y, int ldy, void *workspace, size_t ws_bytes,
                   void *stream) {
    return single(4, x, M, K, ldx, zx, packed, colsum, N, M0, shift, zy, y, ldy, workspace,
                  ws_bytes, stream);
}

int mq_workspace_size_batch(const mq_linear_desc *descs, int count, size_t *bytes) {
    if (!descs || !bytes || count < 1 || count > MQ_MAX_BATCH) return MQ_ERR_INVALID_ARG;
    for (int i = 0; i < count; ++i) {
        if (descs[i].bits != 8 && descs[i].bits != 4) return MQ_ERR_INVALID_ARG;
        if (abits_of(descs[i]) != 8 && abits_of(descs[i]) != 16) return MQ_ERR_INVALID_ARG;
        if (obits_of(descs[i]) != 8 && obits_of(descs[i]) != 16) return MQ_ERR_INVALID_ARG;
    }
    *bytes = batch_plan(descs, count).bytes;
    return MQ_OK;
}

int mq_workspace_size_a16(int M, int N, int K, int bits, size_t *bytes) {
    if (!bytes || M < 0 || N < 0 || K < 0 || (bits != 8 && bits != 4)) return MQ_ERR_INVALID_ARG;
    mq_linear_desc d{};
    d.x = reinterpret_cast<const void *>(16);  // placeholder addresses: only sizes are planned
    d.colsum = reinterpret_cast<const int32_t *>(16);
    d.M = M;
    d.N = N;
    d.K = K;
    d.ldx = K;
    d.bits = bits;
    d.abits = 16;
    *bytes = batch_plan(&d, 1).bytes;
    return MQ_OK;
}

int mq_linear_w8a16(const int16_t *x, int M, int K, int ldx, int32_t zx, const void *packed,
                    const int32_t *colsum, int N, const int32_t *M0, const int32_t *shift,
                    int32_t zy, int16_t *y, int ldy, void *workspace, size_t ws_bytes,
                    void *stream) {
    return single_a16(8, x, M, K, ldx, zx, packed, colsum, N, M0, shift, zy, y, ldy, workspace,
                      ws_bytes, stream);
}

int mq_linear_w4a16(const int16_t *x, int M, int K, int ldx, int32_t zx, const void *packed,
                    const int32_t *colsum, int N, const int32_t *M0, const int32_t *shift,
                    int32_t zy, int16_t *y, int ldy, void *workspace, size_t ws_bytes,
                    void *stream) {
    return single_a16(4, x, M, K, ldx, zx, packed, colsum, N, M0, shift, zy, y, ldy, workspace,
                      ws_bytes, stream);
}

int mq_linear_batch(const mq_linear_desc *descs, int count, void *workspace, size_t ws_bytes,
                    void *stream) {
    return run_batch(descs, count, workspace, ws_bytes, stream);
}

namespace {

bool code_range(int type, int32_t *lo, int32_t *hi) {
    if (type == MQ_TYPE_I8) {
        *lo = -128;
        *hi = 127;
        return true;
    }
    if (type == MQ_TYPE_I16) {
        *lo = -32768;
        *hi = 32767;
        return true;
    }
    return false;
}

bool float_type(int type) {
    return type == MQ_TYPE_F32 || type == MQ_TYPE_F16 || type == MQ_TYPE_BF16;
}

size_t type_size(int type) { return type == MQ_TYPE_F32 ? 4 : (type == MQ_TYPE_I8 ? 1 : 2); }

bool aligned_to(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

int mq_quantize(const void *x, int in_type, int64_t n, float alpha, int32_t z, void *q,
                int out_type, void *stream) {
    int32_t lo, hi;
    if (!float_type(in_type) || !code_range(out_type, &lo, &hi) || n < 0) return MQ_ERR_INVALID_ARG;
    if (!(std::isfinite(alpha) && alpha > 0.0f) || z < lo || z > hi) return MQ_ERR_INVALID_ARG;
    if (n == 0) return MQ_OK;
    if (!x || !q) return MQ_ERR_INVALID_ARG;
    if (!aligned_to(x, type_size(in_type)) || !aligned_to(q, type_size(out_type)))
        return MQ_ERR_ALIGNMENT;
    return mq::launch_glue(0, in_type, out_type, x, q, n, alpha, 0, z, 0, 1, lo, hi, stream);
}

int mq_dequantize(const void *q, int in_type, int64_t n, float alpha, int32_t z, float *f,
                  void *stream) {
    int32_t lo, hi;
    if (!code_range(in_type, &lo, &hi) || n < 0) return MQ_ERR_INVALID_ARG;
    if (!std::isfinite(alpha) || z < lo || z > hi) return MQ_ERR_INVALID_ARG;
    if (n == 0) return MQ_OK;
    if (!q || !f) return MQ_ERR_INVALID_ARG;
    if (!aligned_to(q, type_size(in_type)) || !aligned_to(f, 4)) return MQ_ERR_ALIGNMENT;
    return mq::launch_glue(1, in_type, MQ_TYPE_F32, q, f, n, alpha, z, 0, 0, 1, 0, 0, stream);
}

int mq_requantize(const void *q, int in_type, int64_t n, int32_t zx, int32_t M0, int32_t shift,
                  int32_t zy, void *y, int out_type, void *stream) {
    int32_t ilo, ihi, lo, hi;
    if (!code_range(in_type, &ilo, &ihi) || !code_range(out_type, &lo, &hi) || n < 0)
        return MQ_ERR_INVALID_ARG;
    if (zx < ilo || zx > ihi || zy < lo || zy > hi || M0 < 0 || shift < 1 || shift > 62)
        return MQ_ERR_INVALID_ARG;
    if (n == 0) return MQ_OK;
    if (!q || !y) return MQ_ERR_INVALID_ARG;
    if (!aligned_to(q, type_size(in_type)) || !aligned_to(y, type_size(out_type)))
        return MQ_ERR_ALIGNMENT;
    return mq::launch_glue(2, in_type, out_type, q, y, n, 0.0f, zx, zy, M0, shift, lo, hi, stream);
}

namespace {

int check_fold(const mq_fold_desc &d) {
    if (d.N < 0 || d.K < 0 || (d.bits != 8 && d.bits != 4) ||
        d.scheme < MQ_WEIGHTS_SYM_CHANNEL || d.scheme > MQ_WEIGHTS_ASYM_TENSOR)
        return MQ_ERR_INVALID_ARG;
    if (d.bits == 4 && (d.K & 1)) return MQ_ERR_INVALID_ARG;
    if (d.N == 0) return MQ_OK;
    if (!d.colsum || !d.sw || !d.stats || (d.scheme != MQ_WEIGHTS_SYM_CHANNEL && !d.zw))
        return MQ_ERR_INVALID_ARG;
    if (d.K > 0 && (!d.w || !d.packed)) return MQ_ERR_INVALID_ARG;
    if (!aligned_to(d.w, 4) || !aligned_to(d.s_in, 4) || !aligned_to(d.s_out, 4) ||
        !aligned_to(d.colsum, 4) || !aligned_to(d.sw, 4) || !aligned_to(d.zw, 4) ||
        !aligned_to(d.stats, 4))
        return MQ_ERR_ALIGNMENT;
    return MQ_OK;
}

}  // namespace

int mq_fold_quantize_pack_batch(const mq_fold_desc *descs, int count, void *stream) {
    if (count < 0 || count > MQ_FOLD_MAX_JOBS || (count > 0 && !descs)) return MQ_ERR_INVALID_ARG;
    mq::FoldJob jobs[MQ_FOLD_MAX_JOBS];
    int n = 0;
    for (int i = 0; i < count; ++i) {
        const mq_fold_desc &d = descs[i];
        if (const int rc = check_fold(d)) return rc;
        if (d.N == 0) continue;
        jobs[n++] = mq::FoldJob{d.w,  d.N,      d.K,      d.s_in,   d.s_out, d.bits,
                                d.scheme, d.packed, d.colsum, d.sw, d.zw,    d.stats};
    }
    return n ? mq::launch_fold(jobs, n, stream) : MQ_OK;
}

int mq_fold_quantize_pack(const float *w, int N, int K, const float *s_in, const float *s_out,
                          int bits, int scheme, void *packed, int32_t *colsum, float *sw,
                          int32_t *zw, float *stats, void *stream) {
    const mq_fold_desc d{w, N, K, s_in, s_out, bits, scheme, packed, colsum, sw, zw, stats};
    return mq_fold_quantize_pack_batch(&d, 1, stream);
}

int mq_fold_norm(const float *gamma, const float *beta, const float *s, int K, float *gamma_out,
                 float *beta_out) {
    if (K < 0) return MQ_ERR_INVALID_ARG;
    if (K > 0 && (!gamma || !s || !gamma_out || (beta && !beta_out))) return MQ_ERR_INVALID_ARG;
    for (int k = 0; k < K; ++k) {
        if (!(std::isfinite(s[k]) && s[k] > 0.0f)) return MQ_ERR_INVALID_ARG;
        gamma_out[k] = gamma[k] / s[k];
        if (beta) beta_out[k] = beta[k] / s[k];
    }
    return MQ_OK;
}

int mq_row_sums(const int8_t *x, int M, int K, int ldx, int32_t *out, void *stream) {
    if (M < 0 || K < 0 || K > MQ_MAX_K || ldx < K) return MQ_ERR_INVALID_ARG;
    if (M == 0) return MQ_OK;
    if (!out || (K > 0 && !x)) return MQ_ERR_INVALID_ARG;
    if (K % 16 != 0 || ldx % 16 != 0 || (K > 0 && !aligned16(x))) return MQ_ERR_ALIGNMENT;
    mq::RowsumJob j{};
    j.x = x;
    j.out = out;
    j.M = M;
    j.K = K;
    j.ldx = ldx;
    return mq::launch_rowsum(&j, 1, stream);
}

int mq_weight_sq_sums(const void *packed, int N, int K, int bits, int ldw, int32_t *wsq,
                      void *stream) {
    if (N < 0 || K < 0 || K > MQ_MAX_K || (bits != 8 && bits != 4)) return MQ_ERR_INVALID_ARG;
    const int row = K * bits / 8;
    if (ldw < 0 || (ldw > 0 && ldw < row)) return MQ_ERR_INVALID_ARG;
    if (N == 0) return MQ_OK;
    if (!wsq || (K > 0 && !packed)) return MQ_ERR_INVALID_ARG;
    if (K % (bits == 8 ? 16 : 32) != 0 || ldw % 16 != 0 || (K > 0 && !aligned16(packed)))
        return MQ_ERR_ALIGNMENT;
    return mq::launch_weight_sq(static_cast<const uint8_t *>(packed), N, K, bits,
                                ldw > 0 ? ldw : row, wsq, stream);
}

int mq_head_row_sums(const int8_t *x, int M, int heads, int d, int ldx, int32_t *out,
                     void *stream) {
    if (M < 0 || heads < 0 || d < 0 || d > MQ_MAX_K || (int64_t)heads * d > ldx)
        return MQ_ERR_INVALID_ARG;
    if (M == 0 || heads == 0) return MQ_OK;
    if (!out || (d > 0 && !x)) return MQ_ERR_INVALID_ARG;
    if (d % 16 != 0 || ldx % 16 != 0 || (d > 0 && !aligned16(x))) return MQ_ERR_ALIGNMENT;
    for (int h0 = 0; h0 < heads; h0 += mq::ROWSUM_MAX_JOBS) {
        const int n = heads - h0 < mq::ROWSUM_MAX_JOBS ? heads - h0 : mq::ROWSUM_MAX_JOBS;
        mq::RowsumJob jobs[mq::ROWSUM_MAX_JOBS];
        for (int i = 0; i < n; ++i) {
            jobs[i] = mq::RowsumJob{};
            jobs[i].x = x + (size_t)(h0 + i) * (size_t)d;
            jobs[i].out = out + (size_t)(h0 + i) * (size_t)M;
            jobs[i].M = M;
            jobs[i].K = d;
            jobs[i].ldx = ldx;
        }
        const int rc = mq::launch_rowsum(jobs, n, stream);
        if (rc != MQ_OK) return rc;
    }
    return MQ_OK;
}

int mq_transpose_i8(const int8_t *src, int rows, int cols, int lds, int8_t *dst, int ldd,
                    void *stream) {
    if (rows < 0 || cols < 0 || lds < cols || ldd < rows) return MQ_ERR_INVALID_ARG;
    if (rows == 0 || cols == 0) return MQ_OK;
    if (!src || !dst) return MQ_ERR_INVALID_ARG;
    return mq::launch_transpose_i8(src, rows, cols, lds, dst, ldd, stream);
}

int mq_set_wait_limit_ns(uint64_t ns) {
    if (ns == 0) ns = mq::DEFAULT_WAIT_NS;
    if (ns < 1000) ns = 1000;
    if (ns > 60000000000ull) return MQ_ERR_INVALID_ARG;
    mq::g_wait_ns.store(ns, std::memory_order_relaxed);
    return MQ_OK;
}

int mq_test_skip_partials(int cta) {
    if (cta < -1 || cta >= mq::DECODE_MAX_GRID) return MQ_ERR_INVALID_ARG;
    mq::g_skip_cta.store(cta, std::memory_order_relaxed);
    return MQ_OK;
}

int mq_test_decode_kernel(int which) {
    if (which < 0 || which > 2) return MQ_ERR_INVALID_ARG;
    mq::g_decode_kernel.store(which, std::memory_order_relaxed);
    return MQ_OK;
}

int mq_test_prefill_kernel(int which) {
    if (which < 0 || which > 2) return MQ_ERR_INVALID_ARG;
    mq::g_prefill_kernel.store(which, std::memory_order_relaxed);
    return MQ_OK;
}

int mq_test_tmajor_kernel(int which) {
    if (which < 0 || which > 2) return MQ_ERR_INVALID_ARG;
    mq::g_tmajor_kernel.store(which, std::memory_order_relaxed);
    return MQ_OK;
}

int mq_check_device_status(void *stream) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess) return MQ_ERR_CUDA;
    int *status = mq::device_status_ptr();
    if (!status) return MQ_ERR_CUDA;
    int flags = 0;
    if (cudaMemcpy(&flags, status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
        return MQ_ERR_CUDA;
    if (flags & MQ_DEVICE_STATUS_TIMEOUT) {
        if (cudaMemset(status, 0, sizeof(int)) != cudaSuccess) return MQ_ERR_CUDA;
        return MQ_ERR_DEVICE_TIMEOUT;
    }
    return MQ_OK;
}

}  // extern "C"
