// mq_host.cpp -- host half of the libmq C ABI: argument validation,
// fixed-point requantization parameters, host-side packing, dispatch of
// linear problems to the prefill (tensor-core) and decode (weight-streaming)
// kernels, and device status reporting.
#include <cuda_runtime.h>

#include <cmath>
#include <cstring>
#include <vector>

#include "mq_internal.h"

namespace {

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Validate one linear problem; on success fill the kernel-side Problem.
int check_desc(const mq_linear_desc &d, mq::Problem &out) {
    if (d.bits != 8 && d.bits != 4) return MQ_ERR_INVALID_ARG;
    if (d.M < 0 || d.N < 0 || d.K < 0) return MQ_ERR_INVALID_ARG;
    if (d.zx < -128 || d.zx > 127 || d.zy < -128 || d.zy > 127) return MQ_ERR_INVALID_ARG;
    if (d.K > MQ_MAX_K) return MQ_ERR_K_OVERFLOW;
    if (d.zw && d.bits == 8 && d.K > MQ_MAX_K_ASYM8) return MQ_ERR_K_OVERFLOW;
    if (d.M > 0 && d.N > 0) {
        if (!d.colsum || !d.M0 || !d.shift || !d.y || d.ldy < d.N) return MQ_ERR_INVALID_ARG;
        if (d.K > 0) {  // with K == 0 neither x nor the weights are read
            if (!d.x || !d.packed || d.ldx < d.K) return MQ_ERR_INVALID_ARG;
            const int kq = d.bits == 8 ? 16 : 32;  // k per 16-byte weight segment
            if (d.K % kq != 0 || d.ldx % 16 != 0) return MQ_ERR_ALIGNMENT;
            if (!aligned16(d.x) || !aligned16(d.packed)) return MQ_ERR_ALIGNMENT;
        }
    }
    out.x = d.x;
    out.w = static_cast<const uint8_t *>(d.packed);
    out.colsum = d.colsum;
    out.M0 = d.M0;
    out.shift = d.shift;
    out.residual = d.residual;
    out.zw = d.zw;
    out.rowsum = nullptr;
    out.y = d.y;
    out.M = d.M;
    out.N = d.N;
    out.K = d.K;
    out.ldx = d.ldx;
    out.ldy = d.ldy;
    out.zx = d.zx;
    out.zy = d.zy;
    out.bits = d.bits;
    out.tile_begin = 0;
    out.tiles_m = 0;
    return MQ_OK;
}

size_t align16(size_t v) { return (v + 15) & ~static_cast<size_t>(15); }

// Workspace layout of one batch: the decode region first (if any decode
// shape), then one rowsum(x) array per distinct input (x, M, K, ldx) of the
// prefill descriptors with a weight zero point, in order of first use.
// `jobs` (may be null) receives those inputs and `offsets` their byte
// offsets from the start of the rowsum region.
size_t batch_workspace(const mq_linear_desc *descs, int count, bool *any_decode,
                       std::vector<mq::RowsumJob> *jobs, std::vector<size_t> *offsets) {
    bool dec = false;
    std::vector<mq::RowsumJob> uniq;
    std::vector<size_t> offs;
    size_t rows = 0;
    for (int i = 0; i < count; ++i) {
        const mq_linear_desc &d = descs[i];
        if (d.M <= 0 || d.N <= 0) continue;
        if (d.M <= mq::DECODE_MAX_M) {
            dec = true;
            continue;
        }
        if (!d.zw || d.K <= 0) continue;
        bool seen = false;
        for (const auto &j : uniq)
            seen |= j.x == d.x && j.M == d.M && j.K == d.K && j.ldx == d.ldx;
        if (seen) continue;
        mq::RowsumJob j{};
        j.x = d.x;
        j.M = d.M;
        j.K = d.K;
        j.ldx = d.ldx;
        uniq.push_back(j);
        offs.push_back(rows);
        rows += align16(4 * (size_t)d.M);
    }
    if (any_decode) *any_decode = dec;
    if (jobs) *jobs = uniq;
    if (offsets) *offsets = offs;
    return (dec ? mq::DECODE_WS_BYTES : 0) + rows;
}

int run_batch(const mq_linear_desc *descs, int count, void *workspace, size_t ws_bytes,
              void *stream) {
    if (!descs || count < 1 || count > MQ_MAX_BATCH) return MQ_ERR_INVALID_ARG;
    std::vector<mq::Problem> pre, dec8, dec4;
    pre.reserve(count);
    for (int i = 0; i < count; ++i) {
        mq::Problem p{};
        const int rc = check_desc(descs[i], p);
        if (rc != MQ_OK) return rc;
        if (p.M == 0 || p.N == 0) continue;  // nothing to compute or write
        if (p.M <= mq::DECODE_MAX_M)
            (p.bits == 8 ? dec8 : dec4).push_back(p);
        else
            pre.push_back(p);
    }
    // the decode kernel combines split 64-row units in the workspace; prefill
    // descriptors with a weight zero point read rowsum(x) from there
    bool any_decode = false;
    std::vector<mq::RowsumJob> jobs;
    std::vector<size_t> offsets;
    const size_t need = batch_workspace(descs, count, &any_decode, &jobs, &offsets);
    if (need > 0 && (!workspace || ws_bytes < need || !aligned16(workspace)))
        return MQ_ERR_WORKSPACE;
    uint8_t *region = static_cast<uint8_t *>(workspace) + (any_decode ? mq::DECODE_WS_BYTES : 0);
    for (size_t i = 0; i < jobs.size(); ++i)
        jobs[i].out = reinterpret_cast<int32_t *>(region + offsets[i]);
    for (auto &p : pre) {
        if (!p.zw || p.K == 0) continue;
        for (const auto &j : jobs)
            if (j.x == p.x && j.M == p.M && j.K == p.K && j.ldx == p.ldx) p.rowsum = j.out;
    }
    int rc = MQ_OK;
    if (!jobs.empty()) rc = mq::launch_rowsum(jobs.data(), (int)jobs.size(), stream);
    if (rc == MQ_OK && !pre.empty()) rc = mq::launch_prefill(pre.data(), (int)pre.size(), stream);
    if (rc == MQ_OK && !dec8.empty())
        rc = mq::launch_decode(dec8.data(), (int)dec8.size(), workspace, stream);
    if (rc == MQ_OK && !dec4.empty())
        rc = mq::launch_decode(dec4.data(), (int)dec4.size(), workspace, stream);
    return rc;
}

int single(int bits, const int8_t *x, int M, int K, int ldx, int32_t zx, const void *packed,
           const int32_t *colsum, int N, const int32_t *M0, const int32_t *shift, int32_t zy,
           int8_t *y, int ldy, void *workspace, size_t ws_bytes, void *stream) {
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
    *bytes = (M > 0 && M <= mq::DECODE_MAX_M && N > 0) ? mq::DECODE_WS_BYTES : 0;
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
    for (int i = 0; i < count; ++i)
        if (descs[i].bits != 8 && descs[i].bits != 4) return MQ_ERR_INVALID_ARG;
    *bytes = batch_workspace(descs, count, nullptr, nullptr, nullptr);
    return MQ_OK;
}

int mq_linear_batch(const mq_linear_desc *descs, int count, void *workspace, size_t ws_bytes,
                    void *stream) {
    return run_batch(descs, count, workspace, ws_bytes, stream);
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
