// mq_internal.h -- definitions shared by libmq's host code and its kernels.
#pragma once

#include <cstddef>
#include <cstdint>

#include "../../include/mq.h"

// Bits of the device status word (a __device__ int owned by libmq).
#define MQ_DEVICE_STATUS_TIMEOUT 1
#define MQ_DEVICE_STATUS_PACK_RANGE 2

namespace mq {

// One linear problem as the kernels see it (validated by the host).
struct Problem {
    const int8_t *x;
    const uint8_t *w;
    const int32_t *colsum;
    const int32_t *M0;
    const int32_t *shift;
    const int8_t *residual;
    const int32_t *zw;      // per-channel weight zero point, or null
    const int32_t *wsq;     // per-channel sum of squared weight codes, or null
    int8_t *y;
    int32_t M, N, K, ldx, ldy;
    int32_t zx, zy;
    int32_t bits;
    // 16-bit activations: M is the row count 2M' of the plane matrix of the M'
    // int16 tokens (rows 2m = high bytes, 2m + 1 = low bytes - 128), y points
    // to int16 [M'][ldy], and the epilogues form 256 S(2m) + S(2m + 1) +
    // (128 - zx) colsum.  For the prefill kernel x is that plane matrix
    // (ldx = K); the decode kernel reads the int16 codes [M'][ldx] and forms
    // the planes itself.
    int32_t a16;
    int32_t o16;         // 8-bit inputs, int16 output y [M][ldy] (requantized to 16 bits)
    int32_t ldw;         // bytes between weight rows
    int32_t wdynamic;    // weights written by earlier work in the stream: read after the wait
    int32_t tile_begin;  // first global tile / block index of this problem
    int32_t tiles_m;     // prefill: number of 128-row tiles
};

// Largest M served by the weight-streaming decode kernel.
constexpr int DECODE_MAX_M = 16;

// Decode workspace: per CTA of the decode grid (at most DECODE_MAX_GRID) one
// slot of 64 x 16 entries {int32 partial sum, uint32 launch epoch}, written
// by a CTA that contributes to a 64-row unit finished by another CTA.
constexpr int DECODE_MAX_GRID = 320;
constexpr size_t DECODE_WS_BYTES = 8 * (size_t)DECODE_MAX_GRID * 64 * 16;

// Problems per kernel launch (kernel parameter space).
constexpr int PREFILL_MAX_PROBLEMS = 32;
constexpr int DECODE_MAX_PROBLEMS = 64;

// Device status words (__device__ ints owned by libmq, addresses cached per
// device): kernels atomicOr MQ_DEVICE_STATUS_* bits into them.  The pack
// kernel reports out-of-range int4 values in a word of its own.
int *device_status_ptr();
int *pack_status_ptr();

// Limit of every bounded device-side wait, in nanoseconds, for the launches
// made from now on (mq_set_wait_limit_ns; 1 second by default).
uint64_t wait_limit_ns();
// Failure-detection test hook (mq_test_skip_partials): the decode CTA whose
// split-unit sums are not stored, or -1.
int test_skip_cta();

// Launchers (asynchronous on `stream`); return MQ_OK or MQ_ERR_CUDA.  The
// problems of one launch_prefill call have the same a16 and o16; those of one
// launch_decode call the same bits, a16 and o16.
int launch_prefill(const Problem *probs, int count, void *stream);
int launch_decode(const Problem *probs, int count, void *workspace, void *stream);
// Set-up of both token-tile variants of the W4A8 decode kernel on the current
// device (done by the first launch of each variant otherwise).
int prepare_decode_w4a8();
// The weight-streaming kernel for one or two tokens (mq_gemv.cu): whether a
// decode launch suits it (forced: only the structural conditions), and its
// launcher.
bool gemv_suits(const Problem *probs, int count, int sms, bool force);
int launch_gemv(const Problem *probs, int count, void *stream);
// Test hook (mq_test_decode_kernel): 0 chooses the decode kernel by shape, 1
// takes the one-or-two-token kernel whenever it can serve the launch, 2 never.
int test_decode_kernel();
int launch_pack(const int8_t *w, int N, int K, int bits, void *packed, int32_t *colsum,
                int *status, void *stream);
// One row-sum job: out[m] = sum_k x[m][k] (mq_row_sums).
struct RowsumJob {
    const int8_t *x;
    int32_t *out;  // [M] in the workspace
    int32_t M, K, ldx;
};
constexpr int ROWSUM_MAX_JOBS = 64;  // jobs per launch (kernel parameter space)
int launch_rowsum(const RowsumJob *jobs, int count, void *stream);
int launch_transpose_i8(const int8_t *src, int rows, int cols, int lds, int8_t *dst, int ldd,
                        void *stream);

// One distinct int16 input of a batch and where its two int8 planes go:
// out row 2m = high bytes of x row m, row 2m + 1 = low bytes - 128 (pitch K).
struct SplitJob {
    const int16_t *x;
    int8_t *out;  // [2M][K] in the workspace
    int32_t M, K, ldx;
};
constexpr int SPLIT_MAX_JOBS = 64;
int launch_split16(const SplitJob *jobs, int count, void *stream);

// One distinct int8 input of a batch widened for the 256-token prefill kernel
// (mq_prefill2.cu): out = f16 copy [M][K] (pitch K), rowsq[m] = sum_k x[m][k]^2.
struct Widen16Job {
    const int8_t *x;
    uint16_t *out;
    int32_t *rowsq;
    int32_t M, K, ldx;
};
constexpr int WIDEN16_MAX_JOBS = 64;
int launch_widen16(const Widen16Job *jobs, int count, void *stream);
// The 256-token prefill kernel: problems with 8-bit activations and output;
// x16[i] / rowsq[i] are problem i's widened input and row sums of squares.
// y16[i] / ysq[i] (may be null): problem i's output also written as f16 and
// its row sums of squares added (the epilogue; y, the residual and ldy 4-byte
// aligned).
int launch_prefill2(const Problem *probs, const uint16_t *const *x16, const int32_t *const *rowsq,
                    uint16_t *const *y16, int32_t *const *ysq, int count, void *stream);
// wsq[n] = sum_k w[n][k]^2 of packed int8 / int4 weights (ldw bytes a row).
int launch_weight_sq(const uint8_t *packed, int N, int K, int bits, int ldw, int32_t *wsq,
                     void *stream);
// Whether the 256-token kernel can run on the current device (set-up done
// once per device; false when its register split does not fit the compiled
// kernel's launch allocation).
bool prefill2_ready();
// Test hook (mq_test_prefill_kernel): 0 chooses the prefill kernel by shape and
// workspace, 1 takes the 256-token kernel whenever it can serve a problem, 2 never.
int test_prefill_kernel();

// Boundary quantizers (mq_glue.cu): kind 0 quantize (float -> codes),
// 1 dequantize (codes -> f32), 2 requantize (codes -> codes); types are the
// MQ_TYPE_* of mq.h; [lo, hi] is the output code range.
int launch_glue(int kind, int in_type, int out_type, const void *in, void *out, int64_t n,
                float alpha, int32_t zin, int32_t zout, int32_t m0, int32_t shift, int32_t lo,
                int32_t hi, void *stream);

// Offline weight pipeline (mq_fold.cu): fold eq. 1 into f32 weights,
// quantize by `scheme` (MQ_WEIGHTS_*), pack, colsum; one batch of linears in
// three launches.
constexpr int FOLD_MAX_JOBS = MQ_FOLD_MAX_JOBS;
struct FoldJob {
    const float *w;
    int N, K;
    const float *s_in, *s_out;
    int bits, scheme;
    void *packed;
    int32_t *colsum;
    float *sw;
    int32_t *zw;
    float *stats;
};
int launch_fold(const FoldJob *jobs, int count, void *stream);

}  // namespace mq
