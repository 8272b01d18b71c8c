// mq_tmajor.h -- the token-major tensor-core kernel (mq_tmajor.cu): tokens as
// the MMA's M, for short K or few channels (the attention matmuls).
#pragma once

#include "mq_internal.h"

namespace mq {

// Whether the kernel can serve a prefill problem: int8 weights and
// activations, 16-byte aligned x and w with row pitches that are multiples
// of 16 bytes, no residual with an int16 output.
bool tmajor_suits(const Problem &p);
// Launcher (asynchronous on `stream`; the problems of one call have the same
// o16); returns MQ_OK or MQ_ERR_CUDA.  part[i] nonzero (part may be null):
// problem i is a slice of a split K whose y is an int32 [M][ldy] buffer of
// its raw sums sum (x - zx)(w - zw), requantized later by launch_splitk_reduce.
// wt[i] nonzero (wt may be null): problem i's w is stored transposed, int8
// [K][N] with ldw bytes between k-rows (not with part).
int launch_tmajor(const Problem *probs, int count, void *stream, const uint8_t *part = nullptr,
                  const uint8_t *wt = nullptr);

// One split problem's combine: y = requant(sum of the S slices' int32 sums,
// part + s M N, s < S) with M0 / shift / zy (+ residual for int8 outputs).
struct ReduceJob {
    const int32_t *part;
    int32_t S, M, N;
    const int32_t *M0, *shift;
    int32_t zy;
    const int8_t *residual;
    void *y;
    int32_t ldy, o16;
};
constexpr int REDUCE_MAX_JOBS = 32;
int launch_splitk_reduce(const ReduceJob *jobs, int count, void *stream);
// Test hook (mq_test_tmajor_kernel): 0 takes the kernel for K <= 128 or
// N <= 64, 1 whenever it can serve a problem, 2 never.
int test_tmajor_kernel();

}  // namespace mq
