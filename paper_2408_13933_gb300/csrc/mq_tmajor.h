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
// o16); returns MQ_OK or MQ_ERR_CUDA.
int launch_tmajor(const Problem *probs, int count, void *stream);
// Test hook (mq_test_tmajor_kernel): 0 takes the kernel for K <= 128 or
// N <= 64, 1 whenever it can serve a problem, 2 never.
int test_tmajor_kernel();

}  // namespace mq
