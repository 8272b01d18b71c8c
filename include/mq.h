/*
 * mq.h -- C ABI of libmq, the GB300 (sm_103a) integer-only quantized linear
 * layer of MobileQuant (arXiv 2408.13933).
 *
 * The layer (Sec. 3.1; Sec. 4.2 eqs. 2-4; Sec. 5.1 and Appendix A):
 *   x  : int8 activations [M][ldx], static per-tensor scale sx and zero point zx
 *   w  : int8 or int4 weights [N][K], symmetric per output channel (scale sw[n],
 *        zero point 0), the learned equivalent transform already folded in
 *   acc[m][n] = sum_k (x[m][k] - zx) * w[n][k]
 *             = sum_k x[m][k] w[n][k] - zx * colsum[n]            (int32)
 *   y[m][n]   = clamp(zy + round_half_up(acc * M0[n] * 2^-shift[n]), -128, 127)
 *   optionally y[m][n] = clamp(y[m][n] + residual[m][n], -128, 127)
 * with M0[n] * 2^-shift[n] ~= sx * sw[n] / sy the fixed-point form of the
 * output quantizer of eq. 4 (alpha = sy, offset zy).
 *
 * Conventions for every call:
 *   - Every function returns an int status (mq_status); 0 is MQ_OK.  Nothing
 *     throws or aborts across the ABI.
 *   - All buffers belong to the caller.  The library allocates no memory.
 *   - "device" pointers are CUDA device addresses on the current device; "host"
 *     pointers are ordinary CPU memory.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Kernel launches are asynchronous on that stream; argument
 *     errors are reported before anything is launched.
 *   - Kernels never spin forever: every device-side wait has a time limit.  A
 *     kernel that hits it records MQ_ERR_DEVICE_TIMEOUT in a device status
 *     word, abandons its work and exits; mq_check_device_status() reports it.
 *   - Indices: M tokens, K input features, N output features.  All int8
 *     matrices are row-major with the feature index contiguous.
 */
#ifndef MQ_H
#define MQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MQ_OK = 0,
    MQ_ERR_INVALID_ARG = 1,       /* null pointer, bad range, bad bits, bad scale */
    MQ_ERR_UNSUPPORTED_SHAPE = 2, /* a dimension outside the supported range */
    MQ_ERR_K_OVERFLOW = 3,        /* K > MQ_MAX_K: int32 accumulator could overflow */
    MQ_ERR_ALIGNMENT = 4,         /* K, ldx or a pointer violates the 16-byte rule */
    MQ_ERR_CUDA = 5,              /* a CUDA runtime call failed */
    MQ_ERR_DEVICE_TIMEOUT = 6,    /* a kernel gave up on a bounded wait */
    MQ_ERR_WORKSPACE = 7          /* workspace missing or too small */
} mq_status;

/* |acc| <= 255 * 128 * K < 2^31 holds for every input when K <= 65536. */
#define MQ_MAX_K 65536
/* Largest number of linears in one mq_linear_batch call. */
#define MQ_MAX_BATCH 256

/* Human-readable name of a status code (static string, never NULL). */
const char *mq_status_string(int status);

/*
 * Fixed-point requantization parameters (Sec. 3.1: fixed-point operators;
 * eq. 4: output quantizer with static scale sy).  For each output channel n
 * the real multiplier M = (sx * sw[n]) / sy (IEEE double, in that order) is
 * written M = f * 2^e with f in [0.5, 1); then
 *     M0[n] = round_half_away(f * 2^31)   (if that equals 2^31: 2^30 and e+1)
 *     shift[n] = 31 - e                   (must lie in [1, 62])
 * so M0[n] * 2^-shift[n] = M within a relative 2^-31.  M < 2^-32 gives
 * M0 = 0, shift = 1 (output == zy).  M >= 2^30 is MQ_ERR_INVALID_ARG.
 *   sw    : host float [N], each finite and > 0
 *   sx, sy: finite and > 0
 *   M0, shift: host int32 [N], written by the call
 * Errors: MQ_ERR_INVALID_ARG (null pointer, N < 0, bad scale, M >= 2^30).
 */
int mq_requant_params(const float *sw, int N, float sx, float sy, int32_t *M0,
                      int32_t *shift);

/* Bytes of the packed weight buffer: N*K for bits 8, N*K/2 for bits 4.
 * Errors: MQ_ERR_INVALID_ARG (negative size, bits not 4/8, odd K for 4). */
int mq_packed_size(int N, int K, int bits, size_t *bytes);

/*
 * Pack weight values and compute colsum (the zero-point correction term of
 * the identity sum((x-zx)w) = sum(xw) - zx*colsum(w); eq. 4's offset applied
 * to the input).
 *   w      : int8 [N][K] values; for bits 4 each must lie in [-8, 7]
 *   bits   : 8 -> packed is an int8 copy [N][K];
 *            4 -> packed is uint8 [N][K/2], byte j of row n holds k = 2j in
 *                 bits 0-3 and k = 2j+1 in bits 4-7 (two's complement)
 *   packed : mq_packed_size bytes, written
 *   colsum : int32 [N], written: colsum[n] = sum_k w[n][k]
 *   on_device = 0: w, packed, colsum are host pointers; the call is synchronous.
 *   on_device = 1: they are device pointers; a kernel runs on `stream` and the
 *                  call waits for it (to report out-of-range int4 values).
 * Errors: MQ_ERR_INVALID_ARG (null, bad bits, odd K for int4, int4 value out
 * of range -- packed/colsum contents are then unspecified), MQ_ERR_CUDA.
 */
int mq_pack_weights(const int8_t *w, int N, int K, int bits, void *packed,
                    int32_t *colsum, int on_device, void *stream);

/*
 * Device workspace bytes a mq_linear_* call of this shape needs or can use.
 * Decode path (1 <= M <= 16): a fixed size (2.5 MB, the decode region)
 * holding, per CTA of the decode grid, int32 partial sums tagged with a
 * launch number, used to combine 64-row units whose K range is split among
 * CTAs.  Tensor-core path (M > 16) from M = 256 tokens and N = 256 output
 * channels on: room for the
 * 256-token kernel's widened input, i.e. an f16 copy of x (2 M K bytes) and
 * its row sums of squares (4 M bytes), placed after the size of the decode
 * region, each rounded up to 1024 bytes, plus 1024 bytes of alignment slack.
 * That part is optional: a prefill call given less (even no workspace) runs
 * the 128-token kernel instead, bit-identical and slower.  Prefill shapes
 * below that (M < 256 or N < 256, int8 weights, K >= 512) whose tiles would
 * leave most SMs idle: room, also optional, for S slices' int32 partial sums
 * (S M N 4 bytes, S = the SMs over the token-major kernel's tiles, at most 8,
 * from the first 1024-byte boundary after the decode region's size, plus 1024
 * bytes of slack): with it the call splits K over S launches' worth of tiles
 * and combines them in one more launch, bit-identical (a forced prefill kernel,
 * mq_test_prefill_kernel, never splits).  Otherwise 0.  For mq_linear_batch use
 * mq_workspace_size_batch.
 * Workspace contract: device memory, 16-byte aligned, zero-filled before its
 * first use.  The decode region (the first mq_workspace_size(1, 1, 0, 4)
 * bytes) is left zero-filled again by every call that completes, so the
 * workspace can be reused by later calls on the same stream; the widened
 * inputs and partial sums after it are scratch, overwritten by each call.  Calls that may run
 * concurrently (different streams) need different workspaces.  After
 * MQ_ERR_DEVICE_TIMEOUT the decode region must be zero-filled again.
 * Errors: MQ_ERR_INVALID_ARG.
 */
int mq_workspace_size(int M, int N, int K, int bits, size_t *bytes);

/*
 * One quantized linear layer, int8 activations x int8 weights (W8A8): the
 * integer-only linear of Sec. 3.1 (int8 x int8 products, int32 accumulation,
 * fixed-point requantization) with the static per-tensor activation
 * quantizer of eqs. 2-4 (Sec. 4.2) on its input (sx, zx) and output (sy, zy)
 * and symmetric per-channel weights (Appendix A).
 *   x        : device int8 [M][ldx], ldx >= K
 *   zx       : input zero point in [-128, 127]
 *   packed   : device, from mq_pack_weights(bits = 8)
 *   colsum   : device int32 [N]
 *   M0, shift: device int32 [N], from mq_requant_params
 *   zy       : output zero point in [-128, 127]
 *   y        : device int8 [M][ldy], ldy >= N, written
 *   workspace: device, ws_bytes >= mq_workspace_size (may be NULL when 0);
 *              see the workspace contract at mq_workspace_size
 * Requirements: 0 <= M, N; 0 <= K <= MQ_MAX_K; K % 16 == 0; ldx % 16 == 0;
 * x and packed 16-byte aligned.  Kernels are launched with programmatic
 * stream serialization: a call may start while the previous kernel in the
 * stream is finishing, and it reads `packed` (a constant input) before
 * waiting for that kernel; x, colsum, M0, shift, residual, y and the
 * workspace are touched only after it has completed.  So `packed` must not be
 * written by kernels still running in the same stream.  With K == 0 (every
 * output is requant(0), i.e. zy) x and packed are not read and may be NULL.  M <= 16 runs the
 * weight-streaming decode kernel, larger M the tcgen05 tensor-core kernel;
 * both are bit-exact.
 * Errors: MQ_ERR_INVALID_ARG, MQ_ERR_K_OVERFLOW, MQ_ERR_ALIGNMENT,
 * MQ_ERR_WORKSPACE (decode shape without a large enough workspace),
 * MQ_ERR_CUDA (launch failure).
 */
int mq_linear_w8a8(const int8_t *x, int M, int K, int ldx, int32_t zx,
                   const void *packed, const int32_t *colsum, int N,
                   const int32_t *M0, const int32_t *shift, int32_t zy,
                   int8_t *y, int ldy, void *workspace, size_t ws_bytes,
                   void *stream);

/* The same layer with int4 weights (W4A8; Sec. 5.1 W4A8 setting and the
 * symmetric per-channel scheme of Appendix A).  `packed` comes from
 * mq_pack_weights(bits = 4).  Requires K % 32 == 0 (16-byte weight rows);
 * other requirements and errors as mq_linear_w8a8. */
int mq_linear_w4a8(const int8_t *x, int M, int K, int ldx, int32_t zx,
                   const void *packed, const int32_t *colsum, int N,
                   const int32_t *M0, const int32_t *shift, int32_t zy,
                   int8_t *y, int ldy, void *workspace, size_t ws_bytes,
                   void *stream);

/*
 * mq_linear_w4a8 for decode shapes (1 <= M <= 16) without a workspace
 * argument and without allocating device memory.  The paper has no
 * counterpart: this is a deployment variant of the same layer.
 *
 * For callers that cannot provide device memory around a decode step: a C
 * program with no device allocator of its own, or a serving loop whose memory
 * pool is fixed after warm-up and must not grow mid-generation.  The split-K
 * combine scratch (2.5 MB) is a static device array inside libmq, one
 * per device, and no call allocates or frees device memory.  The scratch
 * needs no clearing: it starts zeroed, and each launch tags the sums it
 * leaves there with its own launch number, so a later launch ignores them
 * (also after MQ_ERR_DEVICE_TIMEOUT).
 *
 * The first call on each device does set-up with that device current: it
 * looks up the scratch's address and prepares both decode-kernel variants
 * (M <= 8 and M > 8).  Make that first call before any stream capture.  Every
 * call on a device shares the one scratch, so calls must not overlap: two
 * calls on different streams or from different host threads race and give
 * wrong results.  Calls issued in order on one stream are fine.
 *
 * Arguments and requirements as mq_linear_w4a8.  The result is identical to
 * mq_linear_w4a8 on the same inputs.
 * Errors: MQ_ERR_UNSUPPORTED_SHAPE for M > 16, which the scratch does not
 * hold (use mq_linear_w4a8); otherwise as mq_linear_w4a8, but
 * MQ_ERR_WORKSPACE does not occur.
 */
int mq_linear_w4a8_noalloc(const int8_t *x, int M, int K, int ldx, int32_t zx,
                           const void *packed, const int32_t *colsum, int N,
                           const int32_t *M0, const int32_t *shift, int32_t zy,
                           int8_t *y, int ldy, void *stream);

/*
 * One quantized linear layer with 16-bit activations and outputs (W8A16): the
 * paper's 16-bit-activation baseline and the width it keeps around
 * non-linear operators (Sec. 4.1, Sec. 5.6, Table 5).  The 16-bit code range
 * is the signed int16 range (the unsigned codes shifted by -32768).
 *   x        : device int16 [M][ldx] (ldx in elements), ldx >= K
 *   zx       : input zero point in [-32768, 32767]
 *   packed, colsum, M0, shift: as mq_linear_w8a8 (int8 weights)
 *   zy       : output zero point in [-32768, 32767]
 *   y        : device int16 [M][ldy], ldy >= N, written
 *   workspace: device, ws_bytes >= mq_workspace_size_a16(M, N, K, 8)
 *   acc[m][n] = sum_k (x[m][k] - zx) * w[n][k]        (exact, |acc| < 2^40)
 *   y[m][n]   = clamp(zy + floor(acc M0[n] / 2^shift[n] + 1/2), -32768, 32767)
 * Method: with hi the signed high byte and lo the unsigned low byte of a
 * code, x = 256 hi + (lo - 128) + 128; both planes hi and lo - 128 are int8
 * values, which the int8 kernels contract exactly, and their epilogues form
 * 256 S_hi + S_lo + (128 - zx) colsum[n] in int64 and requantize it.
 * 2M <= 16 runs the decode kernel, which splits the codes into the planes
 * as it builds its operands; larger M runs the tensor-core kernel after a
 * pre-pass that writes the planes as rows 2m and 2m+1 of a [2M][K] int8
 * matrix in the workspace.
 * Requirements: 0 <= M, N; 0 <= K <= MQ_MAX_K; K % 16 == 0; ldx % 8 == 0;
 * x and packed 16-byte aligned.  No residual.  Weights with a zero point
 * (the matmul of self-attention in the paper's W8A16 setting, between 16-bit
 * and 8-bit activations, Sec. 5.6) go through mq_linear_batch with `zw` and
 * abits 16: acc = sum_k (x - zx)(w - zw[n]), exact in int64 for every K.  The
 * stream rules of mq_linear_w8a8 apply.
 * Errors: MQ_ERR_INVALID_ARG, MQ_ERR_K_OVERFLOW, MQ_ERR_ALIGNMENT,
 * MQ_ERR_WORKSPACE, MQ_ERR_CUDA.
 */
int mq_linear_w8a16(const int16_t *x, int M, int K, int ldx, int32_t zx,
                    const void *packed, const int32_t *colsum, int N,
                    const int32_t *M0, const int32_t *shift, int32_t zy,
                    int16_t *y, int ldy, void *workspace, size_t ws_bytes,
                    void *stream);

/* The same layer with int4 weights (W4A16).  Requires K % 32 == 0; otherwise
 * as mq_linear_w8a16. */
int mq_linear_w4a16(const int16_t *x, int M, int K, int ldx, int32_t zx,
                    const void *packed, const int32_t *colsum, int N,
                    const int32_t *M0, const int32_t *shift, int32_t zy,
                    int16_t *y, int ldy, void *workspace, size_t ws_bytes,
                    void *stream);

/*
 * Device workspace bytes of one mq_linear_w8a16 / mq_linear_w4a16 call: the
 * decode workspace (see mq_workspace_size) when 1 <= 2M <= 16; otherwise the
 * two int8 planes of x (2 M K bytes, rounded up to 128), which are scratch,
 * overwritten by each call.  The decode part follows the contract of
 * mq_workspace_size.
 * Errors: MQ_ERR_INVALID_ARG.
 */
int mq_workspace_size_a16(int M, int N, int K, int bits, size_t *bytes);

/*
 * Several independent linears in as few launches as possible (one per kernel
 * family): a decoder block's projections that read the same activations, or
 * a whole step's worth of small decode GEMVs.  Each descriptor has the
 * meaning and requirements of one mq_linear_w8a8 / mq_linear_w4a8 call (with
 * abits 16: mq_linear_w8a16 / mq_linear_w4a16); in
 * addition `residual` (device int8 [M][ldy], may be NULL) is added to the
 * requantized output with int8 saturation, the int8 residual glue between
 * chained layers.  Descriptors must not write overlapping outputs.
 *
 * Asymmetric weights: `zw` (device int32 [N], may be NULL for symmetric
 * weights) is a per-output-channel weight zero point, the asymmetric weight
 * quantizer of the paper's main W8A8 / W4A8 runs (Sec. 4.2 eqs. 2-4 applied
 * to weights, Sec. 5.1; a per-tensor zero point is the case of equal zw[n]):
 *   acc[m][n] = sum_k (x[m][k] - zx) * (w[n][k] - zw[n])
 *             = sum_k x (w - zw[n]) - zx (colsum[n] - K zw[n])
 * zw[n] must lie in the weight code range ([-128, 127] for bits 8, [-8, 7]
 * for bits 4), and with int8 weights and 8-bit activations K <= MQ_MAX_K_ASYM8
 * (so that |acc| <= 255 * 255 * K stays below 2^31; 16-bit activations
 * accumulate in int64).  No workspace beyond that of the
 * symmetric case: the weights are widened to w - zw[n] on the fly.
 *
 *   descs     : host array of `count` descriptors (1 <= count <= MQ_MAX_BATCH)
 *   workspace : device, ws_bytes >= mq_workspace_size_batch(descs, count)
 * Errors: as the single calls, and MQ_ERR_K_OVERFLOW for int8 weights with
 * zw and K > MQ_MAX_K_ASYM8; the index of the first bad descriptor is not
 * reported, nothing is launched when any descriptor is invalid.
 *
 * 16-bit output from 8-bit inputs (abits 8, obits 16): y is int16 [M][ldy]
 * and zy lies in [-32768, 32767]; everything else is as for 8-bit outputs,
 * without a residual.  For products whose result feeds a non-linear operator,
 * which MobileQuant keeps in 16-bit integers (Sec. 4.1): the attention scores
 * Q K^T ahead of the softmax, with the keys as the "weights" (their zero point
 * as zw, their row sums from mq_row_sums as colsum).
 * Weight row pitch: `ldw` bytes between weight rows (0: K * bits / 8; else at
 * least that and a multiple of 16), so that a head's slice of a projection
 * output ([T][heads * d], one head's d columns) can serve as the weights
 * without a copy.
 * Row sums derived by the call: in a descriptor with int8 weights, `colsum`
 * may be NULL.  The token-major kernel (mq_test_tmajor_kernel) contracts
 * x - zx and w - zw directly and needs no row sums; for a problem any other
 * kernel serves, the call first computes colsum[n] = sum_k w[n][k] into its
 * workspace (N * 4 bytes per distinct weight matrix, counted by
 * mq_workspace_size_batch; rounded up to 128 bytes).  For weights written on
 * the device every call (keys, V^T in attention) this replaces a separate
 * row-sum launch.  The single-linear calls still require colsum.
 * Transposed weights (`wt`, int8 weights with 8-bit activations, else
 * MQ_ERR_INVALID_ARG): `packed` holds w[n][k] at packed[k * ldw + n], i.e. an
 * activation matrix [K][N] such as V in attention's P V (its head-g columns
 * with ldw = the row pitch of V), read without a transpose.  ldw is at least
 * N (0 means N; smaller: MQ_ERR_INVALID_ARG) and, when given, a multiple of 16
 * (else MQ_ERR_ALIGNMENT, as for unaligned x or packed).  Only the token-major
 * kernel reads this layout: with K > 0 the descriptor must be a prefill shape
 * (M > 16) that kernel can serve (rows of x and of packed 16-byte multiples, no
 * residual with an int16 output); otherwise, or with the token-major kernel
 * forbidden (mq_test_tmajor_kernel), the call returns MQ_ERR_UNSUPPORTED_SHAPE
 * before anything is launched.  colsum is not read (the kernel folds the zero
 * points).
 * Weights written on the device: the kernels read `packed` before waiting for
 * the previous kernel in the stream (see mq_linear_w8a8).  A descriptor whose
 * weights are produced by earlier work on the same stream (keys, or V^T from
 * mq_transpose_i8, in attention) sets `wdynamic` nonzero; every launch that
 * holds such a descriptor then reads all its weights after the previous
 * kernel has completed.
 */
typedef struct mq_linear_desc {
    const void *x;          /* int8 [M][ldx], or int16 with abits == 16 */
    const void *packed;
    const int32_t *colsum;  /* may be NULL with int8 weights (bits 8), see below */
    const int32_t *M0;
    const int32_t *shift;
    const int8_t *residual; /* may be NULL; int8 activations only */
    const int32_t *zw;      /* may be NULL: symmetric weights */
    void *y;                /* int8 [M][ldy], or int16 with abits == 16 */
    int32_t M, N, K, ldx, ldy;
    int32_t zx, zy;
    int32_t bits;  /* weight bits: 8 or 4 */
    int32_t abits; /* activation and output bits: 8 (0 reads as 8) or 16, see mq_linear_w8a16 */
    int32_t obits; /* output bits: 0 (= abits), or 16 with abits 8: int16 y, see below */
    int32_t ldw;   /* bytes between weight rows; 0: packed rows (K * bits / 8) */
    int32_t wdynamic; /* nonzero: packed is written by earlier work on the stream, see above */
    const int32_t *wsq; /* may be NULL: device int32 [N], wsq[n] = sum_k w[n][k]^2 of the weight
                           codes (mq_weight_sq_sums), see below */
    void *y16;          /* may be NULL: device f16 [M][N], also written: y as f16, see below */
    int32_t *ysq;       /* with y16: device int32 [M], zero-filled by the caller; the call adds
                           sum_n y[m][n]^2 */
    const void *x16;    /* may be NULL: device f16 [M][K], an f16 copy of x (a y16 of an earlier
                           call), see below */
    const int32_t *xsq; /* with x16: device int32 [M], sum_k x[m][k]^2 (that call's ysq) */
    int32_t wt;         /* nonzero: packed holds the weights transposed, int8 [K][N] with
                           `ldw` bytes between k-rows (0: N), see below */
} mq_linear_desc;

/*
 * Weight sums of squares (`wsq`, optional, symmetric weights only): the
 * tensor-core kernel sums the exact products in f32 runs that must stay
 * within 2^24.  With wsq it bounds every partial sum of a tile by
 * sqrt(max_m sum_k x[m][k]^2 * max_n wsq[n]) (Cauchy-Schwarz) and, where that
 * bound allows, sums the whole K in one run; without it the bound takes
 * |w| <= 128 and long K splits into several runs.  Either way the result is
 * exact; wsq is read only by the 256-token prefill kernel, and only when it
 * has no weight zero point.  Like colsum it is a per-weight constant: compute
 * it once with mq_weight_sq_sums.
 */

/*
 * Chained layers (`y16` / `ysq`, `x16` / `xsq`, optional, 8-bit activations and
 * output): the 256-token prefill kernel contracts an f16 copy of x and needs
 * each token row's sum of squares; by default every call computes both in a
 * pre-pass into its workspace.  A call given `y16` and `ysq` also writes its
 * output y (after the residual) as f16 [M][N] (pitch N) into y16 and adds each
 * row's sum of squares into ysq (zero-filled by the caller): where the
 * 256-token kernel computes y, its epilogue does this on the way out, otherwise
 * the call runs the pre-pass on y after computing it.  A later call whose x is
 * that y passes them as `x16` / `xsq` and skips its pre-pass for that input.
 * The copy must be of x exactly (the kernel contracts x16, not x).
 * Requirements: y16 with ysq, x16 with xsq, both only with abits 8 and obits
 * 8; y16 and x16 16-byte aligned; with y16, N % 16 == 0, ldy % 16 == 0 and y
 * 16-byte aligned.
 */

/* Largest K for int8 weights with a weight zero point: 255 * 255 * K < 2^31. */
#define MQ_MAX_K_ASYM8 32768

/*
 * Device workspace bytes one mq_linear_batch call over `descs` needs: the
 * decode workspace (see mq_workspace_size) if any descriptor has
 * 1 <= M <= 16 (abits 8) or 1 <= 2M <= 16 (abits 16); plus 2*M*K bytes
 * (rounded up to 128) for every distinct input (x, M, K, ldx) of the
 * descriptors with abits 16 and 2M > 16, which holds its two int8 planes
 * (filled by the call; descriptors reading the same input, e.g. q/k/v/gate/up
 * of one block, share them).  Then, optionally, room for the 256-token
 * prefill kernel (see mq_workspace_size): for every distinct 8-bit input of
 * the descriptors with abits 8, obits 8, M >= 256 and N >= 256, its f16 copy (2 M K
 * bytes) and row sums of squares (4 M bytes), each rounded up to 1024, placed
 * after the decode region's size, plus 1024 bytes of alignment slack; a call
 * given only the required part runs those descriptors on the 128-token
 * kernel.  The required part also holds, for descriptors without colsum that
 * the token-major kernel does not serve, their weights' row sums (4 N bytes,
 * rounded up to 128, per distinct weight matrix).  Last, optionally, the
 * split-K partial sums, for a call made only of small prefill descriptors (see
 * mq_workspace_size; S is shared by the call, from all of them).  0 when none
 * applies.  The decode region (the first
 * mq_workspace_size(1, 1, 0, 4) bytes) follows the contract of
 * mq_workspace_size: zero-filled before first use and left zero by every
 * call that completes; the other regions are scratch, overwritten by each
 * call.
 * Errors: MQ_ERR_INVALID_ARG (null pointers, count out of range, bad bits or
 * abits).
 */
int mq_workspace_size_batch(const mq_linear_desc *descs, int count, size_t *bytes);

int mq_linear_batch(const mq_linear_desc *descs, int count, void *workspace,
                    size_t ws_bytes, void *stream);

/* ---- Boundary quantizers --------------------------------------------------
 * The steps on either side of the linear in an integer block: activations of
 * linears are 8-bit, those around non-linear operators 16-bit integers
 * (Sec. 4.1), and every change of domain is a static per-tensor quantizer
 * (Sec. 3.1).  Element types: */
#define MQ_TYPE_F32 0
#define MQ_TYPE_F16 1
#define MQ_TYPE_BF16 2
#define MQ_TYPE_I8 3
#define MQ_TYPE_I16 4

/*
 * Static per-tensor activation quantizer, the forward quantizer of eqs. 2-4
 * (Sec. 4.2) in the signed code range:
 *   q[i] = clamp(rint(x[i] / alpha) + z, qmin, qmax)
 * x[i] / alpha is the correctly rounded f32 quotient (f16 and bf16 values are
 * widened to f32 exactly first); rint rounds ties to even; NaN gives z and
 * +-inf saturates.
 *   x     : device, n values of in_type (MQ_TYPE_F32, MQ_TYPE_F16, MQ_TYPE_BF16)
 *   q     : device, n codes of out_type (MQ_TYPE_I8 or MQ_TYPE_I16), written
 *   alpha : finite, > 0;  z inside the output code range
 * Requirements: n >= 0; x and q aligned to their element size (16-byte
 * alignment of both takes the vector path).  Launched with programmatic
 * stream serialization; x is read only after the previous kernel completes.
 * Errors: MQ_ERR_INVALID_ARG, MQ_ERR_CUDA.
 */
int mq_quantize(const void *x, int in_type, int64_t n, float alpha, int32_t z, void *q,
                int out_type, void *stream);

/*
 * Dequantization f[i] = (q[i] - z) * alpha, rounded once to f32.
 *   q: device, n codes of in_type (MQ_TYPE_I8 or MQ_TYPE_I16); f: device f32 [n]
 *   alpha finite; z inside the input code range.  Otherwise as mq_quantize.
 */
int mq_dequantize(const void *q, int in_type, int64_t n, float alpha, int32_t z, float *f,
                  void *stream);

/*
 * Fixed-point requantization between integer domains (int8 / int16 codes in,
 * int8 / int16 codes out):
 *   y[i] = clamp(zy + floor(((q[i] - zx) M0 + 2^(shift-1)) / 2^shift), ymin, ymax)
 * with M0 * 2^-shift ~= alpha_in / alpha_out, e.g. from
 * mq_requant_params(&alpha_in, 1, 1.0f, alpha_out, &M0, &shift).
 *   q, y : device, n codes of in_type / out_type (MQ_TYPE_I8 or MQ_TYPE_I16)
 *   zx, zy inside their code ranges; 0 <= M0 < 2^31; 1 <= shift <= 62
 * Otherwise as mq_quantize.
 */
int mq_requantize(const void *q, int in_type, int64_t n, int32_t zx, int32_t M0, int32_t shift,
                  int32_t zy, void *y, int out_type, void *stream);

/* ---- Offline weight pipeline ---------------------------------------------- */
#define MQ_WEIGHTS_SYM_CHANNEL 0  /* symmetric per output channel (Appendix A) */
#define MQ_WEIGHTS_ASYM_CHANNEL 1 /* asymmetric per output channel (Sec. 5.1: W4A8, down_proj) */
#define MQ_WEIGHTS_ASYM_TENSOR 2  /* asymmetric per tensor (Sec. 5.1: W8A8) */

/*
 * The producer of the weights the layer consumes, on the device, for one
 * linear: fold the equivalent transform of eq. 1 into f32 weights, quantize,
 * pack and compute colsum.  Weights are stored [N out][K in]; eq. 1's S W
 * scales input channel k by s_in[k], and the S^-1 of the next transform
 * (Figure 3: S0 W1 S1^-1, S1 W2) scales output channel n by 1 / s_out[n]:
 *   w'[n][k] = (w[n][k] * s_in[k]) / s_out[n]          (f32, multiply first)
 * then, with every step one f32 operation rounded to nearest:
 *   MQ_WEIGHTS_SYM_CHANNEL: amax = max|w'[n]| (1e-8 if 0), sw = amax / qmax,
 *     q = clamp(rint(w' / sw), -qmax, qmax), qmax 127 (int8); for int4
 *     clamp(., -8, 7) with qmax 7; zw = 0.
 *   MQ_WEIGHTS_ASYM_CHANNEL / _TENSOR: lo = min(min w', 0), hi = max(max w', 0)
 *     over the channel / the tensor, sw = (hi - lo) / (qmax - qmin) (1e-8
 *     span if 0), zw = clamp(rint(qmin - lo / sw)), q = clamp(rint(w' / sw) + zw).
 * rint rounds ties to even.
 *   w       : device f32 [N][K], finite values
 *   s_in    : device f32 [K] or NULL;  s_out: device f32 [N] or NULL (positive)
 *   packed, colsum : as mq_pack_weights(bits) (colsum of the codes)
 *   sw      : device f32 [N], the weight scales (for mq_requant_params)
 *   zw      : device int32 [N], the weight zero points (the `zw` of
 *             mq_linear_desc); may be NULL for MQ_WEIGHTS_SYM_CHANNEL
 *   stats   : device f32 [2N] scratch
 * Requirements: N, K >= 0; bits 8, or 4 with K even; pointers aligned to
 * their element size.  Asynchronous on `stream`.
 * Errors: MQ_ERR_INVALID_ARG, MQ_ERR_ALIGNMENT, MQ_ERR_CUDA.
 */
int mq_fold_quantize_pack(const float *w, int N, int K, const float *s_in, const float *s_out,
                          int bits, int scheme, void *packed, int32_t *colsum, float *sw,
                          int32_t *zw, float *stats, void *stream);

/*
 * mq_fold_quantize_pack over up to MQ_FOLD_MAX_JOBS linears (e.g. the seven of
 * one transformer block) in three launches instead of two or three per
 * linear: the row statistics of every linear, the per-tensor reductions, then
 * every linear's codes.  Each descriptor's fields are the arguments of
 * mq_fold_quantize_pack, with the same requirements; every descriptor is
 * checked before anything is launched.  Outputs (and the stats scratch) of
 * different descriptors must not overlap.  The result is byte-identical to
 * one mq_fold_quantize_pack call per descriptor.
 * Errors: MQ_ERR_INVALID_ARG (also count < 0 or > MQ_FOLD_MAX_JOBS, descs NULL
 * with count > 0), MQ_ERR_ALIGNMENT, MQ_ERR_CUDA.
 */
#define MQ_FOLD_MAX_JOBS 32
typedef struct mq_fold_desc {
    const float *w;
    int32_t N, K;
    const float *s_in, *s_out;
    int32_t bits, scheme;
    void *packed;
    int32_t *colsum;
    float *sw;
    int32_t *zw;
    float *stats;
} mq_fold_desc;
int mq_fold_quantize_pack_batch(const mq_fold_desc *descs, int count, void *stream);

/*
 * The norm's affine before the first transformed linear absorbs S0^-1
 * (Figure 3): gamma_out[k] = gamma[k] / s[k], beta_out[k] = beta[k] / s[k],
 * f32.  Host arrays; beta and beta_out may be NULL (RMSNorm has no shift).
 * Errors: MQ_ERR_INVALID_ARG.
 */
int mq_fold_norm(const float *gamma, const float *beta, const float *s, int K, float *gamma_out,
                 float *beta_out);

/*
 * wsq[n] = sum_k w[n][k]^2 (int32) of packed weights (mq_pack_weights layout,
 * `bits` 8 or 4; `ldw` bytes between rows, 0 for packed rows): the optional
 * `wsq` field of mq_linear_desc.  Requirements: N, K >= 0; K % 16 == 0 (int8)
 * or K % 32 == 0 (int4); K <= MQ_MAX_K; packed 16-byte aligned; ldw 0 or at
 * least K * bits / 8 and a multiple of 16.  Asynchronous on `stream`.
 * Errors: MQ_ERR_INVALID_ARG, MQ_ERR_ALIGNMENT, MQ_ERR_CUDA.
 */
int mq_weight_sq_sums(const void *packed, int N, int K, int bits, int ldw, int32_t *wsq,
                      void *stream);

/* ---- Attention matmul glue ------------------------------------------------ */

/*
 * out[m] = sum_k x[m][k] (int32) for int8 x [M][ldx]: the colsum of an
 * activation matrix used as the "weights" operand (the keys of Q K^T, V^T of
 * P V), or any row sum.  Requirements: M, K >= 0; K % 16 == 0; ldx >= K,
 * ldx % 16 == 0; x 16-byte aligned; K <= MQ_MAX_K.  Asynchronous on
 * `stream` (programmatic dependent launch: x is read after the previous
 * kernel completes).
 * Errors: MQ_ERR_INVALID_ARG, MQ_ERR_ALIGNMENT, MQ_ERR_CUDA.
 */
int mq_row_sums(const int8_t *x, int M, int K, int ldx, int32_t *out, void *stream);

/*
 * out[h][m] = sum_{k < d} x[m][h d + k] (int32) for int8 x [M][ldx] and h < heads:
 * the row sums of every head slice of a projection output [T][heads d] in one
 * launch (the keys' colsum of every KV head for Q K^T).  out is [heads][M]
 * (device int32, written).  Requirements: M, d >= 0; 0 <= heads; d % 16 == 0;
 * ldx >= heads d, ldx % 16 == 0; x 16-byte aligned; d <= MQ_MAX_K.  Asynchronous
 * on `stream` (programmatic dependent launch: x is read after the previous
 * kernel completes).
 * Errors: MQ_ERR_INVALID_ARG, MQ_ERR_ALIGNMENT, MQ_ERR_CUDA.
 */
int mq_head_row_sums(const int8_t *x, int M, int heads, int d, int ldx, int32_t *out,
                     void *stream);

/*
 * dst[c][r] = src[r][c] for int8 src [rows][lds] -> dst [cols][ldd] (lds >=
 * cols, ldd >= rows): V [T][d] -> V^T [d][T], the K-major "weights" operand of
 * P V.  Asynchronous on `stream`.
 * Errors: MQ_ERR_INVALID_ARG, MQ_ERR_CUDA.
 */
int mq_transpose_i8(const int8_t *src, int rows, int cols, int lds, int8_t *dst, int ldd,
                    void *stream);

/*
 * Wait for `stream` and report device-side failures recorded by this
 * library's kernels since the previous call: MQ_ERR_DEVICE_TIMEOUT if a
 * bounded wait expired, MQ_ERR_CUDA if the stream reports a CUDA error,
 * MQ_OK otherwise.  Clears the recorded status.
 */
int mq_check_device_status(void *stream);

/* ---- Failure detection ----------------------------------------------------
 * The paper has no counterpart: these calls serve the library's own failure
 * detection.  Every device-side wait of the kernels (a pipeline barrier, a
 * split-K partner's partial sums) gives up after a time limit; the kernel
 * then records MQ_ERR_DEVICE_TIMEOUT (see mq_check_device_status), abandons
 * its work -- outputs are unspecified -- after letting its in-flight copies
 * and tensor-core operations finish, and exits, so the CUDA context stays
 * usable.
 */

/*
 * Set the limit of every device-side wait, in nanoseconds, for the launches
 * made after this call (process-wide, all devices).  0 restores the default
 * of 1 second; values below 1000 are raised to 1000.  A short limit makes a
 * wait that cannot complete end quickly in a test; in production a limit far
 * above any real wait (the default) only bounds a hang.
 * Errors: MQ_ERR_INVALID_ARG above 60 seconds.
 */
int mq_set_wait_limit_ns(uint64_t ns);

/*
 * Test hook, not for production: from this call on, CTA `cta` of every
 * decode-kernel launch (mq_linear_* with M <= 16, the batch call's decode
 * launches, mq_linear_w4a8_noalloc) skips storing the partial sums of a
 * 64-row unit it shares with an earlier CTA.  The earlier CTA's bounded wait
 * for them then runs out and the launch reports MQ_ERR_DEVICE_TIMEOUT: a
 * split-K partner that never delivers, made on purpose without any fault.
 * -1 (the initial state) turns it off.  After such a timeout a workspace
 * keeps stale entries of that launch; the kernels ignore them (every launch
 * tags its entries with its own number), and zero-filling it again restores
 * the zero-filled state of the workspace contract.
 * Errors: MQ_ERR_INVALID_ARG for cta < -1 or beyond the decode grid.
 */
int mq_test_skip_partials(int cta);

/*
 * Test hook, not for production: the choice between the two decode kernels
 * (M <= 16).  0 (the initial state) chooses by shape: launches of one to four
 * tokens with 8-bit activations whose row groups balance over the SMs take the
 * row-group kernel (each warp streaming a run of 4-row groups), the others the
 * split-K kernel.  1 takes the row-group kernel for every launch it
 * can serve (any such shape, however small), 2 never.  Both are bit-exact; the
 * hook lets the tests run either one on any shape.
 * Errors: MQ_ERR_INVALID_ARG for values other than 0, 1, 2.
 */
int mq_test_decode_kernel(int which);

/*
 * Test hook, not for production: the choice between the two prefill kernels
 * for problems with 8-bit activations and outputs (M > 16).  0 (the initial
 * state) takes the 256-token kernel for M >= 256 and N >= 256 when the workspace has room
 * for the widened inputs (mq_workspace_size, mq_workspace_size_batch count
 * it), the 128-token kernel otherwise.  1 takes the 256-token kernel for every
 * such problem the workspace allows, 2 never.  Both are bit-exact; the hook
 * lets the tests run either one on any shape.
 * Errors: MQ_ERR_INVALID_ARG for values other than 0, 1, 2.
 */
int mq_test_prefill_kernel(int which);

/*
 * Test hook, not for production: the token-major kernel (tokens as the
 * tensor-core MMA's M, 128 a tile; channels as its N) for prefill problems
 * with 8-bit activations and int8 weights, 16-byte aligned x and weights with
 * row pitches that are multiples of 16 bytes, and no residual with an int16
 * output.  0 (the initial state) takes it for such problems with K <= 128 or
 * N <= 64 (the attention matmuls: Q K^T at head dimension K, P V with head
 * dimension N) unless mq_test_prefill_kernel forces the 256-token kernel, 1
 * for every such problem, 2 never.  All kernels are bit-exact; the hook lets
 * the tests run each one on any shape.
 * Errors: MQ_ERR_INVALID_ARG for values other than 0, 1, 2.
 */
int mq_test_tmajor_kernel(int which);

#ifdef __cplusplus
}
#endif
#endif /* MQ_H */
