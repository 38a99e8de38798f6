/* libmcd: the tensor-core GEMM of the batched path, exposed for tests and measurement.
 *
 * With hundreds of packed rows per call (many streams decoded together, Sec. 1 of
 * arXiv 2609.37007: the MultiCodeDecoder's inner loop shared by many utterances) the
 * weight products of a verify call are real GEMMs, Y = X W^T with W the [out, in] weight
 * matrix.  The library computes them on the 5th-generation tensor cores (tcgen05.mma,
 * bf16 operands, fp32 accumulation in tensor memory).
 *
 * Conventions are those of mcd.h: a status is returned, nothing aborts across the ABI.
 */
#ifndef MCD_TC_H
#define MCD_TC_H

#include "mcd.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Y[n][m] = sum_k A[m][k] * B[n][k] for m < M, n < N: A device bf16 (uint16 bit patterns)
 * row-major [M][K], B device bf16 row-major [N][K], Y device fp32 row-major [N][M]; bn
 * is the tile width over N (128 or 256).  Requires M % 128 == 0, K % 64 == 0, N % bn == 0
 * (MCD_ERR_UNSUPPORTED otherwise; MCD_ERR_INVALID_ARG for null pointers or non-positive
 * sizes).  The caller keeps ownership of every buffer.  Allocates its own scratch (the
 * operands re-laid out in 128-byte swizzled tiles), runs on `stream` (a cudaStream_t, or
 * NULL for the default stream) and synchronises it before returning; MCD_ERR_TIMEOUT if a
 * device-side wait gave up. */
mcd_status mcd_tc_gemm(int32_t M, int32_t N, int32_t K, int32_t bn, const uint16_t* A, const uint16_t* B, float* Y,
                       void* stream);

#ifdef __cplusplus
}
#endif

#endif /* MCD_TC_H */
