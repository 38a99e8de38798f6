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
 * is the tile width over N (128 or 256), or 0 for one tile per CTA over the whole GPU (tile
 * width a multiple of 16 up to 256 chosen from the SM count and M / 128; N % 16 == 0).
 * Requires M % 128 == 0, K % 64 == 0, N % bn == 0
 * (MCD_ERR_UNSUPPORTED otherwise; MCD_ERR_INVALID_ARG for null pointers or non-positive
 * sizes).  The caller keeps ownership of every buffer.  Allocates its own scratch (the
 * operands re-laid out in 128-byte swizzled tiles), runs on `stream` (a cudaStream_t, or
 * NULL for the default stream) and synchronises it before returning; MCD_ERR_TIMEOUT if a
 * device-side wait gave up. */
mcd_status mcd_tc_gemm(int32_t M, int32_t N, int32_t K, int32_t bn, const uint16_t* A, const uint16_t* B, float* Y,
                       void* stream);

/* The two halves of mcd_tc_gemm, for callers that lay an operand out once and multiply it
 * many times (weights) and for timing the product alone.
 *
 * mcd_tc_tile: re-lays the device bf16 matrix src, row-major [R][K] with a row stride of ld
 * elements (ld >= K), into the 128-byte swizzled tile layout the product reads: dst (device,
 * R * K * 2 bytes, 1024-byte aligned) holds k-slices of 64 columns, each R rows of 128
 * bytes in groups of 8 rows whose 16-byte chunks are permuted by row % 8.  Requires
 * R % 16 == 0 and K % 64 == 0 (MCD_ERR_UNSUPPORTED), non-null pointers and positive sizes
 * (MCD_ERR_INVALID_ARG).  Asynchronous on `stream`.
 *
 * mcd_tc_gemm_tiled: Y[n][m] = sum_k A[m][k] * B[n][k] from tiled A (M rows) and tiled B
 * (N rows), Y device fp32 [N][M]; bn 0, 128 or 256 and the shape rules of mcd_tc_gemm.  err
 * (device int32, zeroed by the caller) receives MCD_ERR_TIMEOUT if a device-side wait gives
 * up.  Asynchronous on `stream`: no allocation, no synchronisation; the caller owns every
 * buffer. */
mcd_status mcd_tc_tile(int32_t R, int32_t K, int32_t ld, const uint16_t* src, void* dst, void* stream);
mcd_status mcd_tc_gemm_tiled(int32_t M, int32_t N, int32_t K, int32_t bn, const void* A_tiled, const void* B_tiled,
                             float* Y, int32_t* err, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* MCD_TC_H */
