/*
 * CPU oracle for the BSR sparse x dense product -- TEST INFRASTRUCTURE ONLY.
 *
 * Only the tests, the smoke check and the CPU-baseline leg of the benchmark
 * may load this library. It shares no code with the CUDA path and the CUDA
 * path never calls it.
 *
 * Section 2.2 of the paper stores a pruned weight in Block Sparse Row form
 * ("data values, indices, and indptr") following SciPy, and multiplies the
 * kept blocks with the input tensor. With W[M, K] split into R x C blocks
 * (MB = M/R block rows, KB = K/C block columns; Eq. 3 gives the block
 * partition), the arrays are
 *   indptr[MB+1]  block-row offsets, indptr[0] = 0,
 *   indices[nnzb] block-column index of each kept block, ascending per row,
 *   data[nnzb][R][C] the block values, row-major inside the block,
 * and the product over kept blocks is
 *   Y[n, i*R + r] = b[i*R + r] + sum_{p in row i} sum_c X[n, indices[p]*C + c] * data[p][r][c].
 *
 * Everything accumulates in double (ref_bsr_spmm_f32acc: float, the timed
 * CPU baseline). Element types: ORACLE_F32 (float) or
 * ORACLE_BF16 (uint16 bfloat16 bit patterns, widened exactly).
 */
#ifndef REF_BSR_H
#define REF_BSR_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORACLE_F32 = 0, ORACLE_BF16 = 1 };

/* Block (i, j) is kept iff some element w of it has !(|w| <= thr), evaluated
 * in float (so a NaN keeps its block and -0.0 never does). Writes
 * indptr[MB+1] and returns nnzb, or -1 on a bad argument. */
int64_t ref_bsr_count(const void *W, int dtype, int64_t M, int64_t K, int R, int C,
                      float thr, int32_t *indptr);

/* Fills indices[nnzb] (ascending) and data[nnzb*R*C] (bit copies) for the
 * indptr that ref_bsr_count produced with the same arguments. Returns 0. */
int ref_bsr_fill(const void *W, int dtype, int64_t M, int64_t K, int R, int C, float thr,
                 const int32_t *indptr, int32_t *indices, void *data);

/* Scatters the stored blocks into a zeroed dense W_out[M, K]. */
void ref_bsr_to_dense(int dtype, int64_t M, int64_t K, int R, int C, const int32_t *indptr,
                      const int32_t *indices, const void *data, void *W_out);

/* Y[t, m] for the tokens rows[t] (t < n_rows; rows == NULL means token t),
 * before any rounding: double accumulation over the kept blocks in storage
 * order, then + bias[m] (bias may be NULL). X is [N, K] row-major. */
void ref_bsr_spmm(int dtype, int64_t M, int64_t K, int R, int C, const int32_t *indptr,
                  const int32_t *indices, const void *data, const void *X, const float *bias,
                  const int64_t *rows, int64_t n_rows, double *Y);

/* The error scale sum_k |X[n,k]| |W[m,k]| + |bias[m]| over the same tokens. */
void ref_bsr_err_bound(int dtype, int64_t M, int64_t K, int R, int C, const int32_t *indptr,
                       const int32_t *indices, const void *data, const void *X,
                       const float *bias, const int64_t *rows, int64_t n_rows, double *E);

/* Dense Y[t, m] = sum_k X[n_t, k] W[m, k] (k ascending, double) + bias[m]. */
void ref_dense_linear(int dtype, int64_t M, int64_t K, const void *W, const void *X,
                      const float *bias, const int64_t *rows, int64_t n_rows, double *Y);

/* As ref_bsr_spmm with a float accumulator, the timed CPU baseline: the
 * same order per output, every product and partial sum rounded to float,
 * then + bias[m] in float. Block rows are divided among `threads` OpenMP
 * threads (one thread per output, so results do not depend on the count). */
void ref_bsr_spmm_f32acc(int dtype, int64_t M, int64_t K, int R, int C, const int32_t *indptr,
                         const int32_t *indices, const void *data, const void *X, const float *bias,
                         const int64_t *rows, int64_t n_rows, float *Y, int threads);

/* Threads the library may use (1 when built without OpenMP). */
int ref_max_threads(void);

/* Round double results to the output element type: float (round to nearest
 * even), or bfloat16 bits (round to nearest even, overflow to infinity). */
void ref_round_f32(const double *in, float *out, int64_t n);
void ref_round_bf16(const double *in, uint16_t *out, int64_t n);

#ifdef __cplusplus
}
#endif
#endif
