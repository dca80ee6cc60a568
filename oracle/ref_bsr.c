/*
 * CPU oracle for the BSR sparse x dense product -- TEST INFRASTRUCTURE ONLY.
 * Plain, slow and written straight from the definitions; see ref_bsr.h.
 *
 * Built with -ffp-contract=off so that no multiply-add is fused: every sum is
 * the plain left-to-right double sum in the order the definitions state.
 */
#include "ref_bsr.h"

#include <math.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* bfloat16 is the top half of a float: widening is a 16-bit shift. */
static float bf16_to_float(uint16_t h) {
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

static float elem_f(const void *a, int dtype, int64_t i) {
    if (dtype == ORACLE_F32) return ((const float *)a)[i];
    return bf16_to_float(((const uint16_t *)a)[i]);
}

static double elem(const void *a, int dtype, int64_t i) { return (double)elem_f(a, dtype, i); }

static size_t elem_size(int dtype) { return dtype == ORACLE_F32 ? 4 : 2; }

/* Keep rule for one element (Section 2.2 keeps the non-zero blocks; the
 * threshold generalises "non-zero" to "above thr in magnitude"). */
static int keeps(float w, float thr) { return !(fabsf(w) <= thr); }

static int block_kept(const void *W, int dtype, int64_t K, int R, int C, float thr, int64_t i,
                      int64_t j) {
    for (int r = 0; r < R; r++)
        for (int c = 0; c < C; c++)
            if (keeps(elem_f(W, dtype, (i * R + r) * K + j * C + c), thr)) return 1;
    return 0;
}

static int bad_shape(int64_t M, int64_t K, int R, int C, int dtype) {
    return M < 0 || K < 0 || R <= 0 || C <= 0 || M % R || K % C ||
           (dtype != ORACLE_F32 && dtype != ORACLE_BF16);
}

int64_t ref_bsr_count(const void *W, int dtype, int64_t M, int64_t K, int R, int C, float thr,
                      int32_t *indptr) {
    if (bad_shape(M, K, R, C, dtype)) return -1;
    int64_t MB = M / R, KB = K / C, nnzb = 0;
    indptr[0] = 0;
    for (int64_t i = 0; i < MB; i++) {
        for (int64_t j = 0; j < KB; j++) nnzb += block_kept(W, dtype, K, R, C, thr, i, j);
        indptr[i + 1] = (int32_t)nnzb;
    }
    return nnzb;
}

int ref_bsr_fill(const void *W, int dtype, int64_t M, int64_t K, int R, int C, float thr,
                 const int32_t *indptr, int32_t *indices, void *data) {
    int64_t MB = M / R, KB = K / C;
    size_t es = elem_size(dtype);
    for (int64_t i = 0; i < MB; i++) {
        int64_t p = indptr[i];
        for (int64_t j = 0; j < KB; j++) {
            if (!block_kept(W, dtype, K, R, C, thr, i, j)) continue;
            indices[p] = (int32_t)j;
            for (int r = 0; r < R; r++)
                for (int c = 0; c < C; c++)
                    memcpy((char *)data + ((p * R + r) * C + c) * es,
                           (const char *)W + ((i * R + r) * K + j * C + c) * es, es);
            p++;
        }
    }
    return 0;
}

void ref_bsr_to_dense(int dtype, int64_t M, int64_t K, int R, int C, const int32_t *indptr,
                      const int32_t *indices, const void *data, void *W_out) {
    int64_t MB = M / R;
    size_t es = elem_size(dtype);
    memset(W_out, 0, (size_t)(M * K) * es);
    for (int64_t i = 0; i < MB; i++)
        for (int64_t p = indptr[i]; p < indptr[i + 1]; p++)
            for (int r = 0; r < R; r++)
                for (int c = 0; c < C; c++)
                    memcpy((char *)W_out + ((i * R + r) * K + (int64_t)indices[p] * C + c) * es,
                           (const char *)data + ((p * R + r) * C + c) * es, es);
}

/* One output element of the BSR product before the bias: the kept blocks of
 * block row i in storage order, the columns of each block in order. When
 * absolute != 0 the same loop sums |x| |w| instead (the error scale). */
static double row_dot(int dtype, int64_t K, int R, int C, const int32_t *indptr,
                      const int32_t *indices, const void *data, const void *X, int64_t n,
                      int64_t i, int r, int absolute) {
    double acc = 0.0;
    for (int64_t p = indptr[i]; p < indptr[i + 1]; p++) {
        for (int c = 0; c < C; c++) {
            double x = elem(X, dtype, n * K + (int64_t)indices[p] * C + c);
            double w = elem(data, dtype, (p * R + r) * C + c);
            acc += absolute ? fabs(x) * fabs(w) : x * w;
        }
    }
    return acc;
}

static void bsr_apply(int dtype, int64_t M, int64_t K, int R, int C, const int32_t *indptr,
                      const int32_t *indices, const void *data, const void *X, const float *bias,
                      const int64_t *rows, int64_t n_rows, double *Y, int absolute) {
    int64_t MB = M / R;
    for (int64_t t = 0; t < n_rows; t++) {
        int64_t n = rows ? rows[t] : t;
        for (int64_t i = 0; i < MB; i++) {
            for (int r = 0; r < R; r++) {
                int64_t m = i * R + r;
                double acc = row_dot(dtype, K, R, C, indptr, indices, data, X, n, i, r, absolute);
                double b = bias ? (double)bias[m] : 0.0;
                Y[t * M + m] = acc + (absolute ? fabs(b) : b);
            }
        }
    }
}

void ref_bsr_spmm(int dtype, int64_t M, int64_t K, int R, int C, const int32_t *indptr,
                  const int32_t *indices, const void *data, const void *X, const float *bias,
                  const int64_t *rows, int64_t n_rows, double *Y) {
    bsr_apply(dtype, M, K, R, C, indptr, indices, data, X, bias, rows, n_rows, Y, 0);
}

void ref_bsr_err_bound(int dtype, int64_t M, int64_t K, int R, int C, const int32_t *indptr,
                       const int32_t *indices, const void *data, const void *X,
                       const float *bias, const int64_t *rows, int64_t n_rows, double *E) {
    bsr_apply(dtype, M, K, R, C, indptr, indices, data, X, bias, rows, n_rows, E, 1);
}

void ref_dense_linear(int dtype, int64_t M, int64_t K, const void *W, const void *X,
                      const float *bias, const int64_t *rows, int64_t n_rows, double *Y) {
    for (int64_t t = 0; t < n_rows; t++) {
        int64_t n = rows ? rows[t] : t;
        for (int64_t m = 0; m < M; m++) {
            double acc = 0.0;
            for (int64_t k = 0; k < K; k++) acc += elem(X, dtype, n * K + k) * elem(W, dtype, m * K + k);
            Y[t * M + m] = acc + (bias ? (double)bias[m] : 0.0);
        }
    }
}

void ref_round_f32(const double *in, float *out, int64_t n) {
    for (int64_t i = 0; i < n; i++) out[i] = (float)in[i];
}

/* bfloat16 keeps 8 significant bits and float's exponent range: normal
 * values are multiples of 2^(e-8) for |x| in [2^(e-1), 2^e), subnormals
 * multiples of 2^-133. Rounding = nearest multiple, ties to even (the
 * default mode of nearbyint). */
static uint16_t round_bf16(double x) {
    if (isnan(x)) return (uint16_t)(signbit(x) ? 0xFFC0u : 0x7FC0u);
    double q;
    if (fabs(x) >= ldexp(1.0, -126)) {
        int e;
        frexp(x, &e);
        q = ldexp(1.0, e - 8);
    } else {
        q = ldexp(1.0, -133);
    }
    double v = isinf(x) ? x : nearbyint(x / q) * q;
    if (fabs(v) >= ldexp(1.0, 128)) v = copysign(INFINITY, x);
    float f = (float)v; /* exact: v has at most 8 significant bits */
    if (v == 0.0) f = signbit(x) ? -0.0f : 0.0f;
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(u >> 16);
}

void ref_round_bf16(const double *in, uint16_t *out, int64_t n) {
    for (int64_t i = 0; i < n; i++) out[i] = round_bf16(in[i]);
}

/* The same product with a float accumulator (the timed CPU baseline): per
 * output the kept blocks of row i in storage order and the columns of each
 * block in order, each product rounded to float and added to a float sum,
 * then + bias in float. Block rows are independent, so they are shared out
 * among `threads` OpenMP threads; every output is still summed by one
 * thread in the same order, so the result does not depend on the count. */
void ref_bsr_spmm_f32acc(int dtype, int64_t M, int64_t K, int R, int C, const int32_t *indptr,
                         const int32_t *indices, const void *data, const void *X, const float *bias,
                         const int64_t *rows, int64_t n_rows, float *Y, int threads) {
    int64_t MB = M / R;
    (void)threads;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(threads > 0 ? threads : 1)
#endif
    for (int64_t i = 0; i < MB; i++) {
        for (int64_t t = 0; t < n_rows; t++) {
            int64_t n = rows ? rows[t] : t;
            for (int r = 0; r < R; r++) {
                float acc = 0.0f;
                for (int64_t p = indptr[i]; p < indptr[i + 1]; p++)
                    for (int c = 0; c < C; c++) {
                        float x = elem_f(X, dtype, n * K + (int64_t)indices[p] * C + c);
                        float w = elem_f(data, dtype, (p * R + r) * C + c);
                        float prod = x * w;
                        acc = acc + prod;
                    }
                int64_t m = i * R + r;
                Y[t * M + m] = acc + (bias ? bias[m] : 0.0f);
            }
        }
    }
}

int ref_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
