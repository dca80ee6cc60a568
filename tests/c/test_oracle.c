/*
 * Self-checks of the CPU oracle in C (no GPU), against facts that do not
 * depend on the oracle itself:
 *   - with small dyadic values every product and partial sum is exact in
 *     double, so the BSR loop over kept blocks (Section 2.2) must equal the
 *     dense linear layer on the same W bit for bit, in any order;
 *   - keeping every block (0% sparsity) gives MB*KB blocks and the dense
 *     product; an all-zero weight (100% sparsity) gives no block and Y = bias;
 *   - dense -> BSR -> dense returns the weight bit for bit when the removed
 *     blocks are zero;
 *   - the keep rule !(|w| <= threshold): a NaN keeps its block, -0.0 does not.
 * Exit status 0 when every check passes.
 */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "ref_bsr.h"

static int failures = 0;
#define EXPECT(cond, ...)                 \
    do {                                  \
        if (!(cond)) {                    \
            printf("FAIL: " __VA_ARGS__); \
            printf("\n");                 \
            failures++;                   \
        }                                 \
    } while (0)

static uint64_t lcg = 12345;
static int small_int(int lo, int hi) { /* deterministic, uniform enough for a fixture */
    lcg = lcg * 6364136223846793005ull + 1442695040888963407ull;
    return lo + (int)((lcg >> 33) % (uint64_t)(hi - lo + 1));
}

/* W[M, K] fp32 with dyadic values k/8 (|k| <= 7), block (i, j) zeroed when
 * drop(i, j); X[N, K] with values k/4. */
static void fixture(int64_t M, int64_t K, int R, int C, int64_t N, int keep_percent, float *W, float *X, float *b) {
    for (int64_t i = 0; i < M / R; i++)
        for (int64_t j = 0; j < K / C; j++) {
            const int keep = small_int(0, 99) < keep_percent;
            for (int r = 0; r < R; r++)
                for (int c = 0; c < C; c++) {
                    int v = keep ? small_int(-7, 7) : 0;
                    if (keep && r == 0 && c == 0 && v == 0) v = 1;   /* a kept block is never all zero */
                    W[(i * R + r) * K + j * C + c] = (float)v / 8.0f;
                }
        }
    for (int64_t e = 0; e < N * K; e++) X[e] = (float)small_int(-8, 8) / 4.0f;
    for (int64_t m = 0; m < M; m++) b[m] = (float)small_int(-4, 4) / 16.0f;
}

static void check_shape(int64_t M, int64_t K, int R, int C, int64_t N, int keep_percent) {
    const int64_t MB = M / R, KB = K / C;
    float *W = malloc((size_t)(M * K) * 4), *X = malloc((size_t)(N * K) * 4), *b = malloc((size_t)M * 4);
    float *W2 = calloc((size_t)(M * K), 4);
    int32_t *ptr = malloc((size_t)(MB + 1) * 4);
    double *Yb = malloc((size_t)(N * M) * 8), *Yd = malloc((size_t)(N * M) * 8);
    fixture(M, K, R, C, N, keep_percent, W, X, b);
    const int64_t nnzb = ref_bsr_count(W, ORACLE_F32, M, K, R, C, 0.0f, ptr);
    int32_t *ind = malloc((size_t)(nnzb + 1) * 4);
    float *data = malloc((size_t)(nnzb * R * C + 1) * 4);
    ref_bsr_fill(W, ORACLE_F32, M, K, R, C, 0.0f, ptr, ind, data);
    if (keep_percent == 100) EXPECT(nnzb == MB * KB, "%dx%d: all kept, nnzb %lld", R, C, (long long)nnzb);
    if (keep_percent == 0) EXPECT(nnzb == 0, "%dx%d: none kept, nnzb %lld", R, C, (long long)nnzb);
    ref_bsr_to_dense(ORACLE_F32, M, K, R, C, ptr, ind, data, W2);
    EXPECT(memcmp(W, W2, (size_t)(M * K) * 4) == 0, "%dx%d: dense -> BSR -> dense differs", R, C);
    ref_bsr_spmm(ORACLE_F32, M, K, R, C, ptr, ind, data, X, b, NULL, N, Yb);
    ref_dense_linear(ORACLE_F32, M, K, W, X, b, NULL, N, Yd);
    EXPECT(memcmp(Yb, Yd, (size_t)(N * M) * 8) == 0, "%dx%d keep %d%%: BSR product differs from dense", R, C,
           keep_percent);
    if (keep_percent == 0)
        for (int64_t e = 0; e < N * M; e++) EXPECT(Yb[e] == (double)b[e % M], "%dx%d: Y != bias", R, C);
    free(W); free(X); free(b); free(W2); free(ptr); free(Yb); free(Yd); free(ind); free(data);
}

static void check_keep_rule(void) {
    /* 2 x 4 weight, 2 x 2 blocks: block 0 holds a NaN, block 1 only -0.0 and +0.0 */
    float W[8] = {NAN, 0.0f, -0.0f, 0.0f, 0.0f, 0.0f, 0.0f, -0.0f};
    int32_t ptr[2];
    EXPECT(ref_bsr_count(W, ORACLE_F32, 2, 4, 2, 2, 0.0f, ptr) == 1, "NaN keeps its block, -0.0 does not");
    /* threshold: |w| <= thr drops, so a block of values at exactly thr is dropped */
    float V[4] = {0.5f, -0.5f, 0.25f, 0.0f};
    int32_t p1[2];
    EXPECT(ref_bsr_count(V, ORACLE_F32, 2, 2, 2, 2, 0.5f, p1) == 0, "values at the threshold are dropped");
    EXPECT(ref_bsr_count(V, ORACLE_F32, 2, 2, 2, 2, 0.49f, p1) == 1, "values above the threshold keep the block");
}

int main(void) {
    const int shapes[][2] = {{1, 1}, {4, 4}, {8, 1}, {32, 1}, {1, 32}, {16, 16}, {3, 2}};
    for (size_t s = 0; s < sizeof shapes / sizeof shapes[0]; s++) {
        const int R = shapes[s][0], C = shapes[s][1];
        const int64_t M = 4 * R * 3, K = 4 * C * 5;
        check_shape(M, K, R, C, 7, 20);
        check_shape(M, K, R, C, 5, 100);
        check_shape(M, K, R, C, 3, 0);
    }
    check_keep_rule();
    printf(failures ? "FAILED (%d)\n" : "all checks passed\n", failures);
    return failures ? 1 : 0;
}
