/*
 * The C ABI used from plain C (no Python): for a few block shapes and both
 * element types, build the BSR arrays on the GPU (bsr_from_dense), create a
 * handle, run bsr_spmm with device buffers and with host buffers, run the same
 * product through a plan (bsr_plan_*), and check
 *   - indptr, indices and data bit for bit against the CPU oracle's
 *     conversion (Section 2.2's data/indices/indptr),
 *   - every output element against the oracle's fp64 product within
 *     1e-5 (fp32) or 1e-2 (bf16) of sum_k |x||w| + |b|.
 * Inputs come from a splitmix64 counter (Steele, Lea and Flood, OOPSLA 2014);
 * the generator holds none of the product's arithmetic.
 * Exit status 0 when every case passes.
 */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "bsr.h"
#include "ref_bsr.h"

static uint64_t splitmix64(uint64_t *state) {
    uint64_t z = (*state += 0x9E3779B97F4A7C15ull);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* uniform in [0, 1) from the top 24 bits */
static float unit(uint64_t *s) { return (float)(splitmix64(s) >> 40) * (1.0f / 16777216.0f); }

static uint16_t bf16_bits(float f) { /* truncation: any bit pattern is a valid input */
    uint32_t u;
    memcpy(&u, &f, 4);
    return (uint16_t)(u >> 16);
}

static int failures = 0;
#define CHECK(cond, ...)                  \
    do {                                  \
        if (!(cond)) {                    \
            printf("FAIL: " __VA_ARGS__); \
            printf("\n");                 \
            failures++;                   \
            goto done;                    \
        }                                 \
    } while (0)

static double to_double(const void *Y, int dt, int64_t i) {
    if (dt == BSR_F32) return ((const float *)Y)[i];
    uint32_t u = (uint32_t)((const uint16_t *)Y)[i] << 16;
    float f;
    memcpy(&f, &u, 4);
    return f;
}

static void run_case(int R, int C, int dt, int64_t M, int64_t K, int64_t N, double density, uint64_t seed) {
    const size_t es = dt == BSR_F32 ? 4 : 2;
    const int64_t MB = M / R, KB = K / C;
    const double tol = dt == BSR_F32 ? 1e-5 : 1e-2;
    uint64_t s = seed;
    void *W = calloc((size_t)(M * K), es), *X = malloc((size_t)(N * K) * es);
    float *bias = malloc((size_t)M * 4);
    void *Y = malloc((size_t)(N * M) * es), *Yh = malloc((size_t)(N * M) * es), *Yp = malloc((size_t)(N * M) * es);
    int32_t *ptr_ref = malloc((size_t)(MB + 1) * 4), *ptr_gpu = malloc((size_t)(MB + 1) * 4);
    int32_t *ind_ref = NULL, *ind_gpu = NULL;
    void *dat_ref = NULL, *dat_gpu = NULL;
    double *Yref = malloc((size_t)(N * M) * 8), *E = malloc((size_t)(N * M) * 8);
    void *dW = NULL, *dX = NULL, *dY = NULL, *dYp = NULL, *dInd = NULL, *dDat = NULL;
    float *dB = NULL;
    int32_t *dPtr = NULL;
    bsr_handle_t h = NULL;
    bsr_plan_t plan = NULL;
    int64_t nnzb = -1, nnzb_ref;

    /* weight: each block kept with probability `density`, values in +-[0.01, 0.03) */
    for (int64_t i = 0; i < MB; i++)
        for (int64_t j = 0; j < KB; j++) {
            if (unit(&s) >= density) continue;
            for (int r = 0; r < R; r++)
                for (int c = 0; c < C; c++) {
                    const float v = (0.01f + 0.02f * unit(&s)) * (unit(&s) < 0.5f ? -1.0f : 1.0f);
                    const int64_t e = (i * R + r) * K + j * C + c;
                    if (dt == BSR_F32) ((float *)W)[e] = v;
                    else ((uint16_t *)W)[e] = bf16_bits(v);
                }
        }
    for (int64_t e = 0; e < N * K; e++) {
        const float v = 2.0f * unit(&s) - 1.0f;
        if (dt == BSR_F32) ((float *)X)[e] = v;
        else ((uint16_t *)X)[e] = bf16_bits(v);
    }
    for (int64_t m = 0; m < M; m++) bias[m] = 0.02f * (2.0f * unit(&s) - 1.0f);

    /* the oracle's conversion */
    nnzb_ref = ref_bsr_count(W, dt, M, K, R, C, 0.0f, ptr_ref);
    CHECK(nnzb_ref >= 0, "oracle count");
    ind_ref = malloc((size_t)(nnzb_ref + 1) * 4);
    dat_ref = malloc((size_t)(nnzb_ref * R * C + 1) * es);
    ref_bsr_fill(W, dt, M, K, R, C, 0.0f, ptr_ref, ind_ref, dat_ref);

    /* the GPU's conversion: query, then fill */
    CHECK(cudaMalloc(&dW, (size_t)(M * K) * es) == cudaSuccess && cudaMalloc(&dX, (size_t)(N * K) * es) == cudaSuccess &&
              cudaMalloc(&dY, (size_t)(N * M) * es) == cudaSuccess && cudaMalloc(&dYp, (size_t)(N * M) * es) == cudaSuccess &&
              cudaMalloc((void **)&dB, (size_t)M * 4) == cudaSuccess &&
              cudaMalloc((void **)&dPtr, (size_t)(MB + 1) * 4) == cudaSuccess,
          "cudaMalloc");
    cudaMemcpy(dW, W, (size_t)(M * K) * es, cudaMemcpyHostToDevice);
    cudaMemcpy(dX, X, (size_t)(N * K) * es, cudaMemcpyHostToDevice);
    cudaMemcpy(dB, bias, (size_t)M * 4, cudaMemcpyHostToDevice);
    CHECK(bsr_from_dense(dW, M, K, R, C, 0.0f, (bsr_dtype_t)dt, dPtr, NULL, NULL, 0, &nnzb, NULL) == BSR_OK,
          "bsr_from_dense query");
    CHECK(nnzb == nnzb_ref, "nnzb %lld vs oracle %lld", (long long)nnzb, (long long)nnzb_ref);
    CHECK(cudaMalloc((void **)&dInd, (size_t)(nnzb + 1) * 4) == cudaSuccess &&
              cudaMalloc(&dDat, (size_t)(nnzb * R * C + 1) * es) == cudaSuccess,
          "cudaMalloc arrays");
    CHECK(bsr_from_dense(dW, M, K, R, C, 0.0f, (bsr_dtype_t)dt, dPtr, dInd, dDat, nnzb, &nnzb, NULL) == BSR_OK,
          "bsr_from_dense fill");
    ind_gpu = malloc((size_t)(nnzb + 1) * 4);
    dat_gpu = malloc((size_t)(nnzb * R * C + 1) * es);
    cudaMemcpy(ptr_gpu, dPtr, (size_t)(MB + 1) * 4, cudaMemcpyDeviceToHost);
    cudaMemcpy(ind_gpu, dInd, (size_t)nnzb * 4, cudaMemcpyDeviceToHost);
    cudaMemcpy(dat_gpu, dDat, (size_t)(nnzb * R * C) * es, cudaMemcpyDeviceToHost);
    CHECK(memcmp(ptr_gpu, ptr_ref, (size_t)(MB + 1) * 4) == 0, "indptr differs");
    CHECK(memcmp(ind_gpu, ind_ref, (size_t)nnzb * 4) == 0, "indices differ");
    CHECK(memcmp(dat_gpu, dat_ref, (size_t)(nnzb * R * C) * es) == 0, "data differs");

    /* the product: device buffers, host buffers, and a one-product plan */
    CHECK(bsr_create(dPtr, dInd, dDat, R, C, M, K, (bsr_dtype_t)dt, &h) == BSR_OK, "bsr_create");
    CHECK(bsr_spmm(h, dX, dB, dY, N, NULL) == BSR_OK, "bsr_spmm (device buffers)");
    CHECK(bsr_spmm(h, X, dB, Yh, N, NULL) == BSR_OK, "bsr_spmm (host buffers)");
    {
        const void *xs[1] = {dX};
        const float *bs[1] = {dB};
        void *ys[1] = {dYp};
        const int64_t ns[1] = {N};
        CHECK(bsr_plan_create(&h, xs, bs, ys, ns, 1, 0, &plan) == BSR_OK, "bsr_plan_create");
        CHECK(bsr_plan_launch(plan, NULL) == BSR_OK, "bsr_plan_launch");
    }
    CHECK(cudaDeviceSynchronize() == cudaSuccess, "synchronise");
    CHECK(bsr_check_device_status(h) == BSR_OK, "device status");
    cudaMemcpy(Y, dY, (size_t)(N * M) * es, cudaMemcpyDeviceToHost);
    cudaMemcpy(Yp, dYp, (size_t)(N * M) * es, cudaMemcpyDeviceToHost);
    CHECK(memcmp(Y, Yh, (size_t)(N * M) * es) == 0, "host-buffer result differs from device-buffer result");
    CHECK(memcmp(Y, Yp, (size_t)(N * M) * es) == 0, "plan result differs from bsr_spmm");

    ref_bsr_spmm(dt, M, K, R, C, ptr_ref, ind_ref, dat_ref, X, bias, NULL, N, Yref);
    ref_bsr_err_bound(dt, M, K, R, C, ptr_ref, ind_ref, dat_ref, X, bias, NULL, N, E);
    for (int64_t e = 0; e < N * M; e++) {
        const double d = fabs(to_double(Y, dt, e) - Yref[e]);
        CHECK(d <= tol * E[e] + 1e-30, "%dx%d %s: Y[%lld, %lld] = %.9g, oracle %.9g, bound %.3g", R, C,
              dt == BSR_F32 ? "f32" : "bf16", (long long)(e / M), (long long)(e % M), to_double(Y, dt, e),
              Yref[e], tol * E[e]);
    }
    printf("ok %dx%d %s M=%lld K=%lld N=%lld nnzb=%lld\n", R, C, dt == BSR_F32 ? "f32" : "bf16", (long long)M,
           (long long)K, (long long)N, (long long)nnzb);
done:
    bsr_plan_destroy(plan);
    bsr_destroy(h);
    cudaFree(dW); cudaFree(dX); cudaFree(dY); cudaFree(dYp); cudaFree(dB); cudaFree(dPtr); cudaFree(dInd);
    cudaFree(dDat);
    free(W); free(X); free(bias); free(Y); free(Yh); free(Yp); free(ptr_ref); free(ptr_gpu); free(ind_ref);
    free(ind_gpu); free(dat_ref); free(dat_gpu); free(Yref); free(E);
}

int main(void) {
    run_case(32, 1, BSR_F32, 256, 384, 200, 0.2, 1);    /* SIMT kernel, multi-row */
    run_case(1, 1, BSR_F32, 128, 256, 77, 0.3, 2);      /* SIMT kernel, one-row */
    run_case(32, 32, BSR_F32, 256, 256, 130, 0.3, 3);   /* tensor cores, 3xTF32 */
    run_case(16, 16, BSR_BF16, 256, 256, 130, 0.3, 4);  /* tensor cores, bf16 */
    run_case(1, 1, BSR_BF16, 256, 256, 100, 0.3, 5);    /* bf16 re-blocked into 16 x 64 tiles */
    run_case(3, 2, BSR_F32, 255, 256, 50, 0.2, 6);      /* generic kernel */
    printf(failures ? "FAILED (%d)\n" : "all cases passed\n", failures);
    return failures ? 1 : 0;
}
