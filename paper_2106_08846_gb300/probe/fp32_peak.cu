// Measured FP32 FMA peak of the GPU: the denominator of every roofline of the
// SIMT kernels (fp32 multiply-adds on the CUDA cores). Each thread runs
// kChains independent multiply-add chains, either as scalar fma.rn.f32 or as
// packed fma.rn.f32x2 (two fp32 multiply-adds per instruction), so the FMA
// pipe, not latency, sets the rate. Values stay bounded (a * b + c with b
// near 1 and c tiny), and every chain's result is written out so nothing is
// optimised away. Built into its own library (libbsr_probe.so): it is
// measurement infrastructure of the benchmark, not part of the product's C
// ABI (include/bsr.h).
#include <cuda_runtime.h>

#include <cstdint>

namespace {

constexpr int kChains = 8;

typedef unsigned long long f2_t;

__device__ __forceinline__ f2_t ffma2(f2_t a, f2_t b, f2_t c) {
    f2_t d;
    asm volatile("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}

__device__ __forceinline__ float ffma1(float a, float b, float c) {
    float d;
    asm volatile("fma.rn.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

__device__ __forceinline__ f2_t pack2(float lo, float hi) {
    f2_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}

__device__ __forceinline__ float sum2(f2_t v) {
    float lo, hi;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
    return lo + hi;
}

// kChains packed chains: 2 * kChains multiply-adds per iteration per thread.
__global__ void k_fma2(float *out, int64_t iters) {
    const float s = 1.0f + 1e-7f * (float)(threadIdx.x & 7);
    f2_t a[kChains];
#pragma unroll
    for (int k = 0; k < kChains; k++) a[k] = pack2(s + (float)k * 1e-3f, s - (float)k * 1e-3f);
    const f2_t b = pack2(0.9999999f, 1.0000001f), c = pack2(1e-8f, -1e-8f);
    for (int64_t i = 0; i < iters; i++) {
#pragma unroll
        for (int k = 0; k < kChains; k++) a[k] = ffma2(a[k], b, c);
    }
    float t = 0.f;
#pragma unroll
    for (int k = 0; k < kChains; k++) t += sum2(a[k]);
    out[(int64_t)blockIdx.x * blockDim.x + threadIdx.x] = t;
}

// 2 * kChains scalar chains: the same multiply-adds per iteration as k_fma2.
__global__ void k_fma1(float *out, int64_t iters) {
    const float s = 1.0f + 1e-7f * (float)(threadIdx.x & 7);
    float a[2 * kChains];
#pragma unroll
    for (int k = 0; k < 2 * kChains; k++) a[k] = s + (float)k * 1e-3f;
    for (int64_t i = 0; i < iters; i++) {
#pragma unroll
        for (int k = 0; k < 2 * kChains; k++) a[k] = ffma1(a[k], 0.9999999f, 1e-8f);
    }
    float t = 0.f;
#pragma unroll
    for (int k = 0; k < 2 * kChains; k++) t += a[k];
    out[(int64_t)blockIdx.x * blockDim.x + threadIdx.x] = t;
}

}  // namespace

extern "C" {

// Multiply-adds one launch of bsr_probe_fma performs (2 flops each).
int64_t bsr_probe_fma_count(int blocks, int threads, int64_t iters) {
    return (int64_t)blocks * threads * iters * 2 * kChains;
}

// Launches the probe on `stream` (cudaStream_t): packed = 1 runs fma.rn.f32x2,
// 0 scalar fma.rn.f32. out: device, blocks * threads floats. Returns the
// cudaError_t of the launch (0 on success). Asynchronous.
int bsr_probe_fma(float *out, int blocks, int threads, int64_t iters, int packed, void *stream) {
    if (!out || blocks <= 0 || threads <= 0 || threads > 1024 || iters < 0) return (int)cudaErrorInvalidValue;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (packed)
        k_fma2<<<blocks, threads, 0, s>>>(out, iters);
    else
        k_fma1<<<blocks, threads, 0, s>>>(out, iters);
    return (int)cudaGetLastError();
}

}  // extern "C"
