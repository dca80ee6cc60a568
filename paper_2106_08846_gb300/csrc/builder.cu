// GPU construction of the BSR arrays of a dense weight (Section 2.2: "data
// values, indices, and indptr", SciPy convention).
//
//   k_mark     one thread per R x C block: keep iff some |w| > thr (fp32
//              compare written !(|w| <= thr), so NaN keeps a block), and count
//              kept blocks per block row;
//   k_scan     one CTA: exclusive scan of the row counts -> indptr;
//   k_compact  one CTA per block row: ordered compaction of the kept block
//              columns (ascending) and a bit copy of their values.
#include <cuda_bf16.h>

#include "bsr_internal.h"

namespace bsr {

namespace {

__device__ __forceinline__ float widen(float v) { return v; }
__device__ __forceinline__ float widen(uint16_t v) { return __uint_as_float((uint32_t)v << 16); }

template <typename T>
__global__ void k_mark(const T *__restrict__ W, int64_t K, int R, int C, int64_t MB, int64_t KB,
                       float thr, uint8_t *__restrict__ flags, int32_t *__restrict__ counts) {
    const int64_t total = MB * KB;
    for (int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; b < total;
         b += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = b / KB, j = b - i * KB;
        const T *base = W + i * R * K + j * C;
        bool keep = false;
        for (int r = 0; r < R && !keep; r++)
            for (int c = 0; c < C; c++)
                if (!(fabsf(widen(base[(int64_t)r * K + c])) <= thr)) { keep = true; break; }
        flags[b] = keep ? 1 : 0;
        if (keep) atomicAdd(&counts[i], 1);
    }
}

// Inclusive scan inside a warp.
__device__ __forceinline__ int64_t warp_scan(int64_t x, int lane) {
    for (int o = 1; o < 32; o <<= 1) {
        int64_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    return x;
}

// Exclusive block-wide scan of v over blockDim.x (a multiple of 32, <= 1024)
// threads; returns the exclusive prefix and writes the block total.
__device__ int64_t block_exclusive_scan(int64_t v, int64_t *total, int64_t *warp_tot) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int64_t x = warp_scan(v, lane);
    if (lane == 31) warp_tot[wid] = x;
    __syncthreads();
    if (wid == 0) {
        int64_t t = lane < nw ? warp_tot[lane] : 0;
        t = warp_scan(t, lane);
        if (lane < nw) warp_tot[lane] = t;
    }
    __syncthreads();
    int64_t excl = x - v + (wid ? warp_tot[wid - 1] : 0);
    *total = warp_tot[nw - 1];
    __syncthreads();
    return excl;
}

__global__ void k_scan(const int32_t *__restrict__ counts, int64_t MB, int32_t *__restrict__ indptr) {
    __shared__ int64_t warp_tot[32];
    int64_t carry = 0;
    if (threadIdx.x == 0) indptr[0] = 0;
    for (int64_t base = 0; base < MB; base += blockDim.x) {
        const int64_t idx = base + threadIdx.x;
        const int64_t v = idx < MB ? counts[idx] : 0;
        int64_t total;
        const int64_t excl = block_exclusive_scan(v, &total, warp_tot);
        const int64_t incl = carry + excl + v;
        // An nnzb beyond int32 is reported as -1 and rejected by the host.
        if (idx < MB) indptr[idx + 1] = incl > INT32_MAX ? -1 : (int32_t)incl;
        carry += total;
    }
}

constexpr int kCompactThreads = 256;

template <typename B>  // B: uint32_t (fp32 bits) or uint16_t (bf16 bits)
__global__ void __launch_bounds__(kCompactThreads)
k_compact(const B *__restrict__ W, int64_t K, int R, int C, int64_t MB, int64_t KB,
          const uint8_t *__restrict__ flags, const int32_t *__restrict__ indptr,
          int32_t *__restrict__ indices, B *__restrict__ data) {
    __shared__ int64_t warp_tot[32];
    __shared__ int32_t cols[kCompactThreads];
    const int64_t RC = (int64_t)R * C;
    for (int64_t i = blockIdx.x; i < MB; i += gridDim.x) {
        int64_t p = indptr[i];
        for (int64_t j0 = 0; j0 < KB; j0 += kCompactThreads) {
            const int64_t j = j0 + threadIdx.x;
            const int f = j < KB ? flags[i * KB + j] : 0;
            int64_t n;
            const int64_t pos = block_exclusive_scan(f, &n, warp_tot);
            if (f) {
                indices[p + pos] = (int32_t)j;
                cols[pos] = (int32_t)j;
            }
            __syncthreads();
            for (int64_t e = threadIdx.x; e < n * RC; e += kCompactThreads) {
                const int64_t q = e / RC, rc = e - q * RC;
                const int r = (int)(rc / C), c = (int)(rc - (int64_t)r * C);
                data[(p + q) * RC + rc] = W[(i * R + r) * K + (int64_t)cols[q] * C + c];
            }
            p += n;
            __syncthreads();
        }
    }
}

int grid_for(int64_t work, int threads) {
    int64_t g = (work + threads - 1) / threads;
    return (int)std::max<int64_t>(1, std::min<int64_t>(g, 1 << 20));
}

}  // namespace

cudaError_t launch_builder_count(const void *W, bsr_dtype_t dt, int64_t M, int64_t K, int R, int C,
                                 float thr, uint8_t *flags, int32_t *counts, int32_t *indptr,
                                 cudaStream_t s) {
    const int64_t MB = M / R, KB = K / C;
    cudaError_t e = cudaMemsetAsync(counts, 0, (size_t)std::max<int64_t>(MB, 1) * 4, s);
    if (e != cudaSuccess) return e;
    if (MB * KB > 0) {
        const int g = grid_for(MB * KB, 256);
        if (dt == BSR_F32)
            k_mark<float><<<g, 256, 0, s>>>((const float *)W, K, R, C, MB, KB, thr, flags, counts);
        else
            k_mark<uint16_t><<<g, 256, 0, s>>>((const uint16_t *)W, K, R, C, MB, KB, thr, flags, counts);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    k_scan<<<1, 1024, 0, s>>>(counts, MB, indptr);
    return cudaGetLastError();
}

cudaError_t launch_builder_compact(const void *W, bsr_dtype_t dt, int64_t M, int64_t K, int R, int C,
                                   const uint8_t *flags, const int32_t *indptr, int32_t *indices,
                                   void *data, cudaStream_t s) {
    const int64_t MB = M / R, KB = K / C;
    if (MB == 0) return cudaSuccess;
    const int g = (int)std::min<int64_t>(MB, 1 << 20);
    if (dt == BSR_F32)
        k_compact<uint32_t><<<g, kCompactThreads, 0, s>>>((const uint32_t *)W, K, R, C, MB, KB, flags,
                                                          indptr, indices, (uint32_t *)data);
    else
        k_compact<uint16_t><<<g, kCompactThreads, 0, s>>>((const uint16_t *)W, K, R, C, MB, KB, flags,
                                                          indptr, indices, (uint16_t *)data);
    return cudaGetLastError();
}

}  // namespace bsr
