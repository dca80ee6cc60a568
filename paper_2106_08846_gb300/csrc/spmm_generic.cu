// Generic BSR x dense kernel: any R x C block, fp32 or bf16. One thread per
// output element of a (token tile, work item) pair, X and the block values
// read through the cache hierarchy. It is the fallback for block shapes
// without a specialised kernel, and the split-row reduce used by all kernels.
#include <cuda_bf16.h>

#include "bsr_internal.h"
#include "elem.cuh"
#include "launch.cuh"
#include "ptx.cuh"

namespace bsr {

namespace {

template <typename T>
__global__ void __launch_bounds__(256)
k_generic(const Item *__restrict__ items, int n_items, const int32_t *__restrict__ indices,
          const T *__restrict__ data, const T *__restrict__ X, const float *__restrict__ bias,
          T *__restrict__ Y, float *__restrict__ ws, int64_t N, int64_t K, int64_t M, int R, int C,
          int tn, int64_t n_tiles) {
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();   // X, the bias, Y and the workspace may be an earlier kernel's
    const int64_t work = (int64_t)n_items * n_tiles;
    for (int64_t b = blockIdx.x; b < work; b += gridDim.x) {
        const int64_t tile = b / n_items;
        const Item it = items[b - tile * n_items];
        const int64_t n0 = tile * tn;
        const int outs = tn * R;
        for (int o = threadIdx.x; o < outs; o += blockDim.x) {
            const int t = o / R, r = o - t * R;
            const int64_t n = n0 + t;
            if (n >= N) continue;
            const T *xrow = X + n * K;
            float acc = 0.f;
            for (int p = it.p0; p < it.p1; p++) {
                const T *xb = xrow + (int64_t)indices[p] * C;
                const T *wb = data + ((int64_t)p * R + r) * C;
                for (int c = 0; c < C; c++) acc = fmaf(to_f32(xb[c]), to_f32(wb[c]), acc);
            }
            const int64_t m = (int64_t)it.row * R + r;
            if (it.slot < 0)
                Y[n * M + m] = from_f32<T>(acc + (bias ? bias[m] : 0.f));
            else
                ws[((int64_t)it.slot * N + n) * R + r] = acc;
        }
    }
}

// Y[n, row*R + r] = sum over the row's pieces, in piece order, + bias.
template <typename T>
__global__ void k_reduce(const Split *__restrict__ splits, int n_splits, const float *__restrict__ ws,
                         const float *__restrict__ bias, T *__restrict__ Y, int64_t N, int64_t M, int R) {
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();   // the partials come from the product kernel just before
    const int64_t total = (int64_t)n_splits * N * R;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t rest = e / R;
        const int r = (int)(e - rest * R);
        const int64_t s = rest / N, n = rest - s * N;
        const Split sp = splits[s];
        float acc = 0.f;
        for (int k = 0; k < sp.nslot; k++) acc += ws[((int64_t)(sp.slot0 + k) * N + n) * R + r];
        const int64_t m = (int64_t)sp.row * R + r;
        Y[n * M + m] = from_f32<T>(acc + (bias ? bias[m] : 0.f));
    }
}

}  // namespace

cudaError_t launch_generic(const LaunchArgs &a) {
    const Schedule &sc = *a.sc;
    const int n_items = (int)sc.items.size();
    if (n_items == 0) return cudaSuccess;
    const int tn = sc.tn;
    const int64_t n_tiles = (a.N + tn - 1) / tn;
    const int64_t work = (int64_t)n_items * n_tiles;
    const int grid = (int)std::min<int64_t>(work, 1 << 24);
    if (sc.dt == BSR_F32)
        return launch_kernel(k_generic<float>, dim3(grid), dim3(256), 0, a.stream, 1u, (const Item *)sc.d_items,
                             n_items, (const int32_t *)sc.d_indices, (const float *)a.data, (const float *)a.X,
                             a.bias, (float *)a.Y, a.ws, a.N, sc.K, sc.M, sc.R, sc.C, tn, n_tiles);
    return launch_kernel(k_generic<uint16_t>, dim3(grid), dim3(256), 0, a.stream, 1u, (const Item *)sc.d_items,
                         n_items, (const int32_t *)sc.d_indices, (const uint16_t *)a.data, (const uint16_t *)a.X,
                         a.bias, (uint16_t *)a.Y, a.ws, a.N, sc.K, sc.M, sc.R, sc.C, tn, n_tiles);
}

cudaError_t launch_reduce(const LaunchArgs &a) {
    const Schedule &sc = *a.sc;
    const int n_splits = (int)sc.splits.size();
    if (n_splits == 0) return cudaSuccess;
    const int R = sc.ex_R;   // rows per split row (tile rows of re-blocked weights)
    const int64_t total = (int64_t)n_splits * a.N * R;
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((total + 255) / 256, 1 << 20));
    if (sc.dt == BSR_F32)
        return launch_kernel(k_reduce<float>, dim3(grid), dim3(256), 0, a.stream, 1u, (const Split *)sc.d_splits,
                             n_splits, (const float *)a.ws, a.bias, (float *)a.Y, a.N, sc.M, R);
    return launch_kernel(k_reduce<uint16_t>, dim3(grid), dim3(256), 0, a.stream, 1u, (const Split *)sc.d_splits,
                         n_splits, (const float *)a.ws, a.bias, (uint16_t *)a.Y, a.N, sc.M, R);
}

}  // namespace bsr
