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

// Y[n, row*R + r] = sum over the row's pieces, in piece order, + bias. One
// CTA per (split row, tile of `tn` tokens): the tile's tn x R outputs are
// R-contiguous runs of Y, so consecutive threads write consecutive
// addresses; index arithmetic is one 64-bit division per tile and 32-bit
// inside it.
template <typename T>
__global__ void __launch_bounds__(256)
k_reduce(const Split *__restrict__ splits, int n_splits, const float *__restrict__ ws,
         const float *__restrict__ bias, T *__restrict__ Y, int64_t N, int64_t M, int R, int tn, int64_t n_tiles) {
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();   // the partials come from the product kernel just before
    const int64_t work = (int64_t)n_splits * n_tiles;
    for (int64_t b = blockIdx.x; b < work; b += gridDim.x) {
        const int64_t s = b / n_tiles;
        const int64_t n0 = (b - s * n_tiles) * tn;
        const Split sp = splits[s];
        const unsigned outs = (unsigned)(N - n0 < tn ? N - n0 : tn) * (unsigned)R;
        const int64_t m0 = (int64_t)sp.row * R;
        for (unsigned o = threadIdx.x; o < outs; o += blockDim.x) {
            const unsigned t = o / (unsigned)R, r = o - t * (unsigned)R;
            const int64_t n = n0 + t;
            float acc = 0.f;
            for (int k = 0; k < sp.nslot; k++) acc += ws[((int64_t)(sp.slot0 + k) * N + n) * R + r];
            Y[n * M + m0 + r] = from_f32<T>(acc + (bias ? bias[m0 + r] : 0.f));
        }
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
        return launch_kernel(k_generic<float>, dim3(grid), dim3(256), 0, a.stream, (const Item *)sc.d_items,
                             n_items, (const int32_t *)sc.d_indices, (const float *)a.data, (const float *)a.X,
                             a.bias, (float *)a.Y, a.ws, a.N, sc.K, sc.M, sc.R, sc.C, tn, n_tiles);
    return launch_kernel(k_generic<uint16_t>, dim3(grid), dim3(256), 0, a.stream, (const Item *)sc.d_items,
                         n_items, (const int32_t *)sc.d_indices, (const uint16_t *)a.data, (const uint16_t *)a.X,
                         a.bias, (uint16_t *)a.Y, a.ws, a.N, sc.K, sc.M, sc.R, sc.C, tn, n_tiles);
}

cudaError_t launch_reduce(const LaunchArgs &a) {
    const Schedule &sc = *a.sc;
    const int n_splits = (int)sc.splits.size();
    if (n_splits == 0 || a.N == 0) return cudaSuccess;
    const int R = sc.ex_R;   // rows per split row (tile rows of re-blocked weights)
    const int tn = std::max(1, 1024 / R);   // about 1024 outputs per tile
    const int64_t n_tiles = (a.N + tn - 1) / tn;
    const int grid = (int)std::min<int64_t>((int64_t)n_splits * n_tiles, 1 << 20);
    if (sc.dt == BSR_F32)
        return launch_kernel(k_reduce<float>, dim3(grid), dim3(256), 0, a.stream, (const Split *)sc.d_splits,
                             n_splits, (const float *)a.ws, a.bias, (float *)a.Y, a.N, sc.M, R, tn, n_tiles);
    return launch_kernel(k_reduce<uint16_t>, dim3(grid), dim3(256), 0, a.stream, (const Split *)sc.d_splits,
                         n_splits, (const float *)a.ws, a.bias, (uint16_t *)a.Y, a.N, sc.M, R, tn, n_tiles);
}

}  // namespace bsr
