// Persistent SIMT BSR x dense kernel for tall blocks ("xrow"): blocks of 16
// or 32 rows (Section 2.2's kept blocks; the paper's best shape, 32x1, among
// them), with one column or 16 / 32 columns, at token counts large enough to
// give every SM many units of work. fp32 multiply-adds on the CUDA cores.
//
// One CTA per SM walks a contiguous range of units (task, token tile) of
// equal total work, tasks in the outer order, so a task's blob is fetched
// once for many tiles:
//
//  * warp 12, one thread: per task the blob -- item table, records (per
//    chunk the item's first block; per block its X offset inside a stage or
//    its block column) and block values (widened to fp32) -- by one bulk
//    copy once every warp is done with the previous task's; then the X
//    chunks of every unit, [32 S tokens x 256 / S columns], by 2-D TMA
//    (128-byte swizzle) through a 3-stage ring that keeps streaming across
//    units and tasks.
//  * warps 0..11: each owns one item (block row, or a piece of a split row)
//    on one 32-token subtile of every unit, so it holds complete outputs: no
//    partial tiles cross warps. Lane = tg + 8 q: tg picks tokens tg, tg+8,
//    tg+16, tg+24 (conflict-free under the swizzle); q picks one of R / 16
//    groups of 16 outputs and one of NKS = 64 / R lane groups (ks) that
//    take alternate blocks (one column) or a share of every block's
//    columns (wider). A lane accumulates 4 tokens x 16 outputs with packed
//    fma.rn.f32x2 over pairs of adjacent outputs, (x_t, x_t) * (w_r, w_r+1),
//    so the weights come straight from 16-byte shared loads in pairs.
//  * unit epilogue, per warp: the ks lane groups combine by a butterfly of
//    shuffles that halves the outputs each lane keeps, the bias is added and
//    each lane stores its contiguous outputs of 4 tokens (split rows: fp32
//    partials to the workspace for the reduce pass). The producer meanwhile
//    streams the next unit's chunks.
//
// Launched with programmatic stream serialisation: the first blob is
// fetched before the wait for the previous kernel; X, bias and Y after it.
// Every wait is bounded by the global timer; a timeout sets the device
// status word, stops the CTA's pipeline and drains its copies.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "bsr_internal.h"
#include "elem.cuh"
#include "launch.cuh"
#include "ptx.cuh"
#include "xrow.h"

namespace bsr {

namespace {

constexpr int NW = kXrWarps;
constexpr int NS = kXrStages;
constexpr int kItab = kXrItab;
constexpr uint64_t kDrainNs = 200000000ull;   // bound for copies already issued (they take microseconds)

struct XrArgs {
    const unsigned char *blob;   // task t's blob at blob + t * stride
    const int64_t *cost;         // n_tasks + 1 prefix sums of the work of one unit of each task
    uint32_t stride, hdr, ib;    // blob bytes per task, item-table bytes, record-region bytes
    int n_tasks, G;
    const float *bias;
    void *Y;
    float *ws;
    int *status;
    int64_t N, K, M;
    int C, nchunks;
    uint32_t blob_off, bar_off, misc_off;   // shared-memory offsets
    uint64_t wait_ns;
    int stall_chunk;             // test hook: this chunk of each CTA's first unit is never loaded (-1: none)
};

// Ring stage geometry for element type T and S subtiles: 32 S token rows of
// 128 bytes per box, boxes of 128 / sizeof(T) columns side by side.
template <typename T, int S>
struct Geo {
    static constexpr int TN = 32 * S;
    static constexpr int KC = 256 / S;
    static constexpr int kBoxCols = 128 / (int)sizeof(T);
    static constexpr int kBoxes = KC / kBoxCols;
    static constexpr uint32_t kBoxBytes = TN * 128;
    static constexpr uint32_t kBytes = kBoxes * kBoxBytes;
    // byte offset of chunk column kk at token row 0, before the swizzle
    __device__ static __forceinline__ uint32_t off0(int kk) {
        return (uint32_t)((kk / kBoxCols) * kBoxBytes + (kk % kBoxCols) * (int)sizeof(T));
    }
};

__device__ __forceinline__ float ld_x(const unsigned char *p, float) { return *reinterpret_cast<const float *>(p); }
__device__ __forceinline__ float ld_x(const unsigned char *p, uint16_t) {
    return to_f32(*reinterpret_cast<const uint16_t *>(p));
}
// two consecutive columns of one token
__device__ __forceinline__ float2 ld_x2(const unsigned char *p, float) { return *reinterpret_cast<const float2 *>(p); }
__device__ __forceinline__ float2 ld_x2(const unsigned char *p, uint16_t) {
    const uint32_t v = *reinterpret_cast<const uint32_t *>(p);
    return make_float2(__uint_as_float(v << 16), __uint_as_float(v & 0xffff0000u));
}

typedef unsigned long long f2_t;   // two packed fp32
__device__ __forceinline__ f2_t pack2(float lo, float hi) {
    f2_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void unpack2(f2_t v, float &lo, float &hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ f2_t ffma2(f2_t a, f2_t b, f2_t c) {
    f2_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ f2_t fadd2(f2_t a, f2_t b) {
    f2_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ f2_t shfl_xor2(f2_t v, int m) {
    float lo, hi;
    unpack2(v, lo, hi);
    return pack2(__shfl_xor_sync(0xffffffffu, lo, m), __shfl_xor_sync(0xffffffffu, hi, m));
}

__device__ __forceinline__ void set_status(int *status, int code) { atomicCAS(status, DEV_OK, code); }
__device__ __forceinline__ bool aborted(const int *flag) { return *reinterpret_cast<const volatile int *>(flag) != 0; }

// 4 tokens x 16 outputs (8 pairs of adjacent outputs) += x (4 tokens) * w (16 outputs)
struct Acc {
    f2_t a[4][8];
    __device__ __forceinline__ void zero() {
#pragma unroll
        for (int i = 0; i < 4; i++)
#pragma unroll
            for (int j = 0; j < 8; j++) a[i][j] = 0ull;
    }
    __device__ __forceinline__ void fma(const float (&x)[4], const float4 (&w)[4]) {
        f2_t wp[8];
#pragma unroll
        for (int j = 0; j < 4; j++) {
            wp[2 * j] = pack2(w[j].x, w[j].y);
            wp[2 * j + 1] = pack2(w[j].z, w[j].w);
        }
#pragma unroll
        for (int i = 0; i < 4; i++) {
            const f2_t xd = pack2(x[i], x[i]);
#pragma unroll
            for (int j = 0; j < 8; j++) a[i][j] = ffma2(xd, wp[j], a[i][j]);
        }
    }
};

// The first unit of a CTA range that starts at work W: units are (task t,
// tile i) in task-major order, unit u = t * n_tiles + i covers work
// [pre[t] n_tiles + i c_t, + c_t) with c_t = pre[t+1] - pre[t]; a unit
// belongs to the range holding its midpoint.
__device__ __forceinline__ int64_t first_unit(const int64_t *pre, int n_tasks, int64_t n_tiles, int64_t W) {
    int lo = 0, hi = n_tasks - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (__ldg(pre + mid) * n_tiles <= W) lo = mid;
        else hi = mid - 1;
    }
    const int64_t p0 = __ldg(pre + lo), ct = __ldg(pre + lo + 1) - p0;
    const int64_t num = 2 * W - 2 * p0 * n_tiles - ct;
    int64_t i = num <= 0 ? 0 : (num + 2 * ct - 1) / (2 * ct);
    if (i > n_tiles) i = n_tiles;
    return (int64_t)lo * n_tiles + i;
}

struct Shared {
    unsigned char *base;
    uint64_t *full, *empty, *wbar, *bfree;
    int *misc;     // [0] abort flag
    int *itab;     // the blob's item table
    int32_t *I;    // records
    float *W;      // block values
};

// One unit's blocks of chunk c for one lane: one-column blocks, lane group
// ks takes blocks lo+ks, lo+ks+NKS, ...
template <typename T, int R, int S>
__device__ __forceinline__ void chunk_c1(Acc &acc, const unsigned char *lane_st, const int32_t *bo, const float *wv,
                                         int lo, int hi, int ks, int rg, uint32_t tgx) {
    constexpr int NKS = 64 / R;
    for (int lb = lo + ks; lb < hi; lb += NKS) {
        const uint32_t off = (uint32_t)bo[lb] ^ tgx;
        const float4 *wp = reinterpret_cast<const float4 *>(wv + lb * (R + 4) + rg * 16);
        float4 w[4];
#pragma unroll
        for (int j = 0; j < 4; j++) w[j] = wp[j];
        float x[4];
#pragma unroll
        for (int i = 0; i < 4; i++) x[i] = ld_x(lane_st + off + i * 1024, T());
        acc.fma(x, w);
    }
}

// Wider blocks (C = 16 or 32): lane group ks takes columns [ks cw, ks cw + cw)
// of every block, two at a time (one 8-byte X load per token); a column's
// 16-byte groups of outputs are stored permuted by ks * R / 16 so the lane
// groups' weight loads fall in distinct banks.
template <typename T, int R, int S>
__device__ __forceinline__ void chunk_cw(Acc &acc, const unsigned char *lane_st, const int32_t *bo, const float *wv,
                                         int lo, int hi, int ks, int rg, uint32_t tgx, int C, int kbase) {
    using G = Geo<T, S>;
    constexpr int NKS = 64 / R;
    const int cw = C / NKS;
    const int sw = ks * (R / 16);
    for (int lb = lo; lb < hi; lb++) {
        const int kk0 = bo[lb] * C - kbase + ks * cw;
        const float *wb = wv + (int64_t)lb * C * R + ks * cw * R;
        for (int c2 = 0; c2 < cw; c2 += 2) {
            const unsigned char *xp = lane_st + (G::off0(kk0 + c2) ^ tgx);
            float2 xv[4];
#pragma unroll
            for (int i = 0; i < 4; i++) xv[i] = ld_x2(xp + i * 1024, T());
#pragma unroll
            for (int u = 0; u < 2; u++) {
                const float4 *wc = reinterpret_cast<const float4 *>(wb + (c2 + u) * R);
                float4 w[4];
#pragma unroll
                for (int j = 0; j < 4; j++) w[j] = wc[(rg * 4 + j) ^ sw];
                float x[4];
#pragma unroll
                for (int i = 0; i < 4; i++) x[i] = u == 0 ? xv[i].x : xv[i].y;
                acc.fma(x, w);
            }
        }
    }
}

// Unit epilogue of one warp: combine the NKS lane groups (each round swaps
// half of the kept outputs with the partner lane and adds), add the bias and
// store 4 tokens x 16 / NKS contiguous outputs per lane.
template <typename T, int R, int S>
__device__ __forceinline__ void epilogue(const XrArgs &a, Acc &acc, int row, int slot, int64_t nb, int tg, int rg,
                                         int ks) {
    constexpr int NKS = 64 / R;
    constexpr int NRG = R / 16;
    constexpr int V = 16 / NKS;   // outputs kept per lane: 8 (R = 32) or 4 (R = 16)
    f2_t v[4][V / 2];
    // round 1: partner differs in ks bit 0 (lane ^ 8 NRG); keep pairs [4 b0, 4 b0 + 4)
    const int b0 = ks & 1;
#pragma unroll
    for (int i = 0; i < 4; i++)
#pragma unroll
        for (int j = 0; j < 4; j++) {
            const f2_t keep = b0 ? acc.a[i][4 + j] : acc.a[i][j];
            const f2_t send = b0 ? acc.a[i][j] : acc.a[i][4 + j];
            acc.a[i][j] = fadd2(keep, shfl_xor2(send, 8 * NRG));
        }
    int obase = rg * 16 + b0 * 8;
    if constexpr (NKS == 4) {
        // round 2: partner differs in ks bit 1 (lane ^ 16); keep pairs [2 b1, 2 b1 + 2)
        const int b1 = ks >> 1;
#pragma unroll
        for (int i = 0; i < 4; i++)
#pragma unroll
            for (int j = 0; j < 2; j++) {
                const f2_t keep = b1 ? acc.a[i][2 + j] : acc.a[i][j];
                const f2_t send = b1 ? acc.a[i][j] : acc.a[i][2 + j];
                v[i][j] = fadd2(keep, shfl_xor2(send, 16));
            }
        obase += b1 * 4;
    } else {
#pragma unroll
        for (int i = 0; i < 4; i++)
#pragma unroll
            for (int j = 0; j < 4; j++) v[i][j] = acc.a[i][j];
    }
    const int64_t m = (int64_t)row * R + obase;
    float b[V];
    if (slot < 0 && a.bias) {   // (the bias is only 4-byte aligned)
#pragma unroll
        for (int j = 0; j < V; j++) b[j] = __ldg(a.bias + m + j);
    } else {
#pragma unroll
        for (int j = 0; j < V; j++) b[j] = 0.f;
    }
#pragma unroll
    for (int i = 0; i < 4; i++) {
        const int64_t n = nb + tg + 8 * i;
        if (n >= a.N) continue;
        float o[V];
#pragma unroll
        for (int j = 0; j < V / 2; j++) unpack2(v[i][j], o[2 * j], o[2 * j + 1]);
        if (slot >= 0) {
            float4 *dst = reinterpret_cast<float4 *>(a.ws + ((int64_t)slot * a.N + n) * R + obase);
#pragma unroll
            for (int j = 0; j < V; j += 4) dst[j / 4] = make_float4(o[j], o[j + 1], o[j + 2], o[j + 3]);
        } else if constexpr (sizeof(T) == 4) {
            float4 *dst = reinterpret_cast<float4 *>(reinterpret_cast<float *>(a.Y) + n * a.M + m);
#pragma unroll
            for (int j = 0; j < V; j += 4)
                dst[j / 4] = make_float4(o[j] + b[j], o[j + 1] + b[j + 1], o[j + 2] + b[j + 2], o[j + 3] + b[j + 3]);
        } else {
            uint32_t pk[V / 2];
#pragma unroll
            for (int j = 0; j < V / 2; j++)
                pk[j] = (uint32_t)from_f32<uint16_t>(o[2 * j] + b[2 * j]) |
                        ((uint32_t)from_f32<uint16_t>(o[2 * j + 1] + b[2 * j + 1]) << 16);
            uint16_t *dst = reinterpret_cast<uint16_t *>(a.Y) + n * a.M + m;
            if constexpr (V == 8)
                *reinterpret_cast<uint4 *>(dst) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            else
                *reinterpret_cast<uint2 *>(dst) = make_uint2(pk[0], pk[1]);
        }
    }
}

template <typename T, int R, int S, int CT>
__global__ void __launch_bounds__((NW + 1) * 32, 1)
k_xrow(const __grid_constant__ CUtensorMap xmap, const XrArgs a) {
    using G = Geo<T, S>;
    extern __shared__ unsigned char smem_raw[];
    Shared sh;
    sh.base = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    sh.full = reinterpret_cast<uint64_t *>(sh.base + a.bar_off);
    sh.empty = sh.full + NS;
    sh.wbar = sh.empty + NS;
    sh.bfree = sh.wbar + 1;
    sh.misc = reinterpret_cast<int *>(sh.base + a.misc_off);
    sh.itab = reinterpret_cast<int *>(sh.base + a.blob_off);
    sh.I = reinterpret_cast<int32_t *>(sh.base + a.blob_off + a.hdr);
    sh.W = reinterpret_cast<float *>(sh.base + a.blob_off + a.hdr + a.ib);

    ptx::pdl_launch_dependents();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t n_tiles = (a.N + G::TN - 1) / G::TN;
    const int64_t total = __ldg(a.cost + a.n_tasks) * n_tiles;
    const int64_t P = gridDim.x;
    const int64_t u_begin = first_unit(a.cost, a.n_tasks, n_tiles, total * (int64_t)blockIdx.x / P);
    const int64_t u_end = first_unit(a.cost, a.n_tasks, n_tiles, total * ((int64_t)blockIdx.x + 1) / P);
    const int nch = a.nchunks;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NS; s++) {
            ptx::mbar_init(&sh.full[s], 1);
            ptx::mbar_init(&sh.empty[s], NW);
        }
        ptx::mbar_init(sh.wbar, 1);
        ptx::mbar_init(sh.bfree, NW);
        sh.misc[0] = 0;
        ptx::fence_barrier_init();
    }
    __syncthreads();
    if (u_begin >= u_end) return;

    if (warp == NW) {
        // ---------------- producer: blobs (one per task) and X chunks
        if (lane == 0) {
            int64_t task = u_begin / n_tiles;
            ptx::mbar_arrive_expect_tx(sh.wbar, a.stride);
            ptx::bulk_load(sh.itab, a.blob + task * a.stride, a.stride, sh.wbar);
            int n_loads = 1;   // blobs issued
            ptx::prefetch_tensormap(&xmap);
            ptx::pdl_wait();   // X may be an earlier kernel's output
            int64_t k = 0;     // ring slots used
            bool ok = true;
            int64_t stalled = -1;
            for (int64_t u = u_begin; ok && u < u_end; u++) {
                const int64_t t = u / n_tiles;
                const int32_t n0 = (int32_t)((u % n_tiles) * G::TN);
                if (t != task) {
                    // every warp is done with the previous task's blob
                    if (!ptx::mbar_wait_bounded(sh.bfree, (n_loads - 1) & 1, a.wait_ns) || aborted(sh.misc)) {
                        ok = false;
                        break;
                    }
                    task = t;
                    ptx::mbar_arrive_expect_tx(sh.wbar, a.stride);
                    ptx::bulk_load(sh.itab, a.blob + task * a.stride, a.stride, sh.wbar);
                    n_loads++;
                }
                for (int c = 0; c < nch; c++, k++) {
                    const int s = (int)(k % NS);
                    if (k >= NS && !ptx::mbar_wait_bounded(&sh.empty[s], (uint32_t)((k / NS) - 1) & 1, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    if (aborted(sh.misc)) { ok = false; break; }
                    if (u == u_begin && c == a.stall_chunk) {   // never loaded: its consumers time out
                        stalled = k;
                        continue;
                    }
                    ptx::mbar_arrive_expect_tx(&sh.full[s], G::kBytes);
#pragma unroll
                    for (int b = 0; b < G::kBoxes; b++)
                        ptx::tma_load_2d(sh.base + s * G::kBytes + b * G::kBoxBytes, &xmap,
                                         c * G::KC + b * G::kBoxCols, n0, &sh.full[s]);
                }
            }
            if (!ok) {
                set_status(a.status, DEV_TIMEOUT);
                atomicExch(&sh.misc[0], 1);
            }
            // copies still in flight must land before the CTA exits
            for (int64_t d = k > NS ? k - NS : 0; d < k; d++)
                if (d != stalled) ptx::mbar_wait_bounded(&sh.full[d % NS], (uint32_t)(d / NS) & 1, kDrainNs);
            ptx::mbar_wait_bounded(sh.wbar, (n_loads - 1) & 1, kDrainNs);
        }
        __syncwarp();
        return;
    }

    // ---------------- consumers
    constexpr int NRG = R / 16;
    const int q = lane >> 3, tg = lane & 7;
    const int rg = q % NRG, ks = q / NRG;
    const uint32_t tgx = (uint32_t)tg << 4;
    const int g = warp / S, sub = warp % S;   // item in the task, 32-token subtile
    const unsigned char *lane_base = sh.base + sub * 4096 + tg * 128;
    int64_t task = -1;
    int n_seen = 0;    // blobs waited for
    int64_t k = 0;
    bool ok = true;
    ptx::pdl_wait();   // Y, the bias and the workspace may be an earlier kernel's
    for (int64_t u = u_begin; ok && u < u_end; u++) {
        const int64_t t = u / n_tiles;
        const int64_t n0 = (u % n_tiles) * G::TN;
        if (t != task) {
            const bool got = ptx::mbar_wait_bounded(sh.wbar, n_seen & 1, a.wait_ns) && !aborted(sh.misc);
            if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
            task = t;
            n_seen++;
        }
        const int *it = sh.itab + g * kItab;
        const int row = it[0], slot = it[1], len = it[2];   // len 0: no item for this warp in the task
        const int32_t *cb = sh.I + it[4];
        const int32_t *bo = cb + ((nch + 4) & ~3);
        const float *wv = sh.W + it[3];
        Acc acc;
        acc.zero();
        for (int c = 0; c < nch; c++, k++) {
            const int s = (int)(k % NS);
            const bool got = ptx::mbar_wait_bounded(&sh.full[s], (uint32_t)(k / NS) & 1, a.wait_ns) && !aborted(sh.misc);
            if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
            if (len > 0) {
                const int lo = cb[c], hi = cb[c + 1];
                const unsigned char *lane_st = lane_base + s * G::kBytes;
                if constexpr (CT == 1)
                    chunk_c1<T, R, S>(acc, lane_st, bo, wv, lo, hi, ks, rg, tgx);
                else
                    chunk_cw<T, R, S>(acc, lane_st, bo, wv, lo, hi, ks, rg, tgx, a.C, c * G::KC);
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sh.empty[s]);
        }
        if (!ok) break;
        if (len > 0) epilogue<T, R, S>(a, acc, row, slot, n0 + sub * 32, tg, rg, ks);
        // the producer may replace the blob once every warp is past this task
        __syncwarp();
        if (lane == 0 && (u + 1 == u_end || (u + 1) / n_tiles != t)) ptx::mbar_arrive(sh.bfree);
    }
    if (!ok && lane == 0) {
        set_status(a.status, DEV_TIMEOUT);
        atomicExch(&sh.misc[0], 1);
    }
}

// Block values into the task blobs of both configurations: item i's values
// go to blobs + vdst[s * n_items + i] (floats; -1: none), blocks in packed
// order (perm[s * nnzb + p0_i + b]: the stored block at position b of the
// item). One column: per block its R values, then 4 zeros. Wider: per block
// its columns, per column its R values in 16-byte groups, group j stored at
// j ^ (((c / cw) % NKS) * R / 16) with NKS = 64 / R lane groups of cw = C /
// NKS columns each.
template <typename T>
__global__ void k_pack_xr(const T *__restrict__ data, const Item *__restrict__ items, const int32_t *__restrict__ perm,
                          const int64_t *__restrict__ vdst, int64_t n_items, int64_t nnzb, float *__restrict__ blobs,
                          int R, int C) {
    const int64_t per_block = C == 1 ? R + 4 : (int64_t)C * R;
    const int NKS = 64 / R, cw = C / NKS;
    for (int64_t gi = blockIdx.x; gi < kXrConfigs * n_items; gi += gridDim.x) {
        const int64_t d = vdst[gi];
        if (d < 0) continue;
        const int s = (int)(gi / n_items);
        const Item it = items[gi % n_items];
        const int64_t total = (int64_t)(it.p1 - it.p0) * per_block;
        for (int64_t e = threadIdx.x; e < total; e += blockDim.x) {
            const int64_t b = e / per_block;
            const int64_t w = e - b * per_block;
            const int64_t p = perm[(int64_t)s * nnzb + it.p0 + b];
            float v = 0.f;
            if (C == 1) {
                if (w < R) v = to_f32(data[p * R + w]);
            } else {
                const int c = (int)(w / R), pos = (int)(w - (int64_t)c * R);
                const int grp = pos >> 2, sw = ((c / cw) % NKS) * (R / 16);
                const int r = ((grp ^ sw) << 2) | (pos & 3);   // the row stored at this position
                v = to_f32(data[(p * R + r) * C + c]);
            }
            blobs[d + e] = v;
        }
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
        else
            cudaGetLastError();
    });
    return fn;
}

template <typename T, int S>
cudaError_t encode_x(const void *X, int64_t N, int64_t K, CUtensorMap *map) {
    auto enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const size_t es = sizeof(T);
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)N};
    const cuuint64_t strides[1] = {(cuuint64_t)K * es};
    const cuuint32_t box[2] = {(cuuint32_t)Geo<T, S>::kBoxCols, (cuuint32_t)Geo<T, S>::TN};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, es == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                     const_cast<void *>(X), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <typename K>
cudaError_t allow_smem(K kernel, std::atomic<uint64_t> &done) {
    int dev = 0;
    cudaGetDevice(&dev);
    const uint64_t bit = 1ull << (dev & 63);
    if (done.load() & bit) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kXrMaxSmem);
    if (e == cudaSuccess) done.fetch_or(bit);
    return e;
}

uint32_t stage_bytes(bsr_dtype_t dt, int s) {
    return (uint32_t)(xrow_tokens(s) * xrow_chunk(s) * (dt == BSR_F32 ? 4 : 2));
}

template <typename T, int R, int S, int CT>
cudaError_t launch_t(const LaunchArgs &la, int s) {
    const Schedule &sc = *la.sc;
    const XrPlan &pl = sc.xr;
    XrArgs a;
    a.blob = static_cast<const unsigned char *>(la.data) + pl.blob_off[s];
    a.cost = reinterpret_cast<const int64_t *>(static_cast<const unsigned char *>(la.data) + pl.cost_off[s]);
    a.stride = pl.stride[s];
    a.G = xrow_G(s);
    a.hdr = (uint32_t)(a.G * kItab * 4);
    a.ib = pl.ibytes[s];
    a.n_tasks = pl.n_tasks[s];
    a.bias = la.bias;
    a.Y = la.Y;
    a.ws = la.ws;
    a.status = la.status;
    a.N = la.N;
    a.K = sc.K;
    a.M = sc.M;
    a.C = sc.C;
    a.nchunks = (int)((sc.K + Geo<T, S>::KC - 1) / Geo<T, S>::KC);
    a.blob_off = NS * Geo<T, S>::kBytes;
    a.bar_off = a.blob_off + a.stride;
    a.misc_off = a.bar_off + (2 * NS + 2) * 8;
    a.wait_ns = la.wait_ns;
    a.stall_chunk = la.stall_chunk;
    const uint32_t smem = a.misc_off + 16 + 1024;
    if (smem > (uint32_t)kXrMaxSmem) return cudaErrorInvalidConfiguration;
    static std::atomic<uint64_t> attr_set{0};
    cudaError_t e = allow_smem(k_xrow<T, R, S, CT>, attr_set);
    if (e != cudaSuccess) return e;
    const int64_t n_tiles = (la.N + Geo<T, S>::TN - 1) / Geo<T, S>::TN;
    const int64_t units = n_tiles * a.n_tasks;
    const int64_t grid = std::min<int64_t>(units, sc.sm_count);
    CUtensorMap map;
    if ((e = encode_x<T, S>(la.X, la.N, sc.K, &map)) != cudaSuccess) return e;
    return launch_kernel(k_xrow<T, R, S, CT>, dim3((unsigned)grid), dim3((NW + 1) * 32), smem, la.stream, map, a);
}

template <typename T, int R, int S>
cudaError_t launch_c(const LaunchArgs &la, int s) {
    return la.sc->C == 1 ? launch_t<T, R, S, 1>(la, s) : launch_t<T, R, S, 0>(la, s);
}

template <typename T>
cudaError_t launch_rs(const LaunchArgs &la, int s) {
    const int R = la.sc->R;
    if (R == 32) return s == 0 ? launch_c<T, 32, 2>(la, s) : launch_c<T, 32, 4>(la, s);
    if (R == 16) return s == 0 ? launch_c<T, 16, 2>(la, s) : launch_c<T, 16, 4>(la, s);
    return cudaErrorNotSupported;
}

}  // namespace

bool xrow_supports(int R, int C, bsr_dtype_t dt, int64_t K) {
    (void)dt;
    const bool c_ok = C == 1 || C == 16 || C == 32;
    const int64_t align = dt == BSR_F32 ? 4 : 8;   // TMA row pitch: a multiple of 16 bytes
    return (R == 16 || R == 32) && c_ok && K % align == 0 && K > 0;
}

size_t xrow_smem_bytes(int s, bsr_dtype_t dt, size_t stride) {
    return (size_t)NS * stage_bytes(dt, s) + stride + (2 * NS + 2) * 8 + 16 + 1024;
}

cudaError_t pack_xrow_data(const void *data, bsr_dtype_t dt, const Item *items, const int32_t *perm,
                           const int64_t *vdst, int64_t n_items, int64_t nnzb, int R, int C, float *blobs,
                           cudaStream_t st) {
    if (n_items == 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>(kXrConfigs * n_items, 1 << 16);
    if (dt == BSR_F32)
        k_pack_xr<float><<<grid, 256, 0, st>>>((const float *)data, items, perm, vdst, n_items, nnzb, blobs, R, C);
    else
        k_pack_xr<uint16_t><<<grid, 256, 0, st>>>((const uint16_t *)data, items, perm, vdst, n_items, nnzb, blobs, R,
                                                  C);
    return cudaGetLastError();
}

cudaError_t launch_xrow(const LaunchArgs &la, int s) {
    if (la.N == 0 || la.sc->items.empty()) return cudaSuccess;
    if (s < 0 || s >= kXrConfigs || !la.sc->xr.ok[s] || la.data == nullptr) return cudaErrorInvalidConfiguration;
    return la.sc->dt == BSR_F32 ? launch_rs<float>(la, s) : launch_rs<uint16_t>(la, s);
}

}  // namespace bsr
