// SIMT BSR x dense kernel with X staged through a TMA ring ("xstage").
//
// Each CTA owns a tile of TN = 64 tokens and a task of G work items (block
// rows or pieces of rows, Section 2.2's kept blocks), S = 8/G consumer warps
// per item. The inner product over the kept blocks is FP32-FMA bound, so the
// design goal is a high FMA:issue ratio:
//
//  * X[n0 : n0+64, k0 : k0+128] chunks stream through a 3-stage shared-memory
//    ring: one producer thread issues 2-D TMA tile loads (128-byte swizzle,
//    rows = tokens) and arms the stage's "full" mbarrier; every consumer warp
//    waits for every chunk in order, processes all of its blocks that fall in
//    it, and releases it on the stage's "empty" mbarrier.
//  * The task's block values (repacked at create time to fp32 [p][c][r]),
//    block-column indices and, per item, the first block of every chunk are
//    put in shared memory once, so the per-chunk loop has no search or test.
//  * Lane = tg + 8 q: tg picks 8 tokens (tg, tg+8, ..., tg+56: conflict-free
//    under the swizzle, which XORs the 16-byte column group with tg), q
//    splits into NRG output groups of TR rows and NKS = 4/NRG lanes that take
//    alternate blocks. A lane accumulates an 8 x TR tile with packed
//    fma.rn.f32x2 (pairs of outputs, or pairs of tokens when TR = 1).
//  * Epilogue: shuffle-reduce the NKS partials, sum the S warps of an item in
//    a fixed order through shared memory, add the bias, convert and store
//    (or write an fp32 partial for rows split across CTAs).
//
// Every wait is bounded by the global timer; a timeout sets the device
// status word, stops the CTA's pipeline, drains its TMA loads and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <mutex>

#include "bsr_internal.h"
#include "elem.cuh"
#include "ptx.cuh"
#include "xstage.h"

namespace bsr {

namespace {

constexpr int TN = kXsTokens;
constexpr int KC = kXsChunk;
constexpr int NS = kXsStages;
constexpr int NCW = kXsConsumerWarps;
constexpr int NTHREADS = (NCW + 1) * 32;
constexpr uint64_t kDrainNs = 2000000000ull;   // generous bound for TMA loads already issued

struct XsArgs {
    const Item *items;
    int n_items, G, S, n_tasks;
    const int32_t *indices;
    const int32_t *cb;       // per item: first block of every chunk, [n_items][nchunks + 1]
    const float *wpk;
    const float *bias;
    void *Y;
    float *ws;
    int *status;
    int64_t N, K, M;
    int C, nchunks;
    uint32_t w_off, idx_off, cb_off, bias_off, bar_off, misc_off;
    int w_bulk;              // block values arrive by one bulk copy per item
    uint64_t wait_ns;
    int stall_chunk;    // test hook: this chunk is never loaded (-1: none)
};

// Shared-memory image of one X chunk: 64 token rows, 128-byte swizzled boxes.
template <typename T>
struct Stage;
template <>
struct Stage<float> {
    static constexpr int kBoxCols = 32;                       // 128 bytes of fp32
    static constexpr int kBoxes = KC / kBoxCols;
    static constexpr uint32_t kBoxBytes = TN * 128;
    static constexpr uint32_t kBytes = kBoxes * kBoxBytes;
    // byte offset of column kk in token row tg (token tg + 8 i adds i * 1024)
    __device__ static __forceinline__ uint32_t off(int kk, int tg) {
        return (uint32_t)((kk >> 5) * kBoxBytes + tg * 128 + ((((kk & 31) >> 2) ^ tg) << 4) + (kk & 3) * 4);
    }
};
template <>
struct Stage<uint16_t> {
    static constexpr int kBoxCols = 64;                       // 128 bytes of bf16
    static constexpr int kBoxes = KC / kBoxCols;
    static constexpr uint32_t kBoxBytes = TN * 128;
    static constexpr uint32_t kBytes = kBoxes * kBoxBytes;
    __device__ static __forceinline__ uint32_t off(int kk, int tg) {
        return (uint32_t)((kk >> 6) * kBoxBytes + tg * 128 + ((((kk & 63) >> 3) ^ tg) << 4) + (kk & 7) * 2);
    }
};

__device__ __forceinline__ float ld_x(const unsigned char *p, float) { return *reinterpret_cast<const float *>(p); }
__device__ __forceinline__ float ld_x(const unsigned char *p, uint16_t) {
    return to_f32(*reinterpret_cast<const uint16_t *>(p));
}
// four consecutive columns
__device__ __forceinline__ float4 ld_x4(const unsigned char *p, float) {
    return *reinterpret_cast<const float4 *>(p);
}
__device__ __forceinline__ float4 ld_x4(const unsigned char *p, uint16_t) {
    const uint2 v = *reinterpret_cast<const uint2 *>(p);
    return make_float4(__uint_as_float(v.x << 16), __uint_as_float(v.x & 0xffff0000u), __uint_as_float(v.y << 16),
                       __uint_as_float(v.y & 0xffff0000u));
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

// acc (8 tokens x TR outputs, packed in pairs) += x (8 tokens) * w (TR outputs)
template <int TR>
struct Tile {
    static constexpr int NP = TR >= 2 ? 8 * TR / 2 : 4;   // packed accumulators
    f2_t a[NP];
    __device__ __forceinline__ void zero() {
#pragma unroll
        for (int k = 0; k < NP; k++) a[k] = 0ull;
    }
    __device__ __forceinline__ void fma(const float (&x)[8], const float (&w)[TR]) {
        if constexpr (TR >= 2) {
            f2_t wp[TR / 2];
#pragma unroll
            for (int j = 0; j < TR / 2; j++) wp[j] = pack2(w[2 * j], w[2 * j + 1]);
#pragma unroll
            for (int i = 0; i < 8; i++) {
                const f2_t xx = pack2(x[i], x[i]);
#pragma unroll
                for (int j = 0; j < TR / 2; j++) a[i * (TR / 2) + j] = ffma2(xx, wp[j], a[i * (TR / 2) + j]);
            }
        } else {
            const f2_t ww = pack2(w[0], w[0]);
#pragma unroll
            for (int i = 0; i < 4; i++) a[i] = ffma2(pack2(x[2 * i], x[2 * i + 1]), ww, a[i]);
        }
    }
    // value for token i, output j
    __device__ __forceinline__ float get(int i, int j) const {
        float lo, hi;
        if constexpr (TR >= 2) {
            unpack2(a[i * (TR / 2) + j / 2], lo, hi);
            return (j & 1) ? hi : lo;
        } else {
            unpack2(a[i / 2], lo, hi);
            return (i & 1) ? hi : lo;
        }
    }
};

template <int TR>
__device__ __forceinline__ void load_w(const float *wr, float (&w)[TR]) {
    if constexpr (TR % 4 == 0) {
#pragma unroll
        for (int j = 0; j < TR; j += 4) {
            const float4 v = *reinterpret_cast<const float4 *>(wr + j);
            w[j] = v.x;
            w[j + 1] = v.y;
            w[j + 2] = v.z;
            w[j + 3] = v.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < TR; j++) w[j] = wr[j];
    }
}

__device__ __forceinline__ void set_status(int *status, int code) { atomicCAS(status, DEV_OK, code); }

__device__ __forceinline__ bool aborted(const int *flag) {
    return *reinterpret_cast<const volatile int *>(flag) != 0;
}

template <typename T, int TR, int NRG>
__global__ void __launch_bounds__(NTHREADS, 1)
k_xstage(const __grid_constant__ CUtensorMap xmap, const XsArgs a) {
    using St = Stage<T>;
    constexpr int NKS = 4 / NRG;
    constexpr int R = TR * NRG;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem =
        reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + a.bar_off);
    uint64_t *empty = full + NS;
    uint64_t *wbar = empty + NS;                              // block values landed
    int *misc = reinterpret_cast<int *>(smem + a.misc_off);   // [0] abort flag, then the item table
    int *itab = misc + 4;                                     // per item: row p0 p1 slot woff ioff
    float *W_s = reinterpret_cast<float *>(smem + a.w_off);
    int32_t *I_s = reinterpret_cast<int32_t *>(smem + a.idx_off);
    int32_t *CB = reinterpret_cast<int32_t *>(smem + a.cb_off);   // [item][nchunks + 1]
    float *B_s = reinterpret_cast<float *>(smem + a.bias_off);      // [item][R]

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // consecutive CTAs take different token tiles, so that concurrent CTAs
    // spread their X reads over many tiles
    const int64_t n_tiles = (a.N + TN - 1) / TN;
    const int task = (int)(blockIdx.x / n_tiles);
    const int64_t n0 = (int64_t)(blockIdx.x % n_tiles) * TN;
    const int item_first = task * a.G;
    const int g_count = min(a.G, a.n_items - item_first);
    const int C = a.C;
    const int nch = a.nchunks;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NS; s++) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], NCW);
        }
        ptx::mbar_init(wbar, 1);
        misc[0] = 0;
        int woff = 0, ioff = 0;
        for (int g = 0; g < g_count; g++) {
            const Item it = a.items[item_first + g];
            const int len = it.p1 - it.p0;
            itab[6 * g + 0] = it.row;
            itab[6 * g + 1] = it.p0;
            itab[6 * g + 2] = it.p1;
            itab[6 * g + 3] = it.slot;
            itab[6 * g + 4] = woff;
            itab[6 * g + 5] = ioff;
            woff += len * R * C;
            ioff += len;
        }
        ptx::fence_barrier_init();
    }
    __syncthreads();

    if (warp == NCW) {
        // ---------------- producer: one thread streams X chunks through the ring
        if (lane == 0) {
            ptx::prefetch_tensormap(&xmap);
            if (a.w_bulk) {
                uint32_t total = 0;
                for (int g = 0; g < g_count; g++) total += (uint32_t)(itab[6 * g + 2] - itab[6 * g + 1]) * R * C * 4;
                ptx::mbar_arrive_expect_tx(wbar, total);
                for (int g = 0; g < g_count; g++) {
                    const uint32_t bytes = (uint32_t)(itab[6 * g + 2] - itab[6 * g + 1]) * R * C * 4;
                    if (bytes)
                        ptx::bulk_load(W_s + itab[6 * g + 4], a.wpk + (int64_t)itab[6 * g + 1] * R * C, bytes, wbar);
                }
            }
            int c = 0;
            bool ok = true;
            for (; c < nch; c++) {
                const int s = c % NS;
                if (c >= NS && !ptx::mbar_wait_bounded(&empty[s], ((c / NS) - 1) & 1, a.wait_ns)) {
                    ok = false;
                    break;
                }
                if (aborted(misc)) { ok = false; break; }
                if (c == a.stall_chunk) continue;   // its consumers time out
                ptx::mbar_arrive_expect_tx(&full[s], St::kBytes);
#pragma unroll
                for (int b = 0; b < St::kBoxes; b++)
                    ptx::tma_load_2d(smem + s * St::kBytes + b * St::kBoxBytes, &xmap,
                                     c * KC + b * St::kBoxCols, (int32_t)n0, &full[s]);
            }
            if (!ok) {
                set_status(a.status, DEV_TIMEOUT);
                atomicExch(&misc[0], 1);
            }
            // the last loads issued may still be in flight: wait (bounded) for
            // them so that no TMA write outlives the CTA
            for (int d = max(0, c - NS); d < c; d++)
                if (d != a.stall_chunk) ptx::mbar_wait_bounded(&full[d % NS], (d / NS) & 1, kDrainNs);
            if (a.w_bulk) ptx::mbar_wait_bounded(wbar, 0, kDrainNs);
        }
        return;
    }

    // ---------------- consumers: stage indices, chunk starts, bias (and block
    // values when they cannot come by bulk copy)
    const int ctid = threadIdx.x;   // 0 .. NCW*32-1
    for (int g = 0; g < g_count; g++) {
        const int p0 = itab[6 * g + 1], len = itab[6 * g + 2] - p0;
        const int ioff = itab[6 * g + 5];
        if (!a.w_bulk) {
            const int woff = itab[6 * g + 4];
            const float *src = a.wpk + (int64_t)p0 * R * C;
            for (int e = ctid; e < len * R * C; e += NCW * 32) W_s[woff + e] = __ldg(src + e);
        }
        for (int e = ctid; e < len; e += NCW * 32) I_s[ioff + e] = __ldg(a.indices + p0 + e);
        const int32_t *cbg = a.cb + (int64_t)(item_first + g) * (nch + 1);
        for (int e = ctid; e <= nch; e += NCW * 32) CB[g * (nch + 1) + e] = __ldg(cbg + e);
        const int64_t m0 = (int64_t)itab[6 * g + 0] * R;
        for (int e = ctid; e < R; e += NCW * 32) B_s[g * R + e] = a.bias ? __ldg(a.bias + m0 + e) : 0.f;
    }
    ptx::named_barrier(1, NCW * 32);
    bool wok = true;
    if (a.w_bulk) wok = __all_sync(0xffffffffu, ptx::mbar_wait_bounded(wbar, 0, a.wait_ns));

    const int q = lane >> 3, tg = lane & 7;
    const int rg = q % NRG, ks = q / NRG;
    const int S = a.S;
    const int gi = warp / S, piece = warp % S;
    const bool has_item = gi < g_count;
    const int woff = has_item ? itab[6 * gi + 4] : 0;
    const int ioff = has_item ? itab[6 * gi + 5] : 0;
    const int32_t *cb = CB + (has_item ? gi : 0) * (nch + 1);
    const float *wbase = W_s + woff + rg * TR;

    Tile<TR> acc;
    acc.zero();
    bool ok = wok;
    for (int c = 0; c < nch && ok; c++) {
        const bool got = ptx::mbar_wait_bounded(&full[c % NS], (c / NS) & 1, a.wait_ns) && !aborted(misc);
        ok = __all_sync(0xffffffffu, got);
        if (!ok) break;
        if (has_item) {
            const unsigned char *st = smem + (c % NS) * St::kBytes;
            const int lo = cb[c], hi = cb[c + 1];
            // this warp's blocks piece + S*jj inside [lo, hi); lanes ks take alternate ones
            const int j0 = lo <= piece ? 0 : (lo - piece + S - 1) / S;
            const int j1 = hi <= piece ? 0 : (hi - piece + S - 1) / S;
            const int kbase = c * KC;
            for (int jj = j0 + ks; jj < j1; jj += NKS) {
                const int lb = piece + S * jj;
                const int kk = I_s[ioff + lb] * C - kbase;
                const float *wb = wbase + lb * C * R;
                if ((C & 3) == 0) {
                    for (int c4 = 0; c4 < C; c4 += 4) {
                        const unsigned char *xp = st + St::off(kk + c4, tg);
                        float4 xv[8];
#pragma unroll
                        for (int i = 0; i < 8; i++) xv[i] = ld_x4(xp + i * 1024, T());
#pragma unroll
                        for (int u = 0; u < 4; u++) {
                            float x[8], w[TR];
#pragma unroll
                            for (int i = 0; i < 8; i++)
                                x[i] = u == 0 ? xv[i].x : u == 1 ? xv[i].y : u == 2 ? xv[i].z : xv[i].w;
                            load_w<TR>(wb + (c4 + u) * R, w);
                            acc.fma(x, w);
                        }
                    }
                } else {
                    for (int cc = 0; cc < C; cc++) {
                        const unsigned char *xp = st + St::off(kk + cc, tg);
                        float x[8], w[TR];
#pragma unroll
                        for (int i = 0; i < 8; i++) x[i] = ld_x(xp + i * 1024, T());
                        load_w<TR>(wb + cc * R, w);
                        acc.fma(x, w);
                    }
                }
            }
        }
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&empty[c % NS]);
    }
    if (!ok && lane == 0) {
        set_status(a.status, DEV_TIMEOUT);
        atomicExch(&misc[0], 1);
    }

    // ---------------- epilogue
    float v[8][TR];
#pragma unroll
    for (int i = 0; i < 8; i++)
#pragma unroll
        for (int j = 0; j < TR; j++) {
            float t = acc.get(i, j);
            if constexpr (NKS >= 2) t += __shfl_xor_sync(0xffffffffu, t, 8 * NRG);
            if constexpr (NKS >= 4) t += __shfl_xor_sync(0xffffffffu, t, 16 * NRG);
            v[i][j] = t;
        }
    // every consumer is done with the ring and W_s; the abort verdict is the
    // same for all of them (barrier reduction), so no thread skips a barrier
    if (ptx::named_barrier_or(1, NCW * 32, !ok || aborted(misc))) return;
    constexpr int PS = R + 4;          // padded row of the partial tile (16-byte aligned)
    float *P = reinterpret_cast<float *>(smem);
    if (ks == 0) {
        float *Pw = P + warp * TN * PS;   // this warp's partial tile [TN][R] (padded rows)
#pragma unroll
        for (int i = 0; i < 8; i++) {
            float *dst = Pw + (tg + 8 * i) * PS + rg * TR;
            if constexpr (TR % 4 == 0) {
#pragma unroll
                for (int j = 0; j < TR; j += 4)
                    *reinterpret_cast<float4 *>(dst + j) = make_float4(v[i][j], v[i][j + 1], v[i][j + 2], v[i][j + 3]);
            } else {
#pragma unroll
                for (int j = 0; j < TR; j++) dst[j] = v[i][j];
            }
        }
    }
    ptx::named_barrier(1, NCW * 32);
    constexpr int V = R % 4 == 0 ? 4 : 1;   // outputs per thread and store
    for (int g = 0; g < g_count; g++) {
        const int row = itab[6 * g + 0], slot = itab[6 * g + 3];
        for (int e = ctid; e < TN * R / V; e += NCW * 32) {
            const int t = (e * V) / R, r = e * V - t * R;
            const int64_t n = n0 + t;
            if (n >= a.N) continue;
            float o[V];
#pragma unroll
            for (int u = 0; u < V; u++) o[u] = 0.f;
            for (int pc = 0; pc < S; pc++) {
                const float *src = P + ((g * S + pc) * TN + t) * PS + r;
                if constexpr (V == 4) {
                    const float4 q4 = *reinterpret_cast<const float4 *>(src);
                    o[0] += q4.x; o[1] += q4.y; o[2] += q4.z; o[3] += q4.w;
                } else {
                    o[0] += src[0];
                }
            }
            const int64_t m = (int64_t)row * R + r;
            if (slot < 0) {
#pragma unroll
                for (int u = 0; u < V; u++) o[u] += B_s[g * R + r + u];
                T *dst = reinterpret_cast<T *>(a.Y) + n * a.M + m;
                if constexpr (V == 4 && sizeof(T) == 4) {
                    *reinterpret_cast<float4 *>(dst) = make_float4(o[0], o[1], o[2], o[3]);
                } else if constexpr (V == 4) {
                    uint2 pk;
                    pk.x = (uint32_t)from_f32<T>(o[0]) | ((uint32_t)from_f32<T>(o[1]) << 16);
                    pk.y = (uint32_t)from_f32<T>(o[2]) | ((uint32_t)from_f32<T>(o[3]) << 16);
                    *reinterpret_cast<uint2 *>(dst) = pk;
                } else {
                    dst[0] = from_f32<T>(o[0]);
                }
            } else {
                float *dst = a.ws + ((int64_t)slot * a.N + n) * R + r;
#pragma unroll
                for (int u = 0; u < V; u++) dst[u] = o[u];
            }
        }
    }
}

// W^T per block, widened to fp32: wpk[(p*C + c)*R + r] = data[(p*R + r)*C + c].
template <typename T>
__global__ void k_pack(const T *__restrict__ data, float *__restrict__ wpk, int64_t nnzb, int R, int C) {
    const int64_t total = nnzb * R * C;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = e / ((int64_t)R * C);
        const int rc = (int)(e - p * R * C);
        const int c = rc / R, r = rc - c * R;
        wpk[e] = to_f32(data[(p * R + r) * C + c]);
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

// ring, reused for the epilogue's partial tiles
size_t region_bytes(bsr_dtype_t dt, int R) {
    const size_t ring = (size_t)NS * (dt == BSR_F32 ? Stage<float>::kBytes : Stage<uint16_t>::kBytes);
    const size_t part = (size_t)NCW * TN * (R + 4) * 4;
    return (std::max(ring, part) + 1023) & ~size_t(1023);
}

template <typename T, int TR, int NRG>
cudaError_t launch_t(const LaunchArgs &la, const XsPlan &pl, int G) {
    const Schedule &sc = *la.sc;
    const size_t es = sizeof(T);
    const int gidx = g_index(G);
    const int n_items = (int)sc.items.size();
    if (n_items == 0 || la.N == 0) return cudaSuccess;
    CUtensorMap map;
    auto enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const cuuint64_t dims[2] = {(cuuint64_t)sc.K, (cuuint64_t)la.N};
    const cuuint64_t strides[1] = {(cuuint64_t)sc.K * es};
    const cuuint32_t box[2] = {(cuuint32_t)Stage<T>::kBoxCols, (cuuint32_t)TN};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(&map, es == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                     const_cast<void *>(la.X), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;

    XsArgs a;
    a.items = sc.d_items;
    a.n_items = n_items;
    a.G = G;
    a.S = NCW / G;
    a.n_tasks = (n_items + G - 1) / G;
    a.indices = sc.d_indices;
    a.wpk = static_cast<const float *>(la.data);
    a.bias = la.bias;
    a.Y = la.Y;
    a.ws = la.ws;
    a.status = la.status;
    a.N = la.N;
    a.K = sc.K;
    a.M = sc.M;
    a.C = sc.C;
    a.nchunks = (int)((sc.K + KC - 1) / KC);
    a.w_off = (uint32_t)region_bytes(sc.dt, sc.R);
    a.idx_off = a.w_off + (uint32_t)((pl.task_wbytes[gidx] + 15) & ~size_t(15));
    a.cb_off = a.idx_off + (uint32_t)((pl.task_ibytes[gidx] + 15) & ~size_t(15));
    a.bias_off = a.cb_off + (uint32_t)(((size_t)G * (a.nchunks + 1) * 4 + 15) & ~size_t(15));
    a.bar_off = a.bias_off + (uint32_t)(((size_t)G * sc.R * 4 + 15) & ~size_t(15));
    a.cb = sc.d_xs_cb;
    a.w_bulk = (sc.R * sc.C) % 4 == 0;
    a.misc_off = a.bar_off + (2 * NS + 1) * 8;
    const uint32_t smem = a.misc_off + (4 + 6 * 8) * 4 + 1024;   // + slack to align the base
    a.wait_ns = la.wait_ns;
    a.stall_chunk = la.stall_chunk;
    static std::atomic<uint64_t> attr_set{0};   // per instantiation, one bit per device
    int dev = 0;
    cudaGetDevice(&dev);
    const uint64_t bit = 1ull << (dev & 63);
    if (!(attr_set.load() & bit)) {
        cudaError_t e = cudaFuncSetAttribute(k_xstage<T, TR, NRG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kXsMaxSmem);
        if (e != cudaSuccess) return e;
        attr_set.fetch_or(bit);
    }
    if (smem > kXsMaxSmem) return cudaErrorInvalidConfiguration;
    const int64_t n_tiles = (la.N + TN - 1) / TN;
    const int64_t grid = n_tiles * a.n_tasks;   // tile-fastest order
    if (grid > INT32_MAX) return cudaErrorInvalidConfiguration;
    k_xstage<T, TR, NRG><<<(unsigned)grid, NTHREADS, smem, la.stream>>>(map, a);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_r(const LaunchArgs &la, const XsPlan &pl, int G) {
    switch (la.sc->R) {
        case 1: return launch_t<T, 1, 1>(la, pl, G);
        case 2: return launch_t<T, 2, 1>(la, pl, G);
        case 4: return launch_t<T, 4, 1>(la, pl, G);
        case 8: return launch_t<T, 8, 1>(la, pl, G);
        case 16: return launch_t<T, 8, 2>(la, pl, G);
        case 32: return launch_t<T, 8, 4>(la, pl, G);
    }
    return cudaErrorNotSupported;
}

}  // namespace

size_t xstage_smem_bytes(bsr_dtype_t dt, int R, int64_t K, int G, size_t wbytes, size_t ibytes) {
    const size_t nch = (size_t)((K + KC - 1) / KC);
    return region_bytes(dt, R) + ((wbytes + 15) & ~size_t(15)) + ((ibytes + 15) & ~size_t(15)) +
           (((size_t)G * (nch + 1) * 4 + 15) & ~size_t(15)) + (((size_t)G * R * 4 + 15) & ~size_t(15)) +
           (2 * NS + 1) * 8 + (4 + 6 * 8) * 4 + 1024;
}

size_t xstage_task_budget(bsr_dtype_t dt, int R, int64_t K) {
    const size_t fixed = xstage_smem_bytes(dt, R, K, 8, 0, 0) + 64;
    return fixed >= (size_t)kXsMaxSmem ? 0 : (size_t)kXsMaxSmem - fixed;
}

int g_index(int G) { return G == 1 ? 0 : G == 2 ? 1 : G == 4 ? 2 : 3; }

bool xstage_supports(int R, int C, bsr_dtype_t dt, int64_t K) {
    const bool r_ok = R == 1 || R == 2 || R == 4 || R == 8 || R == 16 || R == 32;
    const bool c_ok = C >= 1 && C <= kXsChunk && kXsChunk % C == 0;
    const int64_t align = dt == BSR_F32 ? 4 : 8;   // TMA row pitch must be a multiple of 16 bytes
    return r_ok && c_ok && K % align == 0 && K > 0;
}

cudaError_t pack_xstage_data(const void *data, bsr_dtype_t dt, int64_t nnzb, int R, int C, float *wpk,
                             cudaStream_t s) {
    const int64_t total = nnzb * R * C;
    if (total == 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>((total + 255) / 256, 1 << 20);
    if (dt == BSR_F32)
        k_pack<float><<<grid, 256, 0, s>>>((const float *)data, wpk, nnzb, R, C);
    else
        k_pack<uint16_t><<<grid, 256, 0, s>>>((const uint16_t *)data, wpk, nnzb, R, C);
    return cudaGetLastError();
}

cudaError_t launch_xstage(const LaunchArgs &la, int G) {
    const XsPlan &pl = la.sc->xs;
    if (la.sc->dt == BSR_F32) return launch_r<float>(la, pl, G);
    return launch_r<uint16_t>(la, pl, G);
}

}  // namespace bsr
