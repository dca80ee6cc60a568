// SIMT BSR x dense kernel with X staged through a TMA ring ("xstage").
//
// Each CTA owns a tile of TN = 64 tokens and a task of G work items (block
// rows or pieces of rows, Section 2.2's kept blocks), with NW consumer warps
// and one producer warp: S = NW/G warps per item for G <= NW (NW = 14), or,
// for one-row blocks (NW = 24), G/NW whole items per warp when G > NW. The
// inner product over the kept blocks is FP32-FMA bound, so the design goal
// is a high share of packed FMAs among the issued instructions:
//
//  * X[n0 : n0+64, k0 : k0+128] chunks stream through a 3-stage
//    shared-memory ring: the producer thread loads each chunk with 2-D TMA
//    tile loads (128-byte swizzle, rows = tokens) into its own stage. A
//    stage's "full" mbarrier counts the chunk's bytes; every consumer warp
//    waits for every chunk in order, processes all of its blocks that fall
//    in it, and releases the stage on the stage's "empty" mbarrier.
//  * Per task, the producer bulk-copies one blob (built at create time):
//    the item table, the items' records -- each block's X offset inside a
//    stage (1-column blocks) or block column, and the first block of every
//    chunk, so the per-chunk loop has no search or test -- and the block
//    values (fp32 [p][c][r]; 1x1 weights sit in the records).
//  * Lane = tg + 8 q: tg picks 8 tokens (tg, tg+8, ..., tg+56: conflict-free
//    under the swizzle, which XORs the 16-byte column group with tg), q
//    splits into NRG output groups of TR rows and NKS = 4/NRG lanes that take
//    alternate blocks (or, for wide blocks, a quarter or half of each
//    block's columns). A lane accumulates an 8 x TR tile with packed
//    fma.rn.f32x2 over pairs of tokens: (x_t, x_t') * (w, w).
//  * Epilogue: shuffle-reduce the NKS partials. A warp that owns whole
//    items stores its tile straight from registers (one item per warp) or
//    through a shared-memory slot; the S warps of a shared item write their
//    partial tiles to slots, and one pass over all of the task's outputs sums
//    them in piece order, adds the bias, converts and stores row segments of
//    Y (or writes an fp32 partial for rows split across CTAs).
//  * The kernel is launched with programmatic stream serialisation: it lets
//    the next kernel start at once, and fetches its blob and sets up its
//    barriers before it waits for the previous kernel (X, bias and Y are
//    touched only after that wait).
//
// Every wait is bounded by the global timer; a timeout sets the device
// status word, stops the CTA's pipeline and drains its TMA loads.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdlib>
#include <mutex>
#include <vector>

#include "bsr_internal.h"
#include "elem.cuh"
#include "launch.cuh"
#include "ptx.cuh"
#include "xstage.h"

namespace bsr {

namespace {

constexpr int TN = kXsTokens;
constexpr int KC = kXsChunk;
constexpr int NS = kXsStages;
constexpr int NCW = kXsConsumerWarps;
constexpr int WD = kXsWDup;
constexpr int kItab = kXsItab;   // ints per item in a task's item table
constexpr uint64_t kDrainNs = 200000000ull;   // bound for TMA loads already issued (they take microseconds)

struct XsArgs {
    int n_items, G, S, n_tasks;
    const unsigned char *blob;   // task t's blob at blob + t * stride (see xstage.h)
    uint32_t stride, hdr, ib;    // blob bytes per task, item-table bytes, record-region bytes
    const float *bias;
    void *Y;
    float *ws;
    int *status;
    int64_t N, K, M;
    int C, nchunks;
    uint32_t blob_off, bias_off, bar_off, misc_off;   // shared-memory offsets
    uint64_t wait_ns;
    int stall_chunk;         // test hook: this chunk is never loaded (-1: none)
};

// Shared-memory image of one X chunk: 64 token rows, 128-byte swizzled boxes.
// off0(kk) is the byte offset of chunk column kk in token row 0; token tg + 8 i
// is at (off0 ^ (tg << 4)) + tg * 128 + i * 1024.
template <typename T>
struct Stage;
template <>
struct Stage<float> {
    static constexpr int kBoxCols = 32;                       // 128 bytes of fp32
    static constexpr int kBoxes = KC / kBoxCols;
    static constexpr uint32_t kBoxBytes = TN * 128;
    static constexpr uint32_t kBytes = kBoxes * kBoxBytes;
    __host__ __device__ static __forceinline__ uint32_t off0(int kk) {
        return (uint32_t)((kk >> 5) * kBoxBytes + (((kk & 31) >> 2) << 4) + (kk & 3) * 4);
    }
};
template <>
struct Stage<uint16_t> {
    static constexpr int kBoxCols = 64;                       // 128 bytes of bf16
    static constexpr int kBoxes = KC / kBoxCols;
    static constexpr uint32_t kBoxBytes = TN * 128;
    static constexpr uint32_t kBytes = kBoxes * kBoxBytes;
    __host__ __device__ static __forceinline__ uint32_t off0(int kk) {
        return (uint32_t)((kk >> 6) * kBoxBytes + (((kk & 63) >> 3) << 4) + (kk & 7) * 2);
    }
};

__device__ __forceinline__ float ld_x(const unsigned char *p, float) { return *reinterpret_cast<const float *>(p); }
__device__ __forceinline__ float ld_x(const unsigned char *p, uint16_t) {
    return to_f32(*reinterpret_cast<const uint16_t *>(p));
}
// four consecutive columns of one token
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

// acc (8 tokens x TR outputs) += x (8 tokens) * w (TR outputs); accumulators
// packed over token pairs (i, i+1) for i even.
template <int TR>
struct Tile {
    f2_t a[4 * TR];
    __device__ __forceinline__ void zero() {
#pragma unroll
        for (int k = 0; k < 4 * TR; k++) a[k] = 0ull;
    }
    // wd[j] = (w_j, w_j): the weight of output j, duplicated for both tokens
    __device__ __forceinline__ void fma(const float (&x)[8], const f2_t (&wd)[TR]) {
#pragma unroll
        for (int ip = 0; ip < 4; ip++) {
            const f2_t xp = pack2(x[2 * ip], x[2 * ip + 1]);
#pragma unroll
            for (int j = 0; j < TR; j++) a[ip * TR + j] = ffma2(xp, wd[j], a[ip * TR + j]);
        }
    }
    __device__ __forceinline__ float get(int i, int j) const {
        float lo, hi;
        unpack2(a[(i >> 1) * TR + j], lo, hi);
        return (i & 1) ? hi : lo;
    }
};

// one output per lane: plain fp32 FMA, no operand pairs to form (measured
// faster than the packed form for this load-bound tile)
template <>
struct Tile<1> {
    float a[8];
    __device__ __forceinline__ void zero() {
#pragma unroll
        for (int k = 0; k < 8; k++) a[k] = 0.f;
    }
    __device__ __forceinline__ void fma(const float (&x)[8], const f2_t (&wd)[1]) {
        float w, w2;
        unpack2(wd[0], w, w2);
#pragma unroll
        for (int i = 0; i < 8; i++) a[i] = fmaf(x[i], w, a[i]);
    }
    __device__ __forceinline__ float get(int i, int) const { return a[i]; }
};

// The TR weights of one block column for this lane, each as a (w, w) pair.
// With WD == 2 the packed values already hold every weight twice, so the
// pairs come straight from shared loads.
template <int TR>
__device__ __forceinline__ void load_wd(const float *wr, f2_t (&wd)[TR]) {
    if constexpr (WD == 2) {
        if constexpr (TR == 1) {
            wd[0] = *reinterpret_cast<const f2_t *>(wr);
        } else {
#pragma unroll
            for (int j = 0; j < TR; j += 2) {
                const ulonglong2 v = *reinterpret_cast<const ulonglong2 *>(wr + 2 * j);
                wd[j] = v.x;
                wd[j + 1] = v.y;
            }
        }
    } else if constexpr (TR % 4 == 0) {
#pragma unroll
        for (int j = 0; j < TR; j += 4) {
            const float4 v = *reinterpret_cast<const float4 *>(wr + j);
            wd[j] = pack2(v.x, v.x);
            wd[j + 1] = pack2(v.y, v.y);
            wd[j + 2] = pack2(v.z, v.z);
            wd[j + 3] = pack2(v.w, v.w);
        }
    } else if constexpr (TR == 2) {
        const float2 v = *reinterpret_cast<const float2 *>(wr);
        wd[0] = pack2(v.x, v.x);
        wd[1] = pack2(v.y, v.y);
    } else {
        wd[0] = pack2(wr[0], wr[0]);
    }
}

__device__ __forceinline__ void set_status(int *status, int code) { atomicCAS(status, DEV_OK, code); }

__device__ __forceinline__ bool aborted(const int *flag) {
    return *reinterpret_cast<const volatile int *>(flag) != 0;
}

struct Shared {
    unsigned char *base;
    uint64_t *full, *empty, *wbar;
    int *misc;          // [0] abort flag, [3] task covers consecutive whole rows
    int *itab;          // the blob's item table (kItab ints per item)
    float *W;           // block values of the task's items
    int32_t *I;         // the task's item records
    float *B;           // [item][R] bias
};

// The blocks of one item that fall in X chunk c, for one lane: blocks
// piece + S*jj inside the chunk's range, lanes ks taking alternate ones.
template <typename T, int TR, int NRG, int CT>
__device__ __forceinline__ void item_chunk(Tile<TR> &acc, const unsigned char *st, const int32_t *idx,
                                           const int32_t *cb, const float *wbase, int c, int piece, int S, int ks,
                                           uint32_t tgx, int C) {
    using St = Stage<T>;
    constexpr int NKS = 4 / NRG;
    constexpr int R = TR * NRG;
    const int lo = cb[c], hi = cb[c + 1];
    if constexpr (CT == 1) {
        // groups of NKS consecutive blocks (ordered on the host so that a
        // group's columns fall in distinct banks), dealt round-robin to the
        // S warps of the item; lane group ks takes block ks of each group
        const int ngr = (hi - lo + NKS - 1) / NKS;
        for (int jg = piece; jg < ngr; jg += S) {
            const int lb = lo + jg * NKS + ks;
            if (NKS > 1 && lb >= hi) continue;
            uint32_t off;
            f2_t wd[TR];
            if constexpr (R == 1) {
                // 1x1: (X offset, weight) in one 8-byte record entry
                const int2 ow = reinterpret_cast<const int2 *>(idx)[lb];
                off = (uint32_t)ow.x ^ tgx;
                wd[0] = pack2(__int_as_float(ow.y), __int_as_float(ow.y));
            } else {
                off = (uint32_t)idx[lb] ^ tgx;
                load_wd<TR>(wbase + lb * R * WD, wd);
            }
            float x[8];
#pragma unroll
            for (int i = 0; i < 8; i++) x[i] = ld_x(st + off + i * 1024, T());
            acc.fma(x, wd);
        }
        return;
    } else {
        // wide blocks (a multiple of 4 columns per lane group): the NKS lane
        // groups split each block's columns, so no lanes idle when a chunk
        // holds fewer blocks than groups; narrow blocks: groups take
        // alternate blocks
        int j0 = lo, j1 = hi;
        if (S > 1) {
            j0 = lo <= piece ? 0 : (lo - piece + S - 1) / S;
            j1 = hi <= piece ? 0 : (hi - piece + S - 1) / S;
        }
        const int kbase = c * KC;
        const bool csplit = NKS > 1 && C % (4 * NKS) == 0;
        const int cw = csplit ? C / NKS : C;
        const int cc0 = csplit ? ks * cw : 0;
        for (int jj = csplit ? j0 : j0 + ks; jj < j1; jj += csplit ? 1 : NKS) {
            const int lb = piece + S * jj;
            const int kk = idx[lb] * C - kbase;
            const float *wb = wbase + lb * C * R * WD;
            if (TR < 8 && (cw & 3) == 0) {   // four columns per load, where registers allow
                for (int c4 = cc0; c4 < cc0 + cw; c4 += 4) {
                    const unsigned char *xp = st + (St::off0(kk + c4) ^ tgx);
                    float4 xv[8];
#pragma unroll
                    for (int i = 0; i < 8; i++) xv[i] = ld_x4(xp + i * 1024, T());
#pragma unroll
                    for (int u = 0; u < 4; u++) {
                        float x[8];
                        f2_t wd[TR];
#pragma unroll
                        for (int i = 0; i < 8; i++)
                            x[i] = u == 0 ? xv[i].x : u == 1 ? xv[i].y : u == 2 ? xv[i].z : xv[i].w;
                        load_wd<TR>(wb + (c4 + u) * R * WD, wd);
                        acc.fma(x, wd);
                    }
                }
            } else {
                for (int cc = cc0; cc < cc0 + cw; cc++) {
                    const unsigned char *xp = st + (St::off0(kk + cc) ^ tgx);
                    float x[8];
                    f2_t wd[TR];
#pragma unroll
                    for (int i = 0; i < 8; i++) x[i] = ld_x(xp + i * 1024, T());
                    load_wd<TR>(wb + cc * R * WD, wd);
                    acc.fma(x, wd);
                }
            }
        }
    }
}

// The lane's 8 x TR tile with the NKS block-splitting lanes summed in.
template <int TR, int NRG>
__device__ __forceinline__ void reduce_tile(const Tile<TR> &acc, float (&v)[8][TR]) {
    constexpr int NKS = 4 / NRG;
#pragma unroll
    for (int i = 0; i < 8; i++)
#pragma unroll
        for (int j = 0; j < TR; j++) {
            float t = acc.get(i, j);
            if constexpr (NKS >= 2) t += __shfl_xor_sync(0xffffffffu, t, 8 * NRG);
            if constexpr (NKS >= 4) t += __shfl_xor_sync(0xffffffffu, t, 16 * NRG);
            v[i][j] = t;
        }
}

// A lane's reduced 8 x TR tile into slot `slot` of the token-major slot
// array ([t][slot][r], token pitch P floats). All NKS lanes of a token group
// hold the same sums; lane ks writes tokens i = ks mod NKS.
template <int TR, int NRG, int P>
__device__ __forceinline__ void write_slot(float *slots, int slot, const float (&v)[8][TR], int tg, int rg, int ks) {
    constexpr int R = TR * NRG;
    constexpr int NKS = 4 / NRG;
    float *base = slots + slot * R + rg * TR;
#pragma unroll
    for (int i = 0; i < 8; i++) {
        if (i % NKS != ks) continue;
        float *dst = base + (tg + 8 * i) * P;
        if constexpr (TR % 4 == 0) {
#pragma unroll
            for (int j = 0; j < TR; j += 4)
                *reinterpret_cast<float4 *>(dst + j) = make_float4(v[i][j], v[i][j + 1], v[i][j + 2], v[i][j + 3]);
        } else if constexpr (TR == 2) {
            *reinterpret_cast<float2 *>(dst) = make_float2(v[i][0], v[i][1]);
        } else {
            dst[0] = v[i][0];
        }
    }
}

// Item gi's finished tile straight from the registers of the one warp that
// owns it: + bias, converted, to Y; or, for a piece of a split row, the fp32
// partial to its workspace slot. The NKS lanes of a token group hold the
// same sums; lane ks stores tokens i = ks mod NKS.
template <typename T, int TR, int NRG>
__device__ __forceinline__ void store_tile(const XsArgs &a, const Shared &sh, const float (&v)[8][TR], int gi,
                                           int64_t n0, int rg, int tg, int ks) {
    constexpr int R = TR * NRG;
    constexpr int NKS = 4 / NRG;
    const int row = sh.itab[kItab * gi + 0], slot = sh.itab[kItab * gi + 3];
    const int64_t m = (int64_t)row * R + rg * TR;
    float b[TR];
#pragma unroll
    for (int j = 0; j < TR; j++) b[j] = slot < 0 ? sh.B[gi * R + rg * TR + j] : 0.f;
#pragma unroll
    for (int i = 0; i < 8; i++) {
        const int64_t n = n0 + tg + 8 * i;
        if (i % NKS != ks || n >= a.N) continue;
        if (slot < 0) {
            T *dst = reinterpret_cast<T *>(a.Y) + n * a.M + m;
            if constexpr (sizeof(T) == 4 && TR % 4 == 0) {
#pragma unroll
                for (int j = 0; j < TR; j += 4)
                    *reinterpret_cast<float4 *>(dst + j) =
                        make_float4(v[i][j] + b[j], v[i][j + 1] + b[j + 1], v[i][j + 2] + b[j + 2], v[i][j + 3] + b[j + 3]);
            } else if constexpr (sizeof(T) == 2 && TR % 4 == 0) {
#pragma unroll
                for (int j = 0; j < TR; j += 4) {
                    uint2 pk;
                    pk.x = (uint32_t)from_f32<T>(v[i][j] + b[j]) | ((uint32_t)from_f32<T>(v[i][j + 1] + b[j + 1]) << 16);
                    pk.y = (uint32_t)from_f32<T>(v[i][j + 2] + b[j + 2]) |
                           ((uint32_t)from_f32<T>(v[i][j + 3] + b[j + 3]) << 16);
                    *reinterpret_cast<uint2 *>(dst + j) = pk;
                }
            } else {
#pragma unroll
                for (int j = 0; j < TR; j++) dst[j] = from_f32<T>(v[i][j] + b[j]);
            }
        } else {
            float *dst = a.ws + ((int64_t)slot * a.N + n) * R + rg * TR;
#pragma unroll
            for (int j = 0; j < TR; j++) dst[j] = v[i][j];
        }
    }
}

// Output pass, after every consumer warp wrote its slot: item g's tile is
// the sum of the S slots g*S .. g*S+S-1 in piece order (a fixed order, so
// results repeat bit for bit) plus the bias; converted and stored to Y, or,
// for a piece of a split row, the fp32 partial to its workspace slot. Lanes
// take VW-wide vectors along the task's outputs and warps take tokens (TPW
// each, loaded together so their shared-memory latencies overlap), so each
// store instruction writes whole row segments of Y.
template <typename T, int R, int NW, int P>
__device__ __forceinline__ void output_pass(const XsArgs &a, const Shared &sh, const float *slots, int S,
                                            int g_count, int64_t n0, int warp, int lane) {
    constexpr int VW = R >= 4 ? 4 : R;   // outputs per vector
    constexpr int VPI = R / VW;          // vectors per item and token
    constexpr int TPW = (TN + NW - 1) / NW;
    const int nvec = g_count * VPI;
    for (int c = lane; c < nvec; c += 32) {
        const int g = c / VPI, r = (c - g * VPI) * VW;
        const int row = sh.itab[kItab * g + 0], wslot = sh.itab[kItab * g + 3];
        float y[TPW][VW];
#pragma unroll
        for (int k = 0; k < TPW; k++)
#pragma unroll
            for (int v = 0; v < VW; v++) y[k][v] = 0.f;
        const float *src = slots + (g * S) * R + r;
        for (int pc = 0; pc < S; pc++, src += R) {
#pragma unroll
            for (int k = 0; k < TPW; k++) {
                const int t = warp + k * NW;
                if (TN % NW != 0 && t >= TN) continue;
                const float *q = src + t * P;
                if constexpr (VW == 4) {
                    const float4 q4 = *reinterpret_cast<const float4 *>(q);
                    y[k][0] += q4.x;
                    y[k][1] += q4.y;
                    y[k][2] += q4.z;
                    y[k][3] += q4.w;
                } else if constexpr (VW == 2) {
                    const float2 q2 = *reinterpret_cast<const float2 *>(q);
                    y[k][0] += q2.x;
                    y[k][1] += q2.y;
                } else {
                    y[k][0] += *q;
                }
            }
        }
        float b[VW];
#pragma unroll
        for (int v = 0; v < VW; v++) b[v] = wslot >= 0 ? 0.f : sh.B[g * R + r + v];
#pragma unroll
        for (int k = 0; k < TPW; k++) {
            const int t = warp + k * NW;
            const int64_t n = n0 + t;
            if ((TN % NW != 0 && t >= TN) || n >= a.N) continue;
            if (wslot >= 0) {
                float *dst = a.ws + ((int64_t)wslot * a.N + n) * R + r;
#pragma unroll
                for (int v = 0; v < VW; v++) dst[v] = y[k][v];
                continue;
            }
            float o[VW];
#pragma unroll
            for (int v = 0; v < VW; v++) o[v] = y[k][v] + b[v];
            T *dst = reinterpret_cast<T *>(a.Y) + n * a.M + (int64_t)row * R + r;
            if constexpr (sizeof(T) == 4 && VW == 4) {
                *reinterpret_cast<float4 *>(dst) = make_float4(o[0], o[1], o[2], o[3]);
            } else if constexpr (sizeof(T) == 4 && VW == 2) {
                *reinterpret_cast<float2 *>(dst) = make_float2(o[0], o[1]);
            } else if constexpr (sizeof(T) == 2 && VW == 4) {
                uint2 pk;
                pk.x = (uint32_t)from_f32<T>(o[0]) | ((uint32_t)from_f32<T>(o[1]) << 16);
                pk.y = (uint32_t)from_f32<T>(o[2]) | ((uint32_t)from_f32<T>(o[3]) << 16);
                *reinterpret_cast<uint2 *>(dst) = pk;
            } else if constexpr (sizeof(T) == 2 && VW == 2) {
                *reinterpret_cast<uint32_t *>(dst) =
                    (uint32_t)from_f32<T>(o[0]) | ((uint32_t)from_f32<T>(o[1]) << 16);
            } else {
                dst[0] = from_f32<T>(o[0]);
            }
        }
    }
}

// NW consumer warps. RW == 1: S = NW/G warps share each item (block-strided)
// and a pairwise tree sums them. RW > 1 (G = NW RW): each warp owns RW
// whole items, with one register tile each, and needs no tree.
template <typename T, int TR, int NRG, int CT, int RW, int NW>
__device__ __forceinline__ void consumer(const XsArgs &a, const Shared &sh, int64_t n0, int task,
                                         int g_count, int warp, int lane) {
    using St = Stage<T>;
    constexpr int R = TR * NRG;
    const int C = CT ? CT : a.C;
    const int nch = a.nchunks;
    const int ctid = threadIdx.x;   // 0 .. NW*32-1
    const int BI = xstage_block_ints(R, C);   // record ints per block

    // ---- the task's blob (item table, records, block values): one bulk
    // copy the producer issued first thing, one round trip
    if (g_count > 0 && !__all_sync(0xffffffffu, ptx::mbar_wait_bounded(sh.wbar, 0, a.wait_ns))) {
        if (lane == 0) {
            set_status(a.status, DEV_TIMEOUT);
            atomicExch(&sh.misc[0], 1);
        }
    }
    ptx::named_barrier(1, NW * 32);
    ptx::pdl_wait();   // the bias, Y and the workspace may be an earlier kernel's
    // the bias, needed only by the output pass (waited for there)
    for (int e = ctid; e < g_count * R; e += NW * 32) {
        const int g = e / R, r = e - g * R;
        if (a.bias)
            ptx::cp_async4(&sh.B[e], a.bias + (int64_t)sh.itab[kItab * g + 0] * R + r);
        else
            sh.B[e] = 0.f;
    }
    bool ok = true;
    float *slots = reinterpret_cast<float *>(sh.base);   // the ring, free once every warp is past it
    constexpr int PRW = xstage_slot_pitch(R, NW * RW);   // token pitch of the slots: one per item (RW > 1)
    constexpr int PS = xstage_slot_pitch(R, NW);         // one per warp

    const int q = lane >> 3, tg = lane & 7;
    const int rg = q % NRG, ks = q / NRG;
    const uint32_t tgx = (uint32_t)tg << 4;
    const unsigned char *lane_base = sh.base + tg * 128;

    if constexpr (RW > 1) {
        Tile<TR> acc[RW];
#pragma unroll
        for (int r = 0; r < RW; r++) acc[r].zero();
        for (int c = 0; c < nch && ok; c++) {
            const bool got = ptx::mbar_wait_bounded(&sh.full[c % NS], (c / NS) & 1, a.wait_ns) && !aborted(sh.misc);
            ok = __all_sync(0xffffffffu, got);
            if (!ok) break;
            const unsigned char *st = lane_base + (c % NS) * St::kBytes;
#pragma unroll
            for (int r = 0; r < RW; r++) {
                const int gi = warp * RW + r;
                if (gi < g_count) {
                    const int32_t *idx = sh.I + sh.itab[kItab * gi + 8];
                    const int32_t *cb = idx + xstage_pad4(BI * sh.itab[kItab * gi + 5]);
                    const float *wbase = sh.W + sh.itab[kItab * gi + 7] + rg * TR * WD;
                    item_chunk<T, TR, NRG, CT>(acc[r], st, idx, cb, wbase, c, 0, 1, ks, tgx, C);
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sh.empty[c % NS]);
        }
        if (!ok && lane == 0) {
            set_status(a.status, DEV_TIMEOUT);
            atomicExch(&sh.misc[0], 1);
        }
        ptx::cp_async_wait_all();   // the bias
        if (ptx::named_barrier_or(1, NW * 32, !ok || aborted(sh.misc))) return;
#pragma unroll
        for (int r = 0; r < RW; r++) {
            const int gi = warp * RW + r;
            float v[8][TR];
            reduce_tile<TR, NRG>(acc[r], v);
            if (gi < g_count) write_slot<TR, NRG, PRW>(slots, gi, v, tg, rg, ks);
        }
        ptx::named_barrier(1, NW * 32);
        output_pass<T, R, NW, PRW>(a, sh, slots, 1, g_count, n0, warp, lane);
        return;
    }

    const int S = a.S;
    const int gi = warp / S, piece = warp % S;
    const bool has_item = gi < g_count;
    const int32_t *idx = sh.I + (has_item ? sh.itab[kItab * gi + 8] : 0);
    const int32_t *cb = idx + (has_item ? xstage_pad4(BI * sh.itab[kItab * gi + 5]) : 0);
    const float *wbase = sh.W + (has_item ? sh.itab[kItab * gi + 7] : 0) + rg * TR * WD;

    Tile<TR> acc;
    acc.zero();
    for (int c = 0; c < nch && ok; c++) {
        const bool got = ptx::mbar_wait_bounded(&sh.full[c % NS], (c / NS) & 1, a.wait_ns) && !aborted(sh.misc);
        ok = __all_sync(0xffffffffu, got);
        if (!ok) break;
        if (has_item)
            item_chunk<T, TR, NRG, CT>(acc, lane_base + (c % NS) * St::kBytes, idx, cb, wbase, c, piece, S, ks, tgx, C);
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&sh.empty[c % NS]);
    }
    if (!ok && lane == 0) {
        set_status(a.status, DEV_TIMEOUT);
        atomicExch(&sh.misc[0], 1);
    }

    // ---- epilogue
    float v[8][TR];
    reduce_tile<TR, NRG>(acc, v);
    // every consumer is done with the ring and the block values; the abort
    // verdict is the same for all of them (barrier reduction)
    ptx::cp_async_wait_all();   // the bias
    if (ptx::named_barrier_or(1, NW * 32, !ok || aborted(sh.misc))) return;
    if (S == 1) {   // one warp per item: no partial tiles to combine
        if (has_item) store_tile<T, TR, NRG>(a, sh, v, gi, n0, rg, tg, ks);
        return;
    }
    // every warp's tile to its slot (slot = warp = item * S + piece), then
    // the output pass over all items
    if (has_item) write_slot<TR, NRG, PS>(slots, warp, v, tg, rg, ks);
    ptx::named_barrier(1, NW * 32);
    output_pass<T, R, NW, PS>(a, sh, slots, S, g_count, n0, warp, lane);
}

// One CTA of the product described by `a`; `cta` is the CTA's index within
// that product's grid (token tiles fastest, then tasks).
template <typename T, int TR, int NRG, int CT, int RW, int NW>
__device__ __forceinline__ void xstage_cta(const CUtensorMap &xmap, const XsArgs &a, unsigned cta) {
    using St = Stage<T>;
    extern __shared__ unsigned char smem_raw[];
    Shared sh;
    sh.base = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    sh.full = reinterpret_cast<uint64_t *>(sh.base + a.bar_off);
    sh.empty = sh.full + NS;
    sh.wbar = sh.empty + NS;
    sh.misc = reinterpret_cast<int *>(sh.base + a.misc_off);
    sh.itab = reinterpret_cast<int *>(sh.base + a.blob_off);
    sh.I = reinterpret_cast<int32_t *>(sh.base + a.blob_off + a.hdr);
    sh.W = reinterpret_cast<float *>(sh.base + a.blob_off + a.hdr + a.ib);
    sh.B = reinterpret_cast<float *>(sh.base + a.bias_off);

    ptx::pdl_launch_dependents();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // tile-fastest order: CTAs running at the same time spread over tiles
    const int64_t n_tiles = (a.N + TN - 1) / TN;
    const int task = (int)(cta / n_tiles);
    const int64_t n0 = (int64_t)(cta % n_tiles) * TN;
    const int item_first = task * a.G;
    const int g_count = task < a.n_tasks ? min(a.G, a.n_items - item_first) : 0;
    const int nch = a.nchunks;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NS; s++) {
            ptx::mbar_init(&sh.full[s], 1);
            ptx::mbar_init(&sh.empty[s], NW);
        }
        ptx::mbar_init(sh.wbar, 1);
        sh.misc[0] = 0;
        ptx::fence_barrier_init();
    }
    __syncthreads();   // the barriers exist before any copy or arrive

    if (warp == NW) {
        // ---------------- producer: block values by bulk copy, then X chunks
        if (lane == 0) {
            if (g_count > 0) {   // the task blob, then the X chunks
                ptx::mbar_arrive_expect_tx(sh.wbar, a.stride);
                ptx::bulk_load(sh.itab, a.blob + (int64_t)task * a.stride, a.stride, sh.wbar);
            }
            ptx::prefetch_tensormap(&xmap);
            ptx::pdl_wait();   // X may be an earlier kernel's output
            int c = 0;
            bool ok = true;
            for (; c < nch; c++) {
                const int s = c % NS;
                // the stage is free once every consumer warp released it
                if (c >= NS && !ptx::mbar_wait_bounded(&sh.empty[s], ((c / NS) - 1) & 1, a.wait_ns)) {
                    ok = false;
                    break;
                }
                if (aborted(sh.misc)) { ok = false; break; }
                if (c == a.stall_chunk) continue;   // its consumers time out
                ptx::mbar_arrive_expect_tx(&sh.full[s], St::kBytes);
#pragma unroll
                for (int b = 0; b < St::kBoxes; b++)
                    ptx::tma_load_2d(sh.base + s * St::kBytes + b * St::kBoxBytes, &xmap, c * KC + b * St::kBoxCols,
                                     (int32_t)n0, &sh.full[s]);
            }
            if (!ok) {
                set_status(a.status, DEV_TIMEOUT);
                atomicExch(&sh.misc[0], 1);
            }
            // the last loads issued may still be in flight: wait (bounded) for
            // them so that no TMA write outlives the CTA
            for (int d = max(0, c - NS); d < c; d++)
                if (d != a.stall_chunk) ptx::mbar_wait_bounded(&sh.full[d % NS], (d / NS) & 1, kDrainNs);
            if (g_count > 0) ptx::mbar_wait_bounded(sh.wbar, 0, kDrainNs);
        }
        __syncwarp();
    } else {
        consumer<T, TR, NRG, CT, RW, NW>(a, sh, n0, task, g_count, warp, lane);
    }
}

template <typename T, int TR, int NRG, int CT, int RW, int NW>
__global__ void __launch_bounds__((NW + 1) * 32, 1)
k_xstage(const __grid_constant__ CUtensorMap xmap, const XsArgs a) {
    xstage_cta<T, TR, NRG, CT, RW, NW>(xmap, a, blockIdx.x);
}

// Several products sharing X in one grid: product h owns CTAs
// start[h] .. start[h+1]-1, with its own arguments and shared-memory layout
// (the launch gives every CTA the largest).
struct XsBatch {
    int n;
    unsigned start[kXsBatchMax + 1];
    XsArgs args[kXsBatchMax];
};

template <typename T, int TR, int NRG, int CT, int RW, int NW>
__global__ void __launch_bounds__((NW + 1) * 32, 1)
k_xstage_batch(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ XsBatch b) {
    int h = 0;
    while (h + 1 < b.n && blockIdx.x >= b.start[h + 1]) h++;
    xstage_cta<T, TR, NRG, CT, RW, NW>(xmap, b.args[h], blockIdx.x - b.start[h]);
}

// Block values into the task blobs of every task size: item i's values go to
// blobs + vdst[g * n_items + i] (floats; -1: none), blocks in the records'
// order (perm: position -> stored block), per block W^T widened to fp32
// with WD copies: [(b*C + c)*R + r]*stride + d <- data[(perm[p0_i + b]*R + r)*C + c]
// (stride WD; 1x1 blocks: stride 2 and one copy, the weight beside its X
// offset in the record).
template <typename T>
__global__ void k_pack(const T *__restrict__ data, const Item *__restrict__ items, const int32_t *__restrict__ perm,
                       const int64_t *__restrict__ vdst, int64_t n_items, float *__restrict__ blobs, int R, int C,
                       int stride) {
    for (int64_t gi = blockIdx.x; gi < kXsTaskSizes * n_items; gi += gridDim.x) {
        const int64_t d = vdst[gi];
        if (d < 0) continue;
        const Item it = items[gi % n_items];
        const int64_t total = (int64_t)(it.p1 - it.p0) * R * C;
        float *dst = blobs + d;
        for (int64_t e = threadIdx.x; e < total; e += blockDim.x) {
            const int64_t b = e / ((int64_t)R * C);
            const int rc = (int)(e - b * R * C);
            const int c = rc / R, r = rc - c * R;
            const float w = to_f32(data[((int64_t)perm[it.p0 + b] * R + r) * C + c]);
            const int copies = R == 1 && C == 1 ? 1 : WD;
            for (int k = 0; k < copies; k++) dst[stride * e + k] = w;
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

// The ring, reused after the main loop for the warps' tile slots (one per
// consumer warp, or one per item for one-row blocks, up to four per warp).
size_t region_bytes(bsr_dtype_t dt, int R) {
    const size_t ring = (size_t)NS * (dt == BSR_F32 ? Stage<float>::kBytes : Stage<uint16_t>::kBytes);
    const int nslots = R == 1 ? 4 * kXsConsumerWarpsR1 : NCW;
    const size_t part = (size_t)TN * xstage_slot_pitch(R, nslots) * 4;
    return (std::max(ring, part) + 1023) & ~size_t(1023);
}

// Kernel arguments and dynamic shared-memory bytes of one product at task
// size G (nothing to launch: n_items == 0 or N == 0 leaves smem = 0).
template <int NW>
cudaError_t make_args(const LaunchArgs &la, const XsPlan &pl, int G, XsArgs &a, uint32_t &smem) {
    const Schedule &sc = *la.sc;
    const int gidx = g_index(G);
    const int n_items = (int)sc.items.size();
    smem = 0;
    if (n_items == 0 || la.N == 0) return cudaSuccess;
    if (sc.xs_blob_off[gidx] < 0 || la.data == nullptr) return cudaErrorInvalidConfiguration;
    a.n_items = n_items;
    a.G = G;
    a.S = G <= NW ? NW / G : 1;
    a.n_tasks = (n_items + G - 1) / G;
    a.blob = static_cast<const unsigned char *>(la.data) + sc.xs_blob_off[gidx];
    a.stride = (uint32_t)sc.xs_blob_stride[gidx];
    a.hdr = (uint32_t)(G * kItab * 4);
    a.ib = (uint32_t)((pl.task_ibytes[gidx] + 15) & ~size_t(15));
    a.bias = la.bias;
    a.Y = la.Y;
    a.ws = la.ws;
    a.status = la.status;
    a.N = la.N;
    a.K = sc.K;
    a.M = sc.M;
    a.C = sc.C;
    a.nchunks = (int)((sc.K + KC - 1) / KC);
    a.blob_off = (uint32_t)region_bytes(sc.dt, sc.R);
    a.bias_off = a.blob_off + a.stride;
    a.bar_off = a.bias_off + (uint32_t)(((size_t)G * sc.R * 4 + 15) & ~size_t(15));
    a.misc_off = a.bar_off + (2 * NS + 1) * 8;
    a.wait_ns = la.wait_ns;
    a.stall_chunk = la.stall_chunk;
    smem = a.misc_off + 4 * 4 + 1024;   // + slack to align the base
    return smem > kXsMaxSmem ? cudaErrorInvalidConfiguration : cudaSuccess;
}

// The 2-D tensor map of X [N, K] for the ring's boxes (TN token rows each).
template <typename T>
cudaError_t encode_x(const void *X, int64_t N, int64_t K, CUtensorMap *map) {
    auto enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const size_t es = sizeof(T);
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)N};
    const cuuint64_t strides[1] = {(cuuint64_t)K * es};
    const cuuint32_t box[2] = {(cuuint32_t)Stage<T>::kBoxCols, (cuuint32_t)TN};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, es == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                     const_cast<void *>(X), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Opt a kernel into the large dynamic shared memory once per device.
template <typename K>
cudaError_t allow_smem(K kernel, std::atomic<uint64_t> &done) {
    int dev = 0;
    cudaGetDevice(&dev);
    const uint64_t bit = 1ull << (dev & 63);
    if (done.load() & bit) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kXsMaxSmem);
    if (e == cudaSuccess) done.fetch_or(bit);
    return e;
}

// n products sharing X (same dtype, K, N, block shape and template); n == 1
// is the plain launch, n > 1 one fused grid.
template <typename T, int TR, int NRG, int CT, int RW, int NW>
cudaError_t launch_t(const LaunchArgs *las, const int *Gs, int n, const XsPlan *const *pls) {
    constexpr int NTHREADS = (NW + 1) * 32;
    const int64_t n_tiles = (las[0].N + TN - 1) / TN;
    if (n == 1) {
        const LaunchArgs &la = las[0];
        XsArgs a;
        uint32_t smem = 0;
        cudaError_t e = make_args<NW>(la, *pls[0], Gs[0], a, smem);
        if (e != cudaSuccess || smem == 0) return e;
        static std::atomic<uint64_t> attr_set{0};   // per instantiation, one bit per device
        if ((e = allow_smem(k_xstage<T, TR, NRG, CT, RW, NW>, attr_set)) != cudaSuccess) return e;
        const int64_t grid = n_tiles * a.n_tasks;   // task-major, tile-fastest
        if (grid > INT32_MAX) return cudaErrorInvalidConfiguration;
        CUtensorMap map;
        if ((e = encode_x<T>(la.X, la.N, la.sc->K, &map)) != cudaSuccess) return e;
        return launch_kernel(k_xstage<T, TR, NRG, CT, RW, NW>, dim3((unsigned)grid), dim3(NTHREADS), smem, la.stream,
                             map, a);
    }
    if (n > kXsBatchMax) return cudaErrorInvalidValue;
    XsBatch b;
    b.n = 0;
    uint32_t smem_max = 0;
    int64_t grid = 0;
    for (int i = 0; i < n; i++) {
        uint32_t smem = 0;
        cudaError_t e = make_args<NW>(las[i], *pls[i], Gs[i], b.args[b.n], smem);
        if (e != cudaSuccess) return e;
        if (smem == 0) continue;   // nothing to do for this product
        b.start[b.n] = (unsigned)grid;
        grid += n_tiles * b.args[b.n].n_tasks;
        smem_max = std::max(smem_max, smem);
        b.n++;
    }
    if (b.n == 0) return cudaSuccess;
    if (grid > INT32_MAX) return cudaErrorInvalidConfiguration;
    b.start[b.n] = (unsigned)grid;
    static std::atomic<uint64_t> attr_set_b{0};
    cudaError_t e = allow_smem(k_xstage_batch<T, TR, NRG, CT, RW, NW>, attr_set_b);
    if (e != cudaSuccess) return e;
    CUtensorMap map;
    if ((e = encode_x<T>(las[0].X, las[0].N, las[0].sc->K, &map)) != cudaSuccess) return e;
    return launch_kernel(k_xstage_batch<T, TR, NRG, CT, RW, NW>, dim3((unsigned)grid), dim3(NTHREADS), smem_max,
                         las[0].stream, map, b);
}

// One-row blocks: kXsConsumerWarpsR1 consumer warps (their register tiles
// are small, and more warps hide the shared-memory latency of the one-load-
// per-FMA loop), each owning G/NW items when G exceeds them. Other blocks:
// kXsConsumerWarps, G <= NW.
template <typename T, int TR, int NRG, int CT>
cudaError_t launch_w(const LaunchArgs *las, const int *Gs, int n, const XsPlan *const *pls) {
    const int G = Gs[0];
    if constexpr (TR == 1 && NRG == 1) {
        constexpr int NW = kXsConsumerWarpsR1;
        switch (G > NW ? G / NW : 1) {
            case 1: return G <= NW ? launch_t<T, TR, NRG, CT, 1, NW>(las, Gs, n, pls) : cudaErrorInvalidConfiguration;
            case 2: return launch_t<T, TR, NRG, CT, 2, NW>(las, Gs, n, pls);
            case 4: return launch_t<T, TR, NRG, CT, 4, NW>(las, Gs, n, pls);
        }
        return cudaErrorInvalidConfiguration;
    } else {
        if (G > NCW) return cudaErrorInvalidConfiguration;
        return launch_t<T, TR, NRG, CT, 1, NCW>(las, Gs, n, pls);
    }
}

template <typename T, int TR, int NRG>
cudaError_t launch_c(const LaunchArgs *las, const int *Gs, int n, const XsPlan *const *pls) {
    if (las[0].sc->C == 1) return launch_w<T, TR, NRG, 1>(las, Gs, n, pls);
    return launch_w<T, TR, NRG, 0>(las, Gs, n, pls);
}

template <typename T>
cudaError_t launch_r(const LaunchArgs *las, const int *Gs, int n, const XsPlan *const *pls) {
    switch (las[0].sc->R) {
        case 1: return launch_c<T, 1, 1>(las, Gs, n, pls);
        case 2: return launch_c<T, 2, 1>(las, Gs, n, pls);
        case 4: return launch_c<T, 4, 1>(las, Gs, n, pls);
        case 8: return launch_c<T, 8, 1>(las, Gs, n, pls);
        case 16: return launch_c<T, 8, 2>(las, Gs, n, pls);
        case 32: return launch_c<T, 8, 4>(las, Gs, n, pls);
    }
    return cudaErrorNotSupported;
}

}  // namespace

size_t xstage_smem_bytes(bsr_dtype_t dt, int R, int64_t K, int G, size_t wbytes, size_t ibytes) {
    (void)K;
    return region_bytes(dt, R) + (size_t)G * kItab * 4 + ((wbytes + 15) & ~size_t(15)) +
           ((ibytes + 15) & ~size_t(15)) + (((size_t)G * R * 4 + 15) & ~size_t(15)) + (2 * NS + 1) * 8 + 4 * 4 + 1024;
}

size_t xstage_task_budget(bsr_dtype_t dt, int R, int64_t K) {
    const size_t fixed = xstage_smem_bytes(dt, R, K, NCW, 0, 0) + 64;
    return fixed >= (size_t)kXsMaxSmem ? 0 : (size_t)kXsMaxSmem - fixed;
}

uint32_t xstage_stage_offset(bsr_dtype_t dt, int kk) {
    return dt == BSR_F32 ? Stage<float>::off0(kk) : Stage<uint16_t>::off0(kk);
}

int g_index(int G) {
    for (int i = 0; i < kXsTaskSizes; i++)
        if (kXsG[i] == G) return i;
    return 0;
}

bool xstage_task_size_ok(int R, int G) {
    return R == 1 ? (G <= kXsConsumerWarpsR1 ? kXsConsumerWarpsR1 % G == 0 : (G == 2 * kXsConsumerWarpsR1 || G == 4 * kXsConsumerWarpsR1))
                  : G <= kXsConsumerWarps;
}

bool xstage_supports(int R, int C, bsr_dtype_t dt, int64_t K) {
    const bool r_ok = R == 1 || R == 2 || R == 4 || R == 8 || R == 16 || R == 32;
    const bool c_ok = C >= 1 && C <= kXsChunk && kXsChunk % C == 0;
    const int64_t align = dt == BSR_F32 ? 4 : 8;   // TMA row pitch must be a multiple of 16 bytes
    return r_ok && c_ok && K % align == 0 && K > 0;
}

cudaError_t pack_xstage_data(const void *data, bsr_dtype_t dt, const Item *items, const int32_t *perm,
                             const int64_t *vdst, int64_t n_items, int R, int C, float *blobs, cudaStream_t s) {
    if (n_items == 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>(kXsTaskSizes * n_items, 1 << 16);
    const int stride = xstage_block_ints(R, C) == 2 ? 2 : WD;
    if (dt == BSR_F32)
        k_pack<float><<<grid, 256, 0, s>>>((const float *)data, items, perm, vdst, n_items, blobs, R, C, stride);
    else
        k_pack<uint16_t><<<grid, 256, 0, s>>>((const uint16_t *)data, items, perm, vdst, n_items, blobs, R, C, stride);
    return cudaGetLastError();
}

cudaError_t launch_xstage(const LaunchArgs &la, int G) {
    const XsPlan *pl = &la.sc->xs;
    if (la.sc->dt == BSR_F32) return launch_r<float>(&la, &G, 1, &pl);
    return launch_r<uint16_t>(&la, &G, 1, &pl);
}

int xstage_fusion_key(const Schedule &sc, int G) {
    const int rw = sc.R == 1 && G > kXsConsumerWarpsR1 ? G / kXsConsumerWarpsR1 : 1;
    return (((int)sc.dt * 64 + sc.R) * 2 + (sc.C == 1 ? 1 : 0)) * 8 + rw;
}

cudaError_t launch_xstage_batch(const LaunchArgs *las, const int *Gs, int n) {
    if (n <= 0) return cudaSuccess;
    if (n > kXsBatchMax) return cudaErrorInvalidValue;
    const XsPlan *pls[kXsBatchMax];
    for (int i = 0; i < n; i++) pls[i] = &las[i].sc->xs;
    if (las[0].sc->dt == BSR_F32) return launch_r<float>(las, Gs, n, pls);
    return launch_r<uint16_t>(las, Gs, n, pls);
}

}  // namespace bsr
