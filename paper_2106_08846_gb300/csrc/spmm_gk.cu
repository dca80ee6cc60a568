// Gathered-K tensor-core BSR x dense kernel ("gk"). A block row of R x C
// blocks is a dense [R x (kept blocks x C)] matrix over the X columns its
// blocks touch (Section 2.2's kept blocks, side by side): the kernel gathers
// exactly those columns of X into the MMA's A operand in tensor memory, so
// one-column blocks (the paper's best shape, 32x1) run on the tensor cores
// with no zero padding between blocks. fp32 runs as 3xTF32 (each operand
// split into a tf32 high part and the remainder; high x high + high x low +
// low x high), bf16 as one bf16 MMA, both accumulating in fp32.
//
// Persistent: one CTA per SM walks a contiguous range of units (task, tile
// of 128 tokens -- the MMA's M and the tensor-memory lanes), tasks in the
// outer order; a task is at most G block rows (items; G R fp32 accumulator
// columns), and X is read once per task, so tasks are as large as tensor
// memory allows:
//
//   warp 0 (one thread)  producer: per task its record (two buffers), then
//                         for every unit the K chunks that hold any of the
//                         task's blocks: the X chunk [128 tokens x 256 bytes]
//                         by 2-D TMA (128-byte swizzle) and, beside it, the
//                         chunk's packed block values (the MMA's B operands,
//                         one per item, over that item's gathered K,
//                         zero-padded to the MMA's K), through a ring of
//                         stages that keeps streaming across units.
//   warps 1..4 (lane 0)  issue the MMAs (warp 1 also owns the tensor
//                         memory): one thread issues an MMA no faster than
//                         every 40-100 ns, so four issuers each run the
//                         MMAs of a contiguous, work-balanced range of the
//                         task's items, from a program built at create time
//                         and loaded beside each chunk's block values (one
//                         16-byte word per MMA: no decoding between MMAs).
//                         Per batch of entries (pieces of a chunk's items,
//                         as many as fill one of up to eight A buffers, so
//                         the gather runs several batches ahead of the MMAs'
//                         completion) and K slice: M = 128, N = R, K = 8
//                         (tf32; three per slice) or 16 (bf16), A from
//                         tensor memory, B from shared memory; commits free
//                         the A buffer, the stage and, per unit, hand the
//                         accumulators to the epilogue.
//   warps 5..12          gather, two groups of four warps (one per 32 lanes)
//                         taking alternate batches, so two batches are in
//                         flight: thread t (token t, tensor-memory lane t) reads its
//                         token's values of each entry's kept columns from
//                         the stage, splits fp32 into tf32 high and low parts,
//                         and stores them with tcgen05.st into the batch's A
//                         buffer (zeros pad each entry's K).
//   warps 13..16         epilogue: each reads its 32 lanes of the
//                         accumulators, adds the bias, turns the tile around
//                         through shared memory and stores whole row segments
//                         of Y, then frees the accumulators for the next unit
//                         (the gather runs ahead meanwhile).
//
// Launched with programmatic stream serialisation. Every wait is bounded by
// the global timer; a timeout sets the device status word, stops issuing,
// lets the issued copies and MMAs finish, frees the tensor memory and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "bsr_internal.h"
#include "elem.cuh"
#include "gk.h"
#include "launch.cuh"
#include "ptx.cuh"
#include "tcgen05.cuh"

namespace bsr {

namespace {

constexpr int TN = kGkTokens;
constexpr int NS_MAX = kGkStages;
constexpr int NA_MAX = kGkASlotsMax;
constexpr int NISS = kGkIssuers;       // MMA-issuing warps (lane 0 of each)
constexpr int NGW = 8;                 // gather warps: two groups of one warp per tensor-memory lane quarter
constexpr int NEW = 4;                 // epilogue warps: one per lane quarter
constexpr int NWARPS = 1 + NISS + NGW + NEW;
constexpr int NTHREADS = NWARPS * 32;
constexpr uint32_t kStageBytes = TN * 256;   // two 128-byte-row boxes of 128 tokens
constexpr uint64_t kDrainNs = 200000000ull;
constexpr int EI = kGkEntryInts;

struct GkArgs {
    int G, n_tasks, ns, na;       // ns: ring stages; na: A buffers
    const int32_t *rec;       // task records
    const int32_t *rec_off;   // per task: record offset (ints)
    const unsigned char *wpk; // packed block values of this task size
    const uint4 *prog;        // chunk MMA programs of this task size
    uint32_t wstage, wslot;   // bytes of a chunk's values (most), of one W stage (values + program)
    uint32_t acols;           // tensor-memory columns of one A buffer
    const float *bias;
    void *Y;
    int *status;
    int64_t N, K, M;
    int C, nchunks;
    uint32_t w_off, rec_smem, rec_bytes, bias_off, stg_off, bar_off, misc_off;   // rec_bytes: one record buffer
    uint64_t wait_ns;
    int stall_chunk;              // test hook: this chunk of each CTA's first unit is never loaded (-1: none)
};

__device__ __forceinline__ void set_status(int *status, int code) { atomicCAS(status, DEV_OK, code); }
__device__ __forceinline__ bool aborted(const int *flag) { return *reinterpret_cast<const volatile int *>(flag) != 0; }
__device__ __forceinline__ int pad4(int n) { return (n + 3) & ~3; }

__device__ __forceinline__ float lds_f32(uint32_t a) {
    float v;
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ float2 lds_f32x2(uint32_t a) {
    float2 v;
    asm volatile("ld.shared.v2.f32 {%0,%1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds_u16(uint32_t a) {
    unsigned short v;
    asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds_u32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint4 lds_128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}

// Gather one entry (m blocks of C = 2^lc columns, K padded to kpad) of this
// thread's token into tensor memory at column `col` (fp32: high parts at
// col, low parts at col + kpad; bf16: pairs). `row` is the stage address of
// the token's row and `sw` its 128-byte swizzle ((row % 8) << 4: 16-byte
// group g of the row sits at g ^ (row % 8)); `cl` lists each block's
// first-column offset in the stage (row 0, unswizzled). Groups of 8 K
// positions (fp32) or 16 (bf16), one tcgen05.st of 8 columns each.
template <bool F32>
__device__ __forceinline__ void gather_entry(uint32_t row, uint32_t sw, const int32_t *cl, int m, int lc, int kpad,
                                            uint32_t col) {
    const int K = m << lc;
    if constexpr (F32) {
        for (int k0 = 0; k0 < kpad; k0 += 8) {
            float v[8];
            if (lc == 0) {   // one column per block
#pragma unroll
                for (int i = 0; i < 8; i++) v[i] = k0 + i < m ? lds_f32(row + ((uint32_t)cl[k0 + i] ^ sw)) : 0.f;
            } else if (lc == 1) {   // two adjacent columns (8 bytes) per block
#pragma unroll
                for (int i = 0; i < 4; i++) {
                    const int b = (k0 >> 1) + i;
                    const float2 p = b < m ? lds_f32x2(row + ((uint32_t)cl[b] ^ sw)) : make_float2(0.f, 0.f);
                    v[2 * i] = p.x;
                    v[2 * i + 1] = p.y;
                }
            } else if (lc == 2) {   // four columns (16 bytes) per block
#pragma unroll
                for (int h = 0; h < 2; h++) {
                    const int b = (k0 >> 2) + h;
                    const uint4 a = b < m ? lds_128(row + ((uint32_t)cl[b] ^ sw)) : make_uint4(0u, 0u, 0u, 0u);
                    v[4 * h] = __uint_as_float(a.x), v[4 * h + 1] = __uint_as_float(a.y);
                    v[4 * h + 2] = __uint_as_float(a.z), v[4 * h + 3] = __uint_as_float(a.w);
                }
            } else if (k0 < K) {   // 8 or more columns: two 16-byte groups of one block
                const uint32_t off = (uint32_t)cl[k0 >> lc] + ((uint32_t)(k0 & ((1 << lc) - 1)) << 2);
                const uint4 a = lds_128(row + (off ^ sw)), c = lds_128(row + ((off + 16u) ^ sw));
                v[0] = __uint_as_float(a.x), v[1] = __uint_as_float(a.y), v[2] = __uint_as_float(a.z),
                v[3] = __uint_as_float(a.w);
                v[4] = __uint_as_float(c.x), v[5] = __uint_as_float(c.y), v[6] = __uint_as_float(c.z),
                v[7] = __uint_as_float(c.w);
            } else {
#pragma unroll
                for (int i = 0; i < 8; i++) v[i] = 0.f;
            }
            uint32_t hi[8], lo[8];
#pragma unroll
            for (int i = 0; i < 8; i++) {
                const float h = __uint_as_float(__float_as_uint(v[i]) & 0xffffe000u);
                hi[i] = __float_as_uint(h);
                lo[i] = __float_as_uint(v[i] - h);
            }
            tc5::st8(col + (uint32_t)k0, hi);
            tc5::st8(col + (uint32_t)(kpad + k0), lo);
        }
    } else {
        for (int k0 = 0; k0 < kpad; k0 += 16) {
            uint32_t p[8];
            if (lc == 0) {   // one bf16 per block: pairs of blocks per column
#pragma unroll
                for (int i = 0; i < 8; i++) {
                    const int b = k0 + 2 * i;
                    const uint32_t e0 = b < m ? lds_u16(row + ((uint32_t)cl[b] ^ sw)) : 0u;
                    const uint32_t e1 = b + 1 < m ? lds_u16(row + ((uint32_t)cl[b + 1] ^ sw)) : 0u;
                    p[i] = e0 | (e1 << 16);
                }
            } else if (lc == 1) {   // two adjacent bf16 (4 bytes) per block
#pragma unroll
                for (int i = 0; i < 8; i++) {
                    const int b = (k0 >> 1) + i;
                    p[i] = b < m ? lds_u32(row + ((uint32_t)cl[b] ^ sw)) : 0u;
                }
            } else if (lc == 2) {   // four bf16 (8 bytes) per block
#pragma unroll
                for (int h = 0; h < 4; h++) {
                    const int b = (k0 >> 2) + h;
                    if (b < m) {
                        const uint32_t a = row + ((uint32_t)cl[b] ^ sw);
                        p[2 * h] = lds_u32(a);
                        p[2 * h + 1] = lds_u32(a + 4u);
                    } else {
                        p[2 * h] = p[2 * h + 1] = 0u;
                    }
                }
            } else {   // 8 or more bf16 (16 bytes) per load
#pragma unroll
                for (int h = 0; h < 2; h++) {
                    const int k = k0 + 8 * h;
                    if (k < K) {
                        const uint32_t off = (uint32_t)cl[k >> lc] + ((uint32_t)(k & ((1 << lc) - 1)) << 1);
                        const uint4 a = lds_128(row + (off ^ sw));
                        p[4 * h] = a.x, p[4 * h + 1] = a.y, p[4 * h + 2] = a.z, p[4 * h + 3] = a.w;
                    } else {
                        p[4 * h] = p[4 * h + 1] = p[4 * h + 2] = p[4 * h + 3] = 0u;
                    }
                }
            }
            tc5::st8(col + (uint32_t)(k0 / 2), p);
        }
    }
}

template <typename T, int R>
__global__ void __launch_bounds__(NTHREADS, 1)
k_gk(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ GkArgs a) {
    ptx::pdl_launch_dependents();
    constexpr bool F32 = sizeof(T) == 4;
    constexpr int KS = F32 ? 8 : 16;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *base =
        reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(base + a.bar_off);
    uint64_t *empty = full + NS_MAX;   // the gather warps + every issuer's MMA commit
    uint64_t *afull = empty + NS_MAX;  // A buffer written (one gather group)
    uint64_t *aempty = afull + NA_MAX; // A buffer consumed (MMA commit)
    uint64_t *accf = aempty + NA_MAX;  // a unit's MMAs completed (MMA commit)
    uint64_t *acce = accf + 1;         // the epilogue read the accumulators (epilogue warps)
    uint64_t *rbar = acce + 1;         // [2] record landed
    uint64_t *rfree = rbar + 2;        // [2] record no longer used (issuer, gather and epilogue warps)
    uint64_t *done = rfree + 2;        // every MMA issued completed
    int *misc = reinterpret_cast<int *>(base + a.misc_off);   // [0] abort flag, [1] tensor-memory address
    unsigned char *W_s = base + a.w_off;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ns = a.ns, na = a.na, nch = a.nchunks;
    const int64_t n_tiles = (a.N + TN - 1) / TN;
    const int64_t units = n_tiles * a.n_tasks, P = gridDim.x;
    const int64_t ub = units * (int64_t)blockIdx.x / P, ue = units * ((int64_t)blockIdx.x + 1) / P;
    const int cb_at = 4, cw_at = 4 + pad4(nch + 1), cp_at = cw_at + pad4(nch + 1), be_at = cp_at + pad4(2 * nch);
    auto rec_s = [&](int j) { return reinterpret_cast<int32_t *>(base + a.rec_smem + (j & 1) * a.rec_bytes); };
    auto bias_s = [&](int j) { return reinterpret_cast<float *>(base + a.bias_off) + (j & 1) * a.G * R; };
    auto last_of_task = [&](int64_t u) { return u + 1 == ue || (u + 1) / n_tiles != u / n_tiles; };

    if (threadIdx.x == 0) {
        for (int s = 0; s < NS_MAX; s++) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], NGW + NISS);
        }
        for (int s = 0; s < NA_MAX; s++) {
            ptx::mbar_init(&afull[s], 4);
            ptx::mbar_init(&aempty[s], NISS);
        }
        ptx::mbar_init(accf, NISS);
        ptx::mbar_init(acce, NEW);
        for (int r = 0; r < 2; r++) {
            ptx::mbar_init(&rbar[r], 1);
            ptx::mbar_init(&rfree[r], NISS + NGW + NEW);
        }
        ptx::mbar_init(done, NISS);
        misc[0] = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 1) tc5::alloc(reinterpret_cast<uint32_t *>(&misc[1]), kGkTmemCols);
    tc5::fence_before();
    __syncthreads();
    tc5::fence_after();
    const uint32_t tmem = (uint32_t)misc[1];
    const uint32_t abase = tmem + (uint32_t)(a.G * R);   // A buffers after the accumulators

    if (warp == 0) {
        // ---------------- producer
        int j = 0;   // record loads issued - 1
        if (lane == 0 && ub < ue) {
            ptx::prefetch_tensormap(&xmap);
            int64_t task = ub / n_tiles;
            const int32_t *grec = a.rec + __ldg(a.rec_off + task);
            ptx::mbar_arrive_expect_tx(&rbar[0], (uint32_t)__ldg(grec + 3));
            ptx::bulk_load(rec_s(0), grec, (uint32_t)__ldg(grec + 3), &rbar[0]);
            ptx::pdl_wait();   // X may be an earlier kernel's output
            bool ok = ptx::mbar_wait_bounded(&rbar[0], 0, a.wait_ns);
            int64_t k = 0, stalled = -1;
            for (int64_t u = ub; ok && u < ue; u++) {
                if (u / n_tiles != task) {
                    task = u / n_tiles;
                    j++;
                    if (j >= 2 && !ptx::mbar_wait_bounded(&rfree[j & 1], ((j >> 1) - 1) & 1, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    grec = a.rec + __ldg(a.rec_off + task);
                    ptx::mbar_arrive_expect_tx(&rbar[j & 1], (uint32_t)__ldg(grec + 3));
                    ptx::bulk_load(rec_s(j), grec, (uint32_t)__ldg(grec + 3), &rbar[j & 1]);
                    if (!ptx::mbar_wait_bounded(&rbar[j & 1], (j >> 1) & 1, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                }
                const int32_t *I = rec_s(j);
                const int64_t wfirst = (int64_t)I[2] * 16;
                const int32_t n0 = (int32_t)((u % n_tiles) * TN);
                for (int c = 0; c < nch; c++) {
                    if (I[cb_at + c] == I[cb_at + c + 1]) continue;   // no block of this task in chunk c
                    const int s = (int)(k % ns);
                    if (k >= ns && !ptx::mbar_wait_bounded(&empty[s], (uint32_t)((k / ns) - 1) & 1, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    if (aborted(misc)) { ok = false; break; }
                    if (u == ub && c == a.stall_chunk) {   // never loaded: its consumers time out
                        stalled = k++;
                        continue;
                    }
                    // the X chunk, the chunk's block values and, after them, its MMA program
                    const uint32_t w0 = (uint32_t)I[cw_at + c] * 16u, wbytes = (uint32_t)I[cw_at + c + 1] * 16u - w0;
                    const uint32_t pbytes = (uint32_t)I[cp_at + 2 * c + 1];
                    constexpr int KC = F32 ? 64 : 128, BOXC = F32 ? 32 : 64;
                    ptx::mbar_arrive_expect_tx(&full[s], kStageBytes + wbytes + pbytes);
                    ptx::tma_load_2d(base + s * kStageBytes, &xmap, c * KC, n0, &full[s]);
                    ptx::tma_load_2d(base + s * kStageBytes + kStageBytes / 2, &xmap, c * KC + BOXC, n0, &full[s]);
                    ptx::bulk_load(W_s + s * a.wslot, a.wpk + wfirst + w0, wbytes, &full[s]);
                    ptx::bulk_load(W_s + s * a.wslot + a.wstage, a.prog + I[cp_at + 2 * c], pbytes, &full[s]);
                    k++;
                }
            }
            if (!ok) {
                set_status(a.status, DEV_TIMEOUT);
                atomicExch(&misc[0], 1);
            }
            // copies still in flight land before the CTA exits
            for (int64_t d = k > ns ? k - ns : 0; d < k; d++)
                if (d != stalled) ptx::mbar_wait_bounded(&full[d % ns], (uint32_t)(d / ns) & 1, kDrainNs);
            ptx::mbar_wait_bounded(&rbar[j & 1], (j >> 1) & 1, kDrainNs);
        }
    } else if (warp <= NISS) {
        // ---------------- MMA issuers: lane 0 of warps 1..NISS, each running
        // its part of every batch's program (its items' MMAs), one word per MMA
        if (lane == 0) {
            const int q = warp - 1;
            bool ok = true;
            int j = -1;
            int64_t task = -1, k = 0, kb = 0, ui = 0;
            for (int64_t u = ub; ok && u < ue; u++, ui++) {
                if (u / n_tiles != task) {
                    task = u / n_tiles;
                    j++;
                    if (!ptx::mbar_wait_bounded(&rbar[j & 1], (j >> 1) & 1, a.wait_ns)) { ok = false; break; }
                }
                const int32_t *I = rec_s(j);
                // the epilogue has read the previous unit's accumulators
                if (ui > 0 && !ptx::mbar_wait_bounded(acce, (uint32_t)(ui - 1) & 1, a.wait_ns)) { ok = false; break; }
                tc5::fence_after();
                for (int c = 0; ok && c < nch; c++) {
                    const int b0 = I[cb_at + c], b1 = I[cb_at + c + 1];
                    if (b0 == b1) continue;
                    const int s = (int)(k % ns);
                    if (!ptx::mbar_wait_bounded(&full[s], (uint32_t)(k / ns) & 1, a.wait_ns) || aborted(misc)) {
                        ok = false;
                        break;
                    }
                    const unsigned char *slot = W_s + s * a.wslot;
                    const uint64_t bd0 = tc5::desc(ptx::smem_addr(slot), 128, 256);
                    const int32_t *hdr = reinterpret_cast<const int32_t *>(slot + a.wstage);
                    const uint4 *pw = reinterpret_cast<const uint4 *>(hdr + pad4((b1 - b0) * NISS + 1));
                    for (int b = b0; b < b1; b++) {
                        const int sl = (int)(kb % na);
                        if (!ptx::mbar_wait_bounded(&afull[sl], (uint32_t)(kb / na) & 1, a.wait_ns) || aborted(misc)) {
                            ok = false;
                            break;
                        }
                        tc5::fence_after();
                        const uint32_t ab = abase + (uint32_t)sl * a.acols;
                        const int i1 = hdr[(b - b0) * NISS + q + 1];
                        int i = hdr[(b - b0) * NISS + q];
                        for (; i + 2 <= i1; i += 2) {   // two words loaded ahead of their MMAs
                            const uint4 w0 = pw[i], w1 = pw[i + 1];
                            tc5::mma_ts<F32>(tmem + w0.y, ab + (w0.z & 0x7fffffffu), bd0 + w0.x, w0.w, w0.z >> 31);
                            tc5::mma_ts<F32>(tmem + w1.y, ab + (w1.z & 0x7fffffffu), bd0 + w1.x, w1.w, w1.z >> 31);
                        }
                        if (i < i1) {
                            const uint4 w0 = pw[i];
                            tc5::mma_ts<F32>(tmem + w0.y, ab + (w0.z & 0x7fffffffu), bd0 + w0.x, w0.w, w0.z >> 31);
                        }
                        tc5::commit(&aempty[sl]);   // the A buffer is free once every issuer's MMAs completed
                        kb++;
                    }
                    if (!ok) break;
                    tc5::commit(&empty[s]);   // and so are the stage's block values
                    k++;
                }
                if (!ok) break;
                tc5::commit(accf);   // the unit's accumulators are complete
                if (last_of_task(u)) ptx::mbar_arrive(&rfree[j & 1]);
            }
            if (!ok) {
                set_status(a.status, DEV_TIMEOUT);
                atomicExch(&misc[0], 1);
            }
            tc5::commit(done);   // every MMA this issuer issued completes before its arrival
            // the tensor memory is freed below: one thread waits for every issuer's MMAs
            if (warp == 1 && !ptx::mbar_wait_bounded(done, 0, kDrainNs)) set_status(a.status, DEV_TIMEOUT);
        }
    } else if (warp <= NISS + NGW) {
        // ---------------- gather; lane quarter = warp % 4, group (the first
        // or the second four gather warps) takes the batches of its parity
        const int q = warp & 3, grp = (warp - 1 - NISS) >> 2;
        const int t = 32 * q + lane;   // token row in the tile = tensor-memory lane
        const uint32_t sw = (uint32_t)(t & 7) << 4;
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        int lc = 0;
        while ((1 << lc) < a.C) lc++;
        bool ok = true;
        int j = -1;
        int64_t task = -1, k = 0, kb = 0;
        for (int64_t u = ub; ok && u < ue; u++) {
            if (u / n_tiles != task) {
                task = u / n_tiles;
                j++;
                const bool got = ptx::mbar_wait_bounded(&rbar[j & 1], (j >> 1) & 1, a.wait_ns);
                if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
            }
            const int32_t *I = rec_s(j);
            const int32_t *ent = I + be_at + pad4(I[1] + 1) + 4 * I[0];
            for (int c = 0; ok && c < nch; c++) {
                const int b0 = I[cb_at + c], b1 = I[cb_at + c + 1];
                if (b0 == b1) continue;
                const int s = (int)(k % ns);
                const bool got = ptx::mbar_wait_bounded(&full[s], (uint32_t)(k / ns) & 1, a.wait_ns) && !aborted(misc);
                if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
                const uint32_t row = ptx::smem_addr(base + s * kStageBytes) + (uint32_t)t * 128u;
                for (int b = b0; b < b1; b++, kb++) {
                    if ((int)(kb & 1) != grp) continue;   // the other group's batch
                    const int sl = (int)(kb % na);
                    bool free = true;
                    if (kb >= na) free = ptx::mbar_wait_bounded(&aempty[sl], (uint32_t)((kb / na) - 1) & 1, a.wait_ns);
                    if (!__all_sync(0xffffffffu, free && !aborted(misc))) { ok = false; break; }
                    tc5::fence_after();
                    const uint32_t ab = abase + (uint32_t)sl * a.acols + lane_off;
                    for (int e = I[be_at + b]; e < I[be_at + b + 1]; e++) {
                        const int32_t *en = ent + EI * e;
                        gather_entry<F32>(row, sw, I + en[6], en[5], lc, en[3] * KS, ab + (uint32_t)en[2]);
                    }
                    tc5::st_wait();
                    tc5::fence_before();
                    __syncwarp();
                    if (lane == 0) ptx::mbar_arrive(&afull[sl]);
                }
                if (!ok) break;
                if (lane == 0) ptx::mbar_arrive(&empty[s]);   // this warp no longer reads the X chunk
                k++;
            }
            if (ok && lane == 0 && last_of_task(u)) ptx::mbar_arrive(&rfree[j & 1]);
        }
        if (!ok && lane == 0) {
            set_status(a.status, DEV_TIMEOUT);
            atomicExch(&misc[0], 1);
        }
    } else {
        // ---------------- epilogue; lane quarter = warp % 4
        const int q = warp & 3;
        const int et = threadIdx.x - 32 * (1 + NISS + NGW);   // 0..127
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        ptx::pdl_wait();   // the bias and Y may be an earlier kernel's
        bool ok = true;
        int j = -1;
        int64_t task = -1, ui = 0;
        for (int64_t u = ub; ok && u < ue; u++, ui++) {
            if (u / n_tiles != task) {
                task = u / n_tiles;
                j++;
                const bool got = ptx::mbar_wait_bounded(&rbar[j & 1], (j >> 1) & 1, a.wait_ns) && !aborted(misc);
                if (ptx::named_barrier_or(2, 32 * NEW, !got)) { ok = false; break; }
                const int32_t *I = rec_s(j);
                float *B = bias_s(j);
                for (int e = et; e < I[0] * R; e += 32 * NEW) {
                    const int g = e / R, r = e - g * R;
                    B[e] = a.bias ? __ldg(a.bias + (int64_t)I[be_at + pad4(I[1] + 1) + 4 * g] * R + r) : 0.f;
                }
                ptx::named_barrier(2, 32 * NEW);
            }
            const int32_t *I = rec_s(j);
            const int32_t *items = I + be_at + pad4(I[1] + 1);
            const float *B = bias_s(j);
            const uint64_t limit = a.wait_ns * (uint64_t)(nch + 2);
            const bool got = ptx::mbar_wait_bounded(accf, (uint32_t)ui & 1, limit) && !aborted(misc);
            if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
            tc5::fence_after();
            // per item and 32-column group: each lane's row of the tile into
            // this warp's staging tile (16-byte groups XOR-swizzled by row), then
            // lanes re-read it as (row, 8-column group) pairs and store whole row
            // segments: 8 rows x 4 groups per instruction
            float *stg = reinterpret_cast<float *>(base + a.stg_off) + (warp - 1 - NISS - NGW) * 32 * 32;
            const uint32_t stg_row = ptx::smem_addr(stg) + (uint32_t)lane * 128u;
            const int64_t row0 = (u % n_tiles) * TN + 32 * q;   // the warp's first token
            for (int g = 0; g < I[0]; g++) {
                const int row = items[4 * g], len = items[4 * g + 1];
#pragma unroll
                for (int c0 = 0; c0 < R; c0 += 32) {
                    constexpr int W = R >= 32 ? 32 : R;
                    uint32_t r[32];
                    if constexpr (W == 32) {
                        tc5::ld32(tmem + lane_off + (uint32_t)(g * R + c0), r);
                    } else {
                        uint32_t r16[16];
                        tc5::ld16(tmem + lane_off + (uint32_t)(g * R + c0), r16);
#pragma unroll
                        for (int i = 0; i < 16; i++) r[i] = r16[i];
                    }
                    tc5::ld_wait();
                    const float *bs = B + g * R + c0;
#pragma unroll
                    for (int c4 = 0; c4 < W / 4; c4++) {
                        float4 o;
                        o.x = (len > 0 ? __uint_as_float(r[4 * c4]) : 0.f) + bs[4 * c4];
                        o.y = (len > 0 ? __uint_as_float(r[4 * c4 + 1]) : 0.f) + bs[4 * c4 + 1];
                        o.z = (len > 0 ? __uint_as_float(r[4 * c4 + 2]) : 0.f) + bs[4 * c4 + 2];
                        o.w = (len > 0 ? __uint_as_float(r[4 * c4 + 3]) : 0.f) + bs[4 * c4 + 3];
                        asm volatile("st.shared.v4.f32 [%0], {%1,%2,%3,%4};" ::"r"(stg_row + ((c4 ^ (lane & 7)) << 4)),
                                     "f"(o.x), "f"(o.y), "f"(o.z), "f"(o.w)
                                     : "memory");
                    }
                    __syncwarp();
                    constexpr int GPR = W / 8;             // 8-column groups per row
                    constexpr int RPI = 32 / GPR;          // rows per instruction
                    const int rr = lane / GPR, gg = lane % GPR;
#pragma unroll
                    for (int p0 = 0; p0 < 32; p0 += RPI) {
                        const int rw = p0 + rr;            // row of the warp's 32
                        const int64_t n = row0 + rw;
                        const uint32_t src = ptx::smem_addr(stg) + (uint32_t)rw * 128u;
                        float4 lo4, hi4;
                        asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                                     : "=f"(lo4.x), "=f"(lo4.y), "=f"(lo4.z), "=f"(lo4.w)
                                     : "r"(src + (uint32_t)(((2 * gg) ^ (rw & 7)) << 4)));
                        asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                                     : "=f"(hi4.x), "=f"(hi4.y), "=f"(hi4.z), "=f"(hi4.w)
                                     : "r"(src + (uint32_t)(((2 * gg + 1) ^ (rw & 7)) << 4)));
                        if (n >= a.N) continue;
                        T *dst = reinterpret_cast<T *>(a.Y) + n * a.M + (int64_t)row * R + c0 + 8 * gg;
                        if constexpr (F32) {
                            reinterpret_cast<float4 *>(dst)[0] = lo4;
                            reinterpret_cast<float4 *>(dst)[1] = hi4;
                        } else {
                            uint4 pk;
                            pk.x = (uint32_t)from_f32<uint16_t>(lo4.x) | ((uint32_t)from_f32<uint16_t>(lo4.y) << 16);
                            pk.y = (uint32_t)from_f32<uint16_t>(lo4.z) | ((uint32_t)from_f32<uint16_t>(lo4.w) << 16);
                            pk.z = (uint32_t)from_f32<uint16_t>(hi4.x) | ((uint32_t)from_f32<uint16_t>(hi4.y) << 16);
                            pk.w = (uint32_t)from_f32<uint16_t>(hi4.z) | ((uint32_t)from_f32<uint16_t>(hi4.w) << 16);
                            *reinterpret_cast<uint4 *>(dst) = pk;
                        }
                    }
                    __syncwarp();   // the staging tile is free again
                }
            }
            tc5::fence_before();
            __syncwarp();
            if (lane == 0) {
                ptx::mbar_arrive(acce);   // the accumulators may be overwritten
                if (last_of_task(u)) ptx::mbar_arrive(&rfree[j & 1]);
            }
        }
        if (!ok && lane == 0) {
            set_status(a.status, DEV_TIMEOUT);
            atomicExch(&misc[0], 1);
        }
    }
    // ---------------- teardown: every MMA issued completed (the issuer waited
    // for them), then free the tensor memory
    tc5::fence_before();
    __syncthreads();
    if (warp == 1) {
        tc5::fence_after();
        tc5::dealloc(tmem, kGkTmemCols);
    }
}

// Block values into the gathered B operands: packed slot p holds stored block
// wsrc[p]; its entry's operand starts at byte wbase[p] of `out`, its first
// column is K row (wslot[p] & 0xffff) of an operand of K = wslot[p] >> 16 rows
// (padded), element (r, c) of the block at K row k = first + c, N row r, in
// the K-major core-matrix layout (8 N rows x 16 bytes; 128 bytes apart along K
// and 256 apart along N within a K slice); fp32 as tf32 high part then low
// part (K R floats later).
template <typename T>
__global__ void k_pack_gk(const T *__restrict__ data, const int32_t *__restrict__ wsrc,
                          const int32_t *__restrict__ wslot, const int64_t *__restrict__ wbase, int64_t n, int R,
                          int C, unsigned char *__restrict__ out) {
    const int64_t total = n * R * C;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = e / ((int64_t)R * C);
        const int rc = (int)(e - p * R * C);
        const int r = rc / C, c = rc - r * C;
        const int src = wsrc[p];
        if (src < 0) continue;
        const int k = (wslot[p] & 0xffff) + c, kpad = wslot[p] >> 16;
        const T v = data[(int64_t)src * R * C + rc];
        if constexpr (sizeof(T) == 4) {
            float *o = reinterpret_cast<float *>(out + wbase[p]);
            const int64_t at = (k >> 3) * (R * 8) + (r >> 3) * 64 + ((k & 7) >> 2) * 32 + (r & 7) * 4 + (k & 3);
            const float w = v, h = __uint_as_float(__float_as_uint(w) & 0xffffe000u);
            o[at] = h;
            o[at + (int64_t)kpad * R] = w - h;
        } else {
            T *o = reinterpret_cast<T *>(out + wbase[p]);
            o[(k >> 4) * (R * 16) + (r >> 3) * 128 + ((k & 15) >> 3) * 64 + (r & 7) * 8 + (k & 7)] = v;
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

template <typename T>
cudaError_t encode_x(const void *X, int64_t N, int64_t K, CUtensorMap *map) {
    auto enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)N};
    const cuuint64_t strides[1] = {(cuuint64_t)K * sizeof(T)};
    const cuuint32_t box[2] = {(cuuint32_t)(128 / sizeof(T)), (cuuint32_t)TN};
    const cuuint32_t estr[2] = {1, 1};
    if (enc(map, sizeof(T) == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
            const_cast<void *>(X), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) !=
        CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    return cudaSuccess;
}

template <typename K>
cudaError_t allow_smem(K kernel, std::atomic<uint64_t> &done) {
    int dev = 0;
    cudaGetDevice(&dev);
    const uint64_t bit = 1ull << (dev & 63);
    if (done.load() & bit) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kGkMaxSmem);
    if (e == cudaSuccess) done.fetch_or(bit);
    return e;
}

constexpr uint32_t kBarBytes = (2 * NS_MAX + 2 * NA_MAX + 2 + 4 + 1) * 8;
constexpr uint32_t kMinSmem = 118 * 1024;   // at least this much: one CTA per SM (each takes all tensor memory)

// Shared-memory layout of one CTA with ns stages: X stages | W stages | two
// records | two bias copies | epilogue staging tiles | barriers | misc; 0 if
// it does not fit.
uint32_t layout(int ns, uint32_t wstage, uint32_t ibytes, int G, int R, GkArgs *a) {
    const uint32_t w_off = ns * kStageBytes, rec_smem = w_off + ns * wstage;
    const uint32_t bias_off = rec_smem + 2 * ibytes;
    const uint32_t stg_off = (bias_off + (uint32_t)((2 * G * R * 4 + 15) & ~15) + 127) & ~127u;
    const uint32_t bar_off = stg_off + NEW * 32 * 32 * 4;   // a 32 x 32 fp32 staging tile per epilogue warp
    const uint32_t misc_off = bar_off + kBarBytes;
    const uint32_t smem = misc_off + 16 + 1024;
    if (a) {
        a->ns = ns;
        a->w_off = w_off;
        a->rec_smem = rec_smem;
        a->rec_bytes = ibytes;
        a->bias_off = bias_off;
        a->stg_off = stg_off;
        a->bar_off = bar_off;
        a->misc_off = misc_off;
    }
    return smem <= (uint32_t)kGkMaxSmem ? std::max(smem, kMinSmem) : 0;
}

template <typename T, int R>
cudaError_t launch_r(const LaunchArgs &la, int G) {
    const Schedule &sc = *la.sc;
    const GkPlan &pl = sc.gk;
    int gi = -1;
    for (int i = 0; i < kGkTaskSizes; i++)
        if (kGkG[i] == G) gi = i;
    if (gi < 0 || pl.off[gi] < 0) return cudaErrorInvalidConfiguration;
    GkArgs a;
    a.G = G;
    a.n_tasks = pl.n_tasks[gi];
    a.rec = pl.d_rec[gi];
    a.rec_off = pl.d_rec_off[gi];
    a.wpk = static_cast<const unsigned char *>(la.data) + pl.off[gi];
    a.wstage = pl.wstage[gi];
    a.wslot = pl.wstage[gi] + pl.pstage[gi];
    a.prog = reinterpret_cast<const uint4 *>(pl.d_prog[gi]);
    if (!a.prog) return cudaErrorInvalidConfiguration;
    a.acols = pl.acols[gi];
    a.na = gk_slots(R, sc.C, sizeof(T) == 4, G);
    a.bias = la.bias;
    a.Y = la.Y;
    a.status = la.status;
    a.N = la.N;
    a.K = sc.K;
    a.M = sc.M;
    a.C = sc.C;
    a.nchunks = (int)((sc.K + gk_chunk_cols(sc.dt) - 1) / gk_chunk_cols(sc.dt));
    a.wait_ns = la.wait_ns;
    a.stall_chunk = la.stall_chunk;
    uint32_t smem = 0;
    for (int ns = NS_MAX; ns >= 2 && !smem; ns--) smem = layout(ns, a.wslot, pl.ibytes[gi], G, R, &a);
    if (!smem || a.na < 2 || (uint32_t)(G * R) + (uint32_t)a.na * a.acols > (uint32_t)kGkTmemCols)
        return cudaErrorInvalidConfiguration;
    static std::atomic<uint64_t> attr_set{0};
    cudaError_t e = allow_smem(k_gk<T, R>, attr_set);
    if (e != cudaSuccess) return e;
    CUtensorMap map;
    if ((e = encode_x<T>(la.X, la.N, sc.K, &map)) != cudaSuccess) return e;
    const int64_t units = ((la.N + TN - 1) / TN) * a.n_tasks;
    const int64_t grid = std::min<int64_t>(units, sc.sm_count);   // persistent: one CTA per SM
    return launch_kernel(k_gk<T, R>, dim3((unsigned)grid), dim3(NTHREADS), smem, la.stream, map, a);
}

template <typename T>
cudaError_t launch_t(const LaunchArgs &la, int G) {
    switch (la.sc->R) {
        case 16: return launch_r<T, 16>(la, G);
        case 32: return launch_r<T, 32>(la, G);
        case 64: return launch_r<T, 64>(la, G);
        case 128: return launch_r<T, 128>(la, G);
    }
    return cudaErrorNotSupported;
}

}  // namespace

bool gk_supports(int R, int C, bsr_dtype_t dt, int64_t K) {
    const bool r_ok = R == 16 || R == 32 || R == 64 || R == 128;
    const bool c_ok = C == 1 || C == 2 || C == 4 || C == 8 || C == 16 || C == 32;
    const int64_t align = dt == BSR_F32 ? 4 : 8;   // TMA row pitch: a multiple of 16 bytes
    return r_ok && c_ok && K % align == 0 && K > 0;
}

size_t gk_smem_bytes(bsr_dtype_t dt, size_t wstage, size_t ibytes, int G, int R) {
    (void)dt;
    // the smallest ring (two stages); more stages are used when they fit
    const uint32_t smem = layout(2, (uint32_t)((wstage + 15) & ~size_t(15)), (uint32_t)((ibytes + 15) & ~size_t(15)),
                                 G, R, nullptr);
    return smem ? smem : (size_t)kGkMaxSmem + 1;
}

cudaError_t pack_gk_data(const void *data, bsr_dtype_t dt, const int32_t *wsrc, const int32_t *wslot,
                         const int64_t *wbase, int64_t n, int R, int C, void *out, cudaStream_t s) {
    const int64_t total = n * R * C;
    if (total == 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>((total + 255) / 256, 1 << 20);
    if (dt == BSR_F32)
        k_pack_gk<float><<<grid, 256, 0, s>>>(static_cast<const float *>(data), wsrc, wslot, wbase, n, R, C,
                                              static_cast<unsigned char *>(out));
    else
        k_pack_gk<uint16_t><<<grid, 256, 0, s>>>(static_cast<const uint16_t *>(data), wsrc, wslot, wbase, n, R, C,
                                                 static_cast<unsigned char *>(out));
    return cudaGetLastError();
}

cudaError_t launch_gk(const LaunchArgs &la, int G) {
    if (la.N == 0 || !la.sc->gk.ok) return la.N == 0 ? cudaSuccess : cudaErrorInvalidConfiguration;
    return la.sc->dt == BSR_F32 ? launch_t<float>(la, G) : launch_t<uint16_t>(la, G);
}

}  // namespace bsr
