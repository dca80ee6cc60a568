// Persistent tcgen05 tensor-core BSR x dense kernel ("tcp"), on the task
// records and packed block values of the "tc" kernel (tc.h): every kept
// block is a dense contraction (Section 2.2), C/16 (bf16) or 3 C/8 (fp32 as
// 3xTF32) MMAs of M = 128 tokens, N = R outputs, accumulated in fp32 in
// tensor memory, with A (the X tile) in tensor memory and B (the block) in
// shared memory.
//
// One CTA per SM walks a contiguous range of units (task, tile of 128
// tokens), task-major, and keeps every pipeline full across unit
// boundaries. A stage is tcp_stage_chunks consecutive 128-byte K chunks of
// X (256 bf16 or 64 fp32 columns) and the task's block values for them:
//
//   warp 0 (one thread)   producer: per task its record (two buffers), then
//                          per unit and stage holding any of the task's
//                          blocks the X boxes [128 tokens x 128 bytes] by 2-D
//                          TMA (128-byte swizzle) into an X ring, and the
//                          stage's packed block values into a W ring.
//   4 loader warps         copy each landed X stage into one of a ring of A
//                          slots in tensor memory (thread t: token t's row,
//                          lane t), fp32 split on the way into a tf32 high
//                          part and the remainder, then free the X buffer.
//                          A in tensor memory costs an MMA no 4 KB
//                          shared-memory read of A: for N = 16 or 32 the MMA
//                          rate is then set by instruction issue.
//   warps 1..NISS          issuers: the issue rate grows with the number of
//                          issuing warps, so each owns a contiguous range of
//                          the task's items (their accumulators), balanced
//                          by block count. The warp decodes 32 entries at
//                          once and lane 0 issues the MMAs of its own, in
//                          entry order; a stacked chunk (one block per item)
//                          is one MMA per issuer over its items' adjacent
//                          accumulators. fp32 runs high x high + high x low
//                          + low x high. Commits free the A slot and the W
//                          buffer, and per unit hand the accumulators to the
//                          epilogue.
//   4 epilogue warps       per unit: read their 32 tensor-memory lanes of
//                          the accumulators, add the bias, turn the tile
//                          around through shared memory and store whole row
//                          segments of Y (split rows: fp32 partials to the
//                          workspace), then free the accumulators.
//
// Tensor memory holds the accumulators (two buffers of G R columns when two
// A slots still fit, so a unit's epilogue overlaps the next unit's MMAs;
// else one) and 128-column A slots. Launched with programmatic stream
// serialisation. Every wait is bounded by the global timer; a timeout sets
// the device status word, stops issuing, lets the issued copies and MMAs
// finish, frees the tensor memory and returns.
#include <cuda.h>

#include <algorithm>
#include <atomic>
#include <cstdlib>

#include "bsr_internal.h"
#include "elem.cuh"
#include "launch.cuh"
#include "ptx.cuh"
#include "tc.h"
#include "tcgen05.cuh"

namespace bsr {

namespace {

constexpr int TN = kTcTokens;
constexpr int NISS = kTcpIssuers;
constexpr int NLW4 = 4;                       // fp32 loader warps: one per tensor-memory lane quarter
constexpr int NEW = 4;                        // epilogue warps: one per tensor-memory lane quarter
constexpr int NXMAX = 6;                      // X ring buffers
constexpr int NWMAX = 8;                      // W ring buffers
constexpr int NAMAX = 3;                      // A slots in tensor memory
constexpr uint32_t kBoxBytes = TN * 128;      // one X box: 128 token rows of 128 bytes
constexpr uint32_t kACols = 128;              // tensor-memory columns of one A slot
constexpr uint64_t kDrainNs = 200000000ull;
constexpr uint32_t kTmemCols = 512;

template <typename T>
struct TcpCfg {
    static constexpr bool F32 = sizeof(T) == 4;
    static constexpr int KC = 128 / (int)sizeof(T);   // K columns per chunk
    static constexpr int SC = kTcpStageChunks;         // chunks per stage (the stage programs' unit)
    static constexpr uint32_t XBYTES = SC * kBoxBytes;
    static constexpr int NLW = F32 ? NLW4 : 0;        // loaders (fp32: A in tensor memory; bf16: A in shared memory)
    static constexpr int NWARPS = 1 + NISS + NLW + NEW;
    static constexpr int NTHREADS = 32 * NWARPS;
};

struct TcpArgs {
    int G, n_tasks, nx, nw, na, nacc;   // ring depths: X, W, A slots; accumulator buffers (1 or 2)
    const int32_t *trec;                // task records
    const int32_t *trec_off;            // per task: record offset (ints)
    const unsigned char *wpk;           // packed block values of this task size
    const uint4 *prog;                  // stage programs of this task size
    const int32_t *stab;                // per task: per stage (program offset / 16, program bytes)
    uint32_t wstage, wslot;             // bytes of a stage's block values (most), of one W buffer (values + program)
    uint32_t stab_bytes;                // bytes of one task's stage table
    const float *bias;
    void *Y;
    float *ws;
    int *status;
    int64_t N, K, M;
    int C, nchunks, nstages;
    uint32_t w_off, rec_smem, rec_bytes, stab_smem, bias_off, stg_off, bar_off, misc_off;
    uint64_t wait_ns;
    int stall_chunk;                    // test hook: the stage holding this chunk in each CTA's first unit is never
                                        // loaded (-1: none)
};

__device__ __forceinline__ void set_status(int *status, int code) { atomicCAS(status, DEV_OK, code); }
__device__ __forceinline__ bool aborted(const int *flag) { return *reinterpret_cast<const volatile int *>(flag) != 0; }
__device__ __forceinline__ int pad4(int n) { return (n + 3) & ~3; }
// The abort flag as the whole warp sees it (one value for every lane)
__device__ __forceinline__ bool warp_aborted(const int *flag) { return __any_sync(0xffffffffu, aborted(flag)); }

__device__ __forceinline__ uint4 lds_128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}

// A warp waits for a phase: lane 0 alone polls (a warp of pollers floods
// the barrier unit that every other warp's waits and arrivals go through),
// then every lane observes the completed phase once itself. `idle`: sleep
// between polls (long waits). True when the phase completed in time.
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, uint64_t limit_ns, bool idle = false) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0)
        ok = idle ? ptx::mbar_wait_bounded_idle(bar, parity, limit_ns) : ptx::mbar_wait_bounded(bar, parity, limit_ns);
    ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    if (ok) ok = __all_sync(0xffffffffu, ptx::mbar_try_wait(bar, parity));
    return ok;
}

template <typename T, int R>
__global__ void __launch_bounds__(TcpCfg<T>::NTHREADS, 1)
k_tcp(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ TcpArgs a) {
    ptx::pdl_launch_dependents();
    using Cfg = TcpCfg<T>;
    constexpr bool F32 = Cfg::F32;
    constexpr int SC = Cfg::SC;
    constexpr int NLW = Cfg::NLW;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *base =
        reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *xfull = reinterpret_cast<uint64_t *>(base + a.bar_off);
    uint64_t *xempty = xfull + NXMAX;   // the loaders copied the X buffer to tensor memory
    uint64_t *wfull = xempty + NXMAX;
    uint64_t *wempty = wfull + NWMAX;   // every issuer's MMAs on the W buffer completed
    uint64_t *afull = wempty + NWMAX;   // A slot written (loader warps)
    uint64_t *aempty = afull + NAMAX;   // every issuer's MMAs on the A slot completed
    uint64_t *accf = aempty + NAMAX;    // [2] a unit's MMAs completed (every issuer)
    uint64_t *acce = accf + 2;          // [2] the epilogue read the accumulator buffer
    uint64_t *rbar = acce + 2;          // [2] record landed
    uint64_t *rfree = rbar + 2;         // [2] record no longer used
    uint64_t *done = rfree + 2;         // every MMA issued completed
    int *misc = reinterpret_cast<int *>(base + a.misc_off);   // [0] abort flag, [1] tensor-memory address
    unsigned char *W_s = base + a.w_off;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nx = a.nx, nw = a.nw, na = a.na, nch = a.nchunks, nst = a.nstages, nacc = a.nacc, C = a.C;
    const int64_t n_tiles = (a.N + TN - 1) / TN;
    const int64_t units = n_tiles * a.n_tasks, P = gridDim.x;
    const int64_t ub = units * (int64_t)blockIdx.x / P, ue = units * ((int64_t)blockIdx.x + 1) / P;
    const int items_at = 4 + pad4(nch + 1);   // record: header, chunk starts, items, entries
    const uint32_t acc_cols = (uint32_t)(a.G * R);
    const uint32_t wblock = (uint32_t)R * C * (F32 ? 8 : 2);   // bytes of one block's B operand(s)
    auto rec_s = [&](int j) { return reinterpret_cast<int32_t *>(base + a.rec_smem + (j & 1) * a.rec_bytes); };
    auto stab_s = [&](int j) { return reinterpret_cast<int32_t *>(base + a.stab_smem + (j & 1) * a.stab_bytes); };
    auto bias_s = [&](int j) { return reinterpret_cast<float *>(base + a.bias_off) + (j & 1) * a.G * R; };
    auto last_of_task = [&](int64_t u) { return u + 1 == ue || (u + 1) / n_tiles != u / n_tiles; };
    // first entry of stage st (st = nst: the end)
    auto stage_lo = [&](const int32_t *I, int st) { return I[4 + min(st * SC, nch)]; };

    if (threadIdx.x == 0) {
        for (int s = 0; s < NXMAX; s++) {
            ptx::mbar_init(&xfull[s], 1);
            ptx::mbar_init(&xempty[s], F32 ? NLW : NISS);   // fp32: the loaders copied it; bf16: the MMAs read it
        }
        for (int s = 0; s < NWMAX; s++) {
            ptx::mbar_init(&wfull[s], 1);
            ptx::mbar_init(&wempty[s], NISS);
        }
        for (int s = 0; s < NAMAX; s++) {
            ptx::mbar_init(&afull[s], NLW > 0 ? NLW : 1);   // (unused without loaders)
            ptx::mbar_init(&aempty[s], NISS);
        }
        for (int b = 0; b < 2; b++) {
            ptx::mbar_init(&accf[b], NISS);
            ptx::mbar_init(&acce[b], NEW);
            ptx::mbar_init(&rbar[b], 1);
            ptx::mbar_init(&rfree[b], NISS + NLW + NEW);
        }
        ptx::mbar_init(done, NISS);
        misc[0] = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 1) tc5::alloc(reinterpret_cast<uint32_t *>(&misc[1]), kTmemCols);
    tc5::fence_before();
    __syncthreads();
    tc5::fence_after();
    const uint32_t tmem = (uint32_t)misc[1];
    const uint32_t abase = tmem + (uint32_t)nacc * acc_cols;   // the A slots, after the accumulators

    if (warp == 0) {
        // ---------------- producer
        if (lane == 0 && ub < ue) {
            ptx::prefetch_tensormap(&xmap);
            auto load_rec = [&](int j, int64_t task) {   // the task record and its stage table
                const int32_t *g = a.trec + __ldg(a.trec_off + task);
                const uint32_t bytes = (uint32_t)(items_at + 4 * __ldg(g + 1) + pad4(__ldg(g + 4 + nch))) * 4u;
                ptx::mbar_arrive_expect_tx(&rbar[j & 1], bytes + a.stab_bytes);
                ptx::bulk_load(rec_s(j), g, bytes, &rbar[j & 1]);
                ptx::bulk_load(stab_s(j), a.stab + task * (int64_t)(a.stab_bytes / 4), a.stab_bytes, &rbar[j & 1]);
            };
            int j = 0;
            int64_t task = ub / n_tiles;
            load_rec(0, task);
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
                    load_rec(j, task);
                    if (!ptx::mbar_wait_bounded(&rbar[j & 1], (j >> 1) & 1, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                }
                const int32_t *I = rec_s(j);
                const int64_t wfirst = I[0];   // the task's first packed block
                const int32_t n0 = (int32_t)((u % n_tiles) * TN);
                for (int st = 0; st < nst; st++) {
                    const int lo = stage_lo(I, st), hi = stage_lo(I, st + 1);
                    if (lo == hi) continue;   // no block of this task in the stage
                    const int sx = (int)(k % nx), sw = (int)(k % nw);
                    if (k >= nx && !ptx::mbar_wait_bounded(&xempty[sx], (uint32_t)((k / nx) - 1) & 1, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    if (k >= nw && !ptx::mbar_wait_bounded(&wempty[sw], (uint32_t)((k / nw) - 1) & 1, a.wait_ns)) {
                        ok = false;
                        break;
                    }
                    if (aborted(misc)) { ok = false; break; }
                    if (u == ub && a.stall_chunk >= 0 && a.stall_chunk / SC == st) {   // never loaded: its consumers time out
                        stalled = k++;
                        continue;
                    }
                    const int c0 = st * SC, cn = min(SC, nch - c0);
                    ptx::mbar_arrive_expect_tx(&xfull[sx], (uint32_t)cn * kBoxBytes);
                    for (int i = 0; i < cn; i++)
                        ptx::tma_load_2d(base + sx * Cfg::XBYTES + i * kBoxBytes, &xmap, (c0 + i) * Cfg::KC, n0, &xfull[sx]);
                    // the stage's block values and, after them, its MMA program
                    const uint32_t wbytes = (uint32_t)(hi - lo) * wblock;
                    const int32_t *tab = stab_s(j) + 2 * st;
                    const uint32_t pbytes = (uint32_t)tab[1];
                    unsigned char *slot = W_s + sw * a.wslot;
                    ptx::mbar_arrive_expect_tx(&wfull[sw], wbytes + pbytes);
                    ptx::bulk_load(slot, a.wpk + (wfirst + lo) * (int64_t)wblock, wbytes, &wfull[sw]);
                    ptx::bulk_load(slot + a.wstage, a.prog + tab[0], pbytes, &wfull[sw]);
                    k++;
                }
            }
            if (!ok) {
                set_status(a.status, DEV_TIMEOUT);
                atomicExch(&misc[0], 1);
            }
            // copies still in flight land before the CTA exits
            for (int64_t d = k > nx ? k - nx : 0; d < k; d++)
                if (d != stalled) ptx::mbar_wait_bounded(&xfull[d % nx], (uint32_t)(d / nx) & 1, kDrainNs);
            for (int64_t d = k > nw ? k - nw : 0; d < k; d++)
                if (d != stalled) ptx::mbar_wait_bounded(&wfull[d % nw], (uint32_t)(d / nw) & 1, kDrainNs);
            ptx::mbar_wait_bounded(&rbar[j & 1], (j >> 1) & 1, kDrainNs);
        }
    } else if (warp <= NISS) {
        // ---------------- MMA issuers: lane 0 of each warp runs its part of
        // every stage's program, one word per MMA
        if (lane == 0) {
            const int q = warp - 1;
            bool ok = true;
            int j = -1;
            int64_t task = -1, k = 0, ui = 0;
            const int32_t *I = rec_s(0);
            for (int64_t u = ub; ok && u < ue; u++, ui++) {
                if (u / n_tiles != task) {
                    task = u / n_tiles;
                    j++;
                    if (!ptx::mbar_wait_bounded(&rbar[j & 1], (j >> 1) & 1, a.wait_ns)) { ok = false; break; }
                    I = rec_s(j);
                }
                const int b = (int)(ui % nacc);
                // the epilogue has read this buffer's previous unit
                if (ui >= nacc && !ptx::mbar_wait_bounded(&acce[b], (uint32_t)((ui / nacc) - 1) & 1, a.wait_ns)) {
                    ok = false;
                    break;
                }
                tc5::fence_after();
                const uint32_t dacc = tmem + (uint32_t)b * acc_cols;
                for (int st = 0; ok && st < nst; st++) {
                    if (stage_lo(I, st) == stage_lo(I, st + 1)) continue;
                    const int sw = (int)(k % nw), sa = (int)(k % na);
                    const int sx = (int)(k % nx);
                    // A: fp32, the loaders wrote the stage's X into A slot sa;
                    // bf16, X landed in buffer sx. The block values and the
                    // program landed
                    const bool got_a = F32 ? ptx::mbar_wait_bounded(&afull[sa], (uint32_t)(k / na) & 1, a.wait_ns)
                                           : ptx::mbar_wait_bounded(&xfull[sx], (uint32_t)(k / nx) & 1, a.wait_ns);
                    if (!got_a || !ptx::mbar_wait_bounded(&wfull[sw], (uint32_t)(k / nw) & 1, a.wait_ns) || aborted(misc)) {
                        ok = false;
                        break;
                    }
                    tc5::fence_after();
                    const unsigned char *slot = W_s + sw * a.wslot;
                    const int32_t *hdr = reinterpret_cast<const int32_t *>(slot + a.wstage);
                    const uint4 *pw = reinterpret_cast<const uint4 *>(hdr + kTcpProgHeader);
                    const uint64_t b0 = tc5::desc(ptx::smem_addr(slot), 128, 256);
                    const int i0 = hdr[q], i1 = hdr[q + 1];
                    int i = i0;
                    if constexpr (F32) {
                        const uint32_t aslot = abase + (uint32_t)sa * kACols;
                        for (; i + 2 <= i1; i += 2) {   // two words loaded ahead of their MMAs
                            const uint4 w0 = pw[i], w1 = pw[i + 1];
                            tc5::mma_ts<true>(dacc + w0.y, aslot + (w0.z & 0x7fffffffu), b0 + w0.x, w0.w, w0.z >> 31);
                            tc5::mma_ts<true>(dacc + w1.y, aslot + (w1.z & 0x7fffffffu), b0 + w1.x, w1.w, w1.z >> 31);
                        }
                        if (i < i1) {
                            const uint4 w0 = pw[i];
                            tc5::mma_ts<true>(dacc + w0.y, aslot + (w0.z & 0x7fffffffu), b0 + w0.x, w0.w, w0.z >> 31);
                        }
                        tc5::commit(&aempty[sa]);   // the A slot and
                    } else {
                        const uint64_t a0 = tc5::desc_sw128(ptx::smem_addr(base + sx * Cfg::XBYTES));
                        for (; i + 2 <= i1; i += 2) {
                            const uint4 w0 = pw[i], w1 = pw[i + 1];
                            tc5::mma_ss<false>(dacc + w0.y, a0 + (w0.z & 0x7fffffffu), b0 + w0.x, w0.w, w0.z >> 31);
                            tc5::mma_ss<false>(dacc + w1.y, a0 + (w1.z & 0x7fffffffu), b0 + w1.x, w1.w, w1.z >> 31);
                        }
                        if (i < i1) {
                            const uint4 w0 = pw[i];
                            tc5::mma_ss<false>(dacc + w0.y, a0 + (w0.z & 0x7fffffffu), b0 + w0.x, w0.w, w0.z >> 31);
                        }
                        tc5::commit(&xempty[sx]);   // the X buffer and
                    }
                    tc5::commit(&wempty[sw]);   // the W buffer are free once every issuer's MMAs on them completed
                    k++;
                }
                if (!ok) break;
                tc5::commit(&accf[b]);   // the unit's accumulators are complete
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
    } else if (NLW > 0 && warp <= NISS + NLW) {
        // ---------------- loaders; lane quarter = warp % 4: thread t copies
        // token t's row of each landed X stage into the stage's A slot
        const int q = warp & 3;
        const int t = 32 * q + lane;
        const uint32_t swz = (uint32_t)(t & 7);   // 128-byte swizzle: 16-byte group g of row t sits at g ^ (t % 8)
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        bool ok = true;
        int j = -1;
        int64_t task = -1, k = 0;
        for (int64_t u = ub; ok && u < ue; u++) {
            if (u / n_tiles != task) {
                task = u / n_tiles;
                j++;
                if (!warp_wait(&rbar[j & 1], (j >> 1) & 1, a.wait_ns)) { ok = false; break; }
            }
            const int32_t *I = rec_s(j);
            for (int st = 0; st < nst; st++) {
                if (stage_lo(I, st) == stage_lo(I, st + 1)) continue;
                const int sx = (int)(k % nx), sa = (int)(k % na);
                bool got = warp_wait(&xfull[sx], (uint32_t)(k / nx) & 1, a.wait_ns);
                if (got && k >= na) got = warp_wait(&aempty[sa], (uint32_t)((k / na) - 1) & 1, a.wait_ns);
                if (!got || warp_aborted(misc)) { ok = false; break; }
                tc5::fence_after();   // the MMAs that read the slot before have completed
                const int cn = min(SC, nch - st * SC);
                const uint32_t col0 = abase + lane_off + (uint32_t)sa * kACols;
                for (int i = 0; i < cn; i++) {
                    const uint32_t row = ptx::smem_addr(base + sx * Cfg::XBYTES + i * kBoxBytes) + (uint32_t)t * 128u;
                    uint32_t r[32];
#pragma unroll
                    for (int g = 0; g < 8; g++) {
                        const uint4 v = lds_128(row + (((uint32_t)g ^ swz) << 4));
                        r[4 * g] = v.x, r[4 * g + 1] = v.y, r[4 * g + 2] = v.z, r[4 * g + 3] = v.w;
                    }
                    if constexpr (F32) {
                        // x = high + low: high = x with the low 13 mantissa bits
                        // cleared (a tf32 value), low = x - high (exact in fp32)
                        uint32_t lo[32];
#pragma unroll
                        for (int e = 0; e < 32; e++) {
                            const uint32_t h = r[e] & 0xffffe000u;
                            lo[e] = __float_as_uint(__uint_as_float(r[e]) - __uint_as_float(h));
                            r[e] = h;
                        }
                        tc5::st32(col0 + 32u * i, r);
                        tc5::st32(col0 + 64u + 32u * i, lo);
                    } else {
                        tc5::st32(col0 + 32u * i, r);   // column c: bf16 elements 2c (low half) and 2c + 1
                    }
                }
                tc5::st_wait();
                tc5::fence_before();
                __syncwarp();
                if (lane == 0) {
                    ptx::mbar_arrive(&xempty[sx]);   // the X buffer may be refilled
                    ptx::mbar_arrive(&afull[sa]);
                }
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
        const int et = threadIdx.x - 32 * (1 + NISS + NLW);   // 0..127
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        ptx::pdl_wait();   // the bias, Y and the workspace may be an earlier kernel's
        bool ok = true;
        int j = -1;
        int64_t task = -1, ui = 0;
        float *stg = reinterpret_cast<float *>(base + a.stg_off) + (warp - 1 - NISS - NLW) * 32 * 32;
        const uint32_t stg_base = ptx::smem_addr(stg), stg_row = stg_base + (uint32_t)lane * 128u;
        for (int64_t u = ub; ok && u < ue; u++, ui++) {
            if (u / n_tiles != task) {
                task = u / n_tiles;
                j++;
                const bool got = warp_wait(&rbar[j & 1], (j >> 1) & 1, a.wait_ns) && !aborted(misc);
                if (ptx::named_barrier_or(1, 32 * NEW, !got)) { ok = false; break; }
                const int32_t *I = rec_s(j);
                float *B = bias_s(j);
                for (int e = et; e < I[1] * R; e += 32 * NEW) {
                    const int g = e / R, r = e - g * R;
                    B[e] = a.bias && I[items_at + 4 * g + 3] < 0 ? __ldg(a.bias + (int64_t)I[items_at + 4 * g] * R + r)
                                                                  : 0.f;   // split rows: the reduce pass adds it
                }
                ptx::named_barrier(1, 32 * NEW);
            }
            const int32_t *I = rec_s(j);
            const int32_t *items = I + items_at;
            const float *B = bias_s(j);
            const int b = (int)(ui % nacc);
            const uint64_t limit = a.wait_ns * (uint64_t)(nst + 2);
            const bool got = warp_wait(&accf[b], (uint32_t)(ui / nacc) & 1, limit, true);
            if (!got || warp_aborted(misc)) { ok = false; break; }
            tc5::fence_after();
            const uint32_t dacc = tmem + lane_off + (uint32_t)b * acc_cols;
            const int64_t row0 = (u % n_tiles) * TN + 32 * q;   // the warp's first token
            // per 32 (or 16) accumulator columns: each lane's row of the
            // tile into the warp's staging tile (16-byte groups XOR-swizzled by
            // row), then lanes re-read it as (row, 8-column group) pairs and
            // store whole row segments of each item in the group
            constexpr int SEG = R < 32 ? R : 32;   // columns of one item in a group of 32
            const int cols = I[1] * R;             // a multiple of 32, or 16 (one item of 16 rows)
            for (int c0 = 0; c0 < cols; c0 += 32) {
                const int wc = min(32, cols - c0);
                uint32_t r[32];
                if (wc == 32) {
                    tc5::ld32(dacc + (uint32_t)c0, r);
                } else {
                    uint32_t r16[16];
                    tc5::ld16(dacc + (uint32_t)c0, r16);
#pragma unroll
                    for (int i = 0; i < 16; i++) r[i] = r16[i], r[16 + i] = 0u;
                }
                tc5::ld_wait();
#pragma unroll
                for (int c4 = 0; c4 < 8; c4++) {
                    if (4 * c4 >= wc) break;
                    const int col = c0 + 4 * c4, g = col / R;
                    const bool any = items[4 * g + 2] > items[4 * g + 1];   // an item with no blocks: the bias alone
                    float o[4];
#pragma unroll
                    for (int i = 0; i < 4; i++) o[i] = (any ? __uint_as_float(r[4 * c4 + i]) : 0.f) + B[col + i];
                    asm volatile("st.shared.v4.f32 [%0], {%1,%2,%3,%4};" ::"r"(stg_row + ((c4 ^ (lane & 7)) << 4)),
                                 "f"(o[0]), "f"(o[1]), "f"(o[2]), "f"(o[3])
                                 : "memory");
                }
                __syncwarp();
                for (int h = 0; h < wc; h += SEG) {
                    constexpr int GPR = SEG / 8;          // 8-column groups per row segment
                    constexpr int RPI = 32 / GPR;         // rows per instruction
                    const int g = (c0 + h) / R, hr = c0 + h - g * R;
                    const int row = items[4 * g], slot = items[4 * g + 3];
                    const int rr = lane / GPR, gg = lane % GPR;
#pragma unroll
                    for (int p0 = 0; p0 < 32; p0 += RPI) {
                        const int rw = p0 + rr;
                        const int64_t n = row0 + rw;
                        const uint32_t src = stg_base + (uint32_t)rw * 128u;
                        const int q0 = (h / 4) + 2 * gg;   // this lane's first 16-byte group in the staged row
                        float4 lo4, hi4;
                        asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                                     : "=f"(lo4.x), "=f"(lo4.y), "=f"(lo4.z), "=f"(lo4.w)
                                     : "r"(src + (uint32_t)((q0 ^ (rw & 7)) << 4)));
                        asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                                     : "=f"(hi4.x), "=f"(hi4.y), "=f"(hi4.z), "=f"(hi4.w)
                                     : "r"(src + (uint32_t)(((q0 + 1) ^ (rw & 7)) << 4)));
                        if (n >= a.N) continue;
                        if (slot >= 0) {
                            float4 *dst = reinterpret_cast<float4 *>(a.ws + ((int64_t)slot * a.N + n) * R + hr + 8 * gg);
                            dst[0] = lo4;
                            dst[1] = hi4;
                        } else if constexpr (F32) {
                            float4 *dst = reinterpret_cast<float4 *>(reinterpret_cast<float *>(a.Y) + n * a.M +
                                                                     (int64_t)row * R + hr + 8 * gg);
                            dst[0] = lo4;
                            dst[1] = hi4;
                        } else {
                            uint4 pk;
                            pk.x = (uint32_t)from_f32<uint16_t>(lo4.x) | ((uint32_t)from_f32<uint16_t>(lo4.y) << 16);
                            pk.y = (uint32_t)from_f32<uint16_t>(lo4.z) | ((uint32_t)from_f32<uint16_t>(lo4.w) << 16);
                            pk.z = (uint32_t)from_f32<uint16_t>(hi4.x) | ((uint32_t)from_f32<uint16_t>(hi4.y) << 16);
                            pk.w = (uint32_t)from_f32<uint16_t>(hi4.z) | ((uint32_t)from_f32<uint16_t>(hi4.w) << 16);
                            *reinterpret_cast<uint4 *>(reinterpret_cast<uint16_t *>(a.Y) + n * a.M + (int64_t)row * R +
                                                       hr + 8 * gg) = pk;
                        }
                    }
                }
                __syncwarp();   // the staging tile is free again
            }
            tc5::fence_before();
            __syncwarp();
            if (lane == 0) {
                ptx::mbar_arrive(&acce[b]);   // the accumulator buffer may be overwritten
                if (last_of_task(u)) ptx::mbar_arrive(&rfree[j & 1]);
            }
        }
        if (!ok && lane == 0) {
            set_status(a.status, DEV_TIMEOUT);
            atomicExch(&misc[0], 1);
        }
    }
    // ---------------- teardown: every MMA issued completed (issuer warp 1
    // waited for them), every tensor-memory access finished; free it
    tc5::fence_before();
    __syncthreads();
    if (warp == 1) {
        tc5::fence_after();
        tc5::dealloc(tmem, kTmemCols);
    }
}

template <typename K>
cudaError_t allow_smem(K kernel, std::atomic<uint64_t> &done) {
    int dev = 0;
    cudaGetDevice(&dev);
    const uint64_t bit = 1ull << (dev & 63);
    if (done.load() & bit) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kTcMaxSmem);
    if (e == cudaSuccess) done.fetch_or(bit);
    return e;
}

constexpr uint32_t kBarBytes = (2 * NXMAX + 2 * NWMAX + 2 * NAMAX + 4 * 2 + 1) * 8;
constexpr uint32_t kMinSmem = 118 * 1024;   // at least this much: one CTA per SM (each takes all tensor memory)

// Shared-memory layout with nx X buffers of xbytes and nw W buffers of
// wslot: X ring | W ring | two records | two stage tables | two bias copies
// | epilogue staging tiles | barriers | misc; 0 if it does not fit.
uint32_t layout(int nx, uint32_t xbytes, int nw, uint32_t wslot, uint32_t ibytes, uint32_t sbytes, int G, int R,
                TcpArgs *a) {
    const uint32_t w_off = nx * xbytes;
    const uint32_t rec_smem = w_off + nw * wslot;
    const uint32_t stab_smem = rec_smem + 2 * ibytes;
    const uint32_t bias_off = stab_smem + 2 * sbytes;
    const uint32_t stg_off = (bias_off + (uint32_t)((2 * G * R * 4 + 15) & ~15) + 127) & ~127u;
    const uint32_t bar_off = stg_off + NEW * 32 * 32 * 4;
    const uint32_t misc_off = bar_off + kBarBytes;
    const uint32_t smem = misc_off + 16 + 1024;
    if (a) {
        a->nx = nx;
        a->nw = nw;
        a->w_off = w_off;
        a->rec_smem = rec_smem;
        a->rec_bytes = ibytes;
        a->stab_smem = stab_smem;
        a->stab_bytes = sbytes;
        a->bias_off = bias_off;
        a->stg_off = stg_off;
        a->bar_off = bar_off;
        a->misc_off = misc_off;
    }
    return smem <= (uint32_t)kTcMaxSmem ? std::max(smem, kMinSmem) : 0;
}

// Tensor-memory split: fp32, two accumulator buffers when two A slots still
// fit beside them, else one, and as many A slots (at most NAMAX) as fit;
// bf16 (A in shared memory), two accumulator buffers when they fit.
void tmem_split(bool f32, int G, int R, int *nacc, int *na) {
    const int left2 = (int)kTmemCols - 2 * G * R, left1 = (int)kTmemCols - G * R;
    if (!f32) {
        *nacc = left2 >= 0 ? 2 : 1;
        *na = left1 >= 0 ? NAMAX : 0;   // (no A slots: only "fits")
        return;
    }
    *nacc = left2 >= 2 * (int)kACols ? 2 : 1;
    *na = std::min(NAMAX, std::max(0, *nacc == 2 ? left2 : left1) / (int)kACols);
}

template <typename T, int R>
cudaError_t launch_r(const LaunchArgs &la, int G) {
    using Cfg = TcpCfg<T>;
    const Schedule &sc = *la.sc;
    if (sc.items.empty()) return cudaSuccess;   // no block rows to compute (the bias is written elsewhere)
    const int gi = tc_g_index(G);
    if (kTcG[gi] != G || sc.tc.w_off[gi] < 0) return cudaErrorInvalidConfiguration;
    TcpArgs a;
    a.G = G;
    a.n_tasks = (int)sc.tc.rec_off[gi].size();
    tmem_split(Cfg::F32, G, R, &a.nacc, &a.na);
    if (a.na < 2) return cudaErrorInvalidConfiguration;
    a.trec = sc.tc.d_rec[gi];
    a.trec_off = sc.tc.d_rec_off[gi];
    a.wpk = static_cast<const unsigned char *>(la.data) + sc.tc.w_off[gi];
    a.prog = reinterpret_cast<const uint4 *>(sc.tc.d_prog[gi]);
    a.stab = sc.tc.d_stab[gi];
    a.wstage = (uint32_t)((sc.tc.tcp_wbytes[gi] + 15) & ~size_t(15));
    a.wslot = a.wstage + (uint32_t)((sc.tc.tcp_pbytes[gi] + 15) & ~size_t(15));
    if (!a.prog || !a.stab) return cudaErrorInvalidConfiguration;
    a.bias = la.bias;
    a.Y = la.Y;
    a.ws = la.ws;
    a.status = la.status;
    a.N = la.N;
    a.K = sc.K;
    a.M = sc.M;
    a.C = sc.ex_C;
    a.nchunks = (int)((sc.K + Cfg::KC - 1) / Cfg::KC);
    a.nstages = (a.nchunks + Cfg::SC - 1) / Cfg::SC;
    a.wait_ns = la.wait_ns;
    a.stall_chunk = la.stall_chunk;
    const uint32_t ibytes = (uint32_t)((sc.tc.task_ibytes[gi] + 15) & ~size_t(15));
    // deepest rings that fit: X first (two or three buffers), then W (up to eight)
    uint32_t smem = 0;
    for (int nx = NXMAX; nx >= 2 && !smem; nx--)
        for (int nw = NWMAX; nw >= 2 && !smem; nw--)
            smem = layout(nx, Cfg::XBYTES, nw, a.wslot, ibytes, (uint32_t)sc.tc.stab_ints * 4u, G, R, &a);
    if (!smem) return cudaErrorInvalidConfiguration;
    static std::atomic<uint64_t> attr_set{0};
    cudaError_t e = allow_smem(k_tcp<T, R>, attr_set);
    if (e != cudaSuccess) return e;
    CUtensorMap map;
    if ((e = tc_encode_x(sc.dt, la.X, la.N, sc.K, &map)) != cudaSuccess) return e;
    const int64_t units = ((la.N + TN - 1) / TN) * a.n_tasks;
    if (units == 0) return cudaSuccess;
    const int64_t grid = std::min<int64_t>(units, sc.sm_count);   // persistent: one CTA per SM
    return launch_kernel(k_tcp<T, R>, dim3((unsigned)grid), dim3(Cfg::NTHREADS), smem, la.stream, map, a);
}

template <typename T>
cudaError_t launch_t(const LaunchArgs &la, int G) {
    switch (la.sc->ex_R) {
        case 16: return launch_r<T, 16>(la, G);
        case 32: return launch_r<T, 32>(la, G);
        case 64: return launch_r<T, 64>(la, G);
        case 128: return launch_r<T, 128>(la, G);
    }
    return cudaErrorNotSupported;
}

}  // namespace

int choose_tcp(const Schedule &sc, int64_t N) {
    static const int mode = [] {
        const char *v = getenv("BSR_TCP");
        return v && *v ? atoi(v) : -1;   // 0: never, 1: whenever a task size fits, unset: by the model
    }();
    static const int forced_g = [] {
        const char *v = getenv("BSR_TCP_G");
        return v ? atoi(v) : 0;
    }();
    if (sc.variant != V_TC || N <= 0 || mode == 0) return -1;
    if (mode != 1) return -1;
    // a task size runs when its A slots fit tensor memory and two X and two W
    // buffers fit shared memory
    const uint32_t xbytes = (uint32_t)tcp_stage_chunks(sc.dt) * kBoxBytes;
    auto usable = [&](int gi) {
        int nacc = 0, na = 0;
        tmem_split(sc.dt == BSR_F32, kTcG[gi], sc.ex_R, &nacc, &na);
        const uint32_t wslot = (uint32_t)((sc.tc.tcp_wbytes[gi] + 15) & ~size_t(15)) +
                               (uint32_t)((sc.tc.tcp_pbytes[gi] + 15) & ~size_t(15));
        const uint32_t ibytes = (uint32_t)((sc.tc.task_ibytes[gi] + 15) & ~size_t(15));
        return sc.tc.w_off[gi] >= 0 && !sc.tc.prog[gi].empty() && na >= 2 &&
               layout(2, xbytes, 2, wslot, ibytes, (uint32_t)sc.tc.stab_ints * 4u, kTcG[gi], sc.ex_R, nullptr) != 0;
    };
    for (int gi = 0; gi < kTcTaskSizes; gi++)
        if (forced_g == kTcG[gi] && usable(gi)) return kTcG[gi];
    // the largest task size that still gives every SM a unit
    const int64_t tiles = (N + TN - 1) / TN;
    int best = -1;
    for (int gi = 0; gi < kTcTaskSizes; gi++) {
        if (!usable(gi)) continue;
        const int64_t units = tiles * (int64_t)sc.tc.rec_off[gi].size();
        if (best < 0 || units >= sc.sm_count) best = kTcG[gi];
    }
    return best;
}

void plan_tcp(Schedule &sc) {
    const int kc = tc_chunk_cols(sc.dt), SC = tcp_stage_chunks(sc.dt);
    const bool f32 = sc.dt == BSR_F32;
    const int64_t nch = (sc.K + kc - 1) / kc, nst = (nch + SC - 1) / SC;
    const int items_at = 4 + (int)tc_pad4(nch + 1);
    const int R = sc.R, C = sc.C;   // the execution block shape (plan_tc runs on re-blocked tiles)
    const uint32_t wb16 = (uint32_t)(tc_block_bytes(R, C, sc.dt) / 16);
    sc.tc.stab_ints = (int)tc_pad4(2 * nst);
    for (int gi = 0; gi < kTcTaskSizes; gi++) {
        std::vector<uint32_t> &prog = sc.tc.prog[gi];
        std::vector<int32_t> &stab = sc.tc.stab[gi];
        prog.clear();
        stab.clear();
        sc.tc.tcp_pbytes[gi] = 0;
        const std::vector<int32_t> &rec = sc.tc.rec[gi];
        if (rec.empty() || (int64_t)kTcG[gi] * R > (int64_t)kTmemCols) continue;
        std::vector<std::vector<uint32_t>> words(NISS);
        for (const int32_t off : sc.tc.rec_off[gi]) {
            const int32_t *I = rec.data() + off;
            const int gc = I[1];
            const int32_t *ent = I + items_at + 4 * gc;
            // issuer of each item: the share of the task's blocks its block-count midpoint falls in
            std::vector<int> owner((size_t)gc, 0);
            std::vector<uint32_t> ufirst(NISS, 0), ucnt(NISS, 0);
            int64_t total = 0, acc = 0;
            for (int g = 0; g < gc; g++) total += I[items_at + 4 * g + 2] - I[items_at + 4 * g + 1];
            for (int g = 0; g < gc; g++) {
                const int64_t len = I[items_at + 4 * g + 2] - I[items_at + 4 * g + 1];
                const int q = total > 0 ? (int)std::min<int64_t>(NISS - 1, (2 * acc + len) * NISS / (2 * total)) : 0;
                acc += len;
                owner[(size_t)g] = q;
                if (ucnt[(size_t)q] == 0) ufirst[(size_t)q] = (uint32_t)g;
                ucnt[(size_t)q]++;
            }
            const size_t tab_at = stab.size();
            stab.resize(tab_at + (size_t)sc.tc.stab_ints, 0);
            for (int64_t st = 0; st < nst; st++) {
                const int32_t slo = I[4 + std::min<int64_t>(st * SC, nch)], shi = I[4 + std::min<int64_t>((st + 1) * SC, nch)];
                if (slo == shi) continue;
                for (auto &w : words) w.clear();
                auto put = [&](int q, uint32_t boff, uint32_t dcol, uint32_t acol, bool accum, uint32_t id) {
                    words[(size_t)q].insert(words[(size_t)q].end(), {boff, dcol, acol | (accum ? 0x80000000u : 0u), id});
                };
                for (int64_t cc = 0; cc < SC && st * SC + cc < nch; cc++) {
                    const int64_t c = st * SC + cc;
                    for (int32_t e = I[4 + c]; e < I[5 + c]; e++) {
                        const uint32_t v = (uint32_t)ent[e];
                        const int g = (int)((v >> 2) & 31u);
                        const bool first = (v >> 7) & 1u;
                        // A: fp32, 8 tensor-memory columns per 32-byte K slice
                        // and 32 per chunk; bf16, descriptor units (16 bytes)
                        // in the X buffer: 2 per 32-byte K slice, 1024 per
                        // 16 KB chunk box
                        const uint32_t acol = f32 ? (uint32_t)cc * 32u + (v & 3u) * 8u : (uint32_t)cc * 1024u + (v & 3u) * 2u;
                        const uint32_t aslice = f32 ? 8u : 2u;
                        const uint32_t boff = (uint32_t)(e - slo) * wb16;
                        if (!f32 && ((v >> 9) & 1u)) continue;   // a stack member: in its head's MMAs
                        if (!f32 && ((v >> 8) & 1u)) {
                            // a stack head: B holds all gc items' blocks; each
                            // issuer's MMA covers its items' rows of it
                            const uint32_t nsr = (uint32_t)(gc * R);
                            for (int q = 0; q < NISS; q++) {
                                if (!ucnt[(size_t)q]) continue;
                                const uint32_t id = tc5::idesc(false, TN, (int)(ucnt[(size_t)q] * R));
                                for (int sl = 0; sl < C / 16; sl++)
                                    put(q, boff + ufirst[(size_t)q] * R * 2u + (uint32_t)sl * nsr * 2u,
                                        ufirst[(size_t)q] * R, acol + aslice * sl, !first || sl > 0, id);
                            }
                            continue;
                        }
                        const int q = owner[(size_t)g];
                        const uint32_t dcol = (uint32_t)g * R;
                        if (f32) {
                            // 3xTF32: high x high + high x low + low x high (low
                            // A parts 64 columns on, low B parts R C floats on)
                            const uint32_t id = tc5::idesc(true, TN, R), blo = (uint32_t)(R * C * 4 / 16);
                            for (int sl = 0; sl < C / 8; sl++) {
                                const uint32_t kb = (uint32_t)sl * R * 2u;
                                put(q, boff + kb, dcol, acol + 8u * sl, !first || sl > 0, id);
                                put(q, boff + blo + kb, dcol, acol + 8u * sl, true, id);
                                put(q, boff + kb, dcol, acol + 64u + 8u * sl, true, id);
                            }
                        } else {
                            const uint32_t id = tc5::idesc(false, TN, R);
                            for (int sl = 0; sl < C / 16; sl++)
                                put(q, boff + (uint32_t)sl * R * 2u, dcol, acol + aslice * sl, !first || sl > 0, id);
                        }
                    }
                }
                // header: issuer q's words are [h[q], h[q + 1]) after it
                const size_t at = prog.size();
                prog.resize(at + kTcpProgHeader, 0u);
                uint32_t n = 0;
                for (int q = 0; q < NISS; q++) {
                    prog[at + (size_t)q] = n;
                    n += (uint32_t)(words[(size_t)q].size() / 4);
                }
                prog[at + NISS] = n;
                for (const auto &w : words) prog.insert(prog.end(), w.begin(), w.end());
                const size_t bytes = (prog.size() - at) * 4;
                stab[tab_at + 2 * (size_t)st] = (int32_t)(at / 4);   // 16-byte units
                stab[tab_at + 2 * (size_t)st + 1] = (int32_t)bytes;
                sc.tc.tcp_pbytes[gi] = std::max(sc.tc.tcp_pbytes[gi], bytes);
            }
        }
        if (prog.size() / 4 > (size_t)INT32_MAX) {   // offsets in 16-byte units must fit an int
            prog.clear();
            stab.clear();
        }
    }
}

cudaError_t launch_tcp(const LaunchArgs &la, int G) {
    if (la.N == 0) return cudaSuccess;
    return la.sc->dt == BSR_F32 ? launch_t<float>(la, G) : launch_t<uint16_t>(la, G);
}

}  // namespace bsr
