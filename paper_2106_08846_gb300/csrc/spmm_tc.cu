// tcgen05 tensor-core BSR x dense kernel ("tc"): bf16 blocks whose both sides
// are multiples of 16 (and narrow bf16 blocks re-blocked at create time into
// zero-filled R x 64 tiles), and fp32 blocks of 32 or more rows as 3xTF32.
// Every kept block is a dense contraction: C/16 (bf16) or 3 C/8 (fp32)
// tcgen05.mma instructions of shape M = 128 tokens, N = R outputs,
// accumulated in fp32 in tensor memory.
//
//   warp 0 (one thread)  producer: the task's work list by one bulk copy,
//                         then per K chunk that holds any of the task's
//                         blocks the X chunk [128 tokens x 128 bytes] by 2-D
//                         TMA (128-byte swizzle) and, beside it in the same
//                         stage, the task's block values for that chunk
//                         (repacked at create time into the MMA's K-major
//                         layout, in task-chunk order); chunks without blocks
//                         are neither loaded nor visited.
//   warp 1 (one thread)  owns the tensor memory (G * R fp32 columns, one
//                         block row per R columns) and issues the MMAs from
//                         the work list (per chunk, one packed entry per
//                         block: column offset, item, first-block flag, stack
//                         head or member); a chunk where every item has one
//                         block is a stack: one MMA per K slice with
//                         N = items x R over their adjacent accumulators. A
//                         tcgen05.commit per chunk releases the stage.
//   warps 2..5           fp32: write the tf32 low parts of every landed X
//                         stage into a twin buffer (the MMAs read the stage
//                         itself as the high parts) for the issuer's
//                         high x high + high x low + low x high; then the
//                         epilogue: each reads its 32 TMEM lanes (tokens),
//                         adds the bias, converts, stages 16-column groups in
//                         the idle X ring and one thread stores them to Y by
//                         2-D TMA (split rows write fp32 partials directly).
//
// Two CTAs share an SM, so that one CTA's set-up, stage round trips and
// epilogue overlap the other's MMAs: bf16 uses a 3-stage ring, fp32 a 2-stage
// ring (plus the low twins).
// Launched with programmatic stream serialisation: set-up and the work list
// come before the wait for the previous kernel; X, bias, Y after it. Every
// wait is bounded by the global timer; a timeout sets the device status word,
// stops issuing, lets the issued copies and MMAs finish, frees the tensor
// memory and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <cstdlib>
#include <mutex>

#include "bsr_internal.h"
#include "elem.cuh"
#include "launch.cuh"
#include "ptx.cuh"
#include "tc.h"
#include "tcgen05.cuh"

namespace bsr {

namespace {

constexpr int TN = kTcTokens;
constexpr uint32_t kStageBytes = TN * 128;   // 16 KB: 128 token rows of 128 bytes (64 bf16 or 32 fp32 columns)
// Per element type: K columns per stage and ring depth (fp32 stages come
// with a second buffer holding the low parts of the split operand).
template <typename T>
struct TcCfg {
    static constexpr int KC = 128 / (int)sizeof(T);
    static constexpr int NS = sizeof(T) == 4 ? kTcStagesF32 : kTcStages;
    static constexpr int NISS = tc_issuers(sizeof(T) == 4);   // MMA-issuing warps (lane 0 of each)
    static constexpr int NTHREADS = tc_threads(sizeof(T) == 4);
};
constexpr uint64_t kDrainNs = 200000000ull;

struct TcArgs {
    CUtensorMap ymap;         // Y [N, M] in 16-column x 128-row boxes, for the epilogue's TMA stores
    int G, n_tasks;           // G: most items in a task (accumulator columns G * R)
    const int32_t *trec;      // task records: header, chunk starts, items, MMA entries
    const int32_t *trec_off;  // per task: record offset (ints)
    const void *wpk;          // block values in the MMA's B layout (fp32: high then low parts), task-chunk order
    uint32_t wstage;          // bytes of one W ring stage
    const float *bias;
    void *Y;
    float *ws;
    int *status;
    int64_t N, K, M;
    int C, nchunks;
    uint32_t w_off, trec_smem, bias_off, bar_off, misc_off;
    uint32_t tmem_cols;
    uint64_t wait_ns;
    int stall_chunk;
};

// fp32 -> (high, low) with high = x with the low 13 mantissa bits cleared
// (a tf32 value) and low = x - high, exact in fp32.
__device__ __forceinline__ float4 tf32_high(float4 v) {
    return make_float4(__uint_as_float(__float_as_uint(v.x) & 0xffffe000u), __uint_as_float(__float_as_uint(v.y) & 0xffffe000u),
                       __uint_as_float(__float_as_uint(v.z) & 0xffffe000u), __uint_as_float(__float_as_uint(v.w) & 0xffffe000u));
}

__device__ __forceinline__ void set_status(int *status, int code) { atomicCAS(status, DEV_OK, code); }
__device__ __forceinline__ bool aborted(const int *flag) { return *reinterpret_cast<const volatile int *>(flag) != 0; }

__device__ __forceinline__ int pad4(int n) { return (n + 3) & ~3; }

// One CTA of the product described by `a`; `cta` is its index in that
// product's grid (task-fastest: the tasks of a token tile run at about the
// same time, so their reads of the tile's X chunks meet in L2; tile-fastest
// read X from DRAM twice on 1024-wide fp32 16x16 weights, 107.6 -> 102.2 us).
template <typename T, int R>
__device__ __forceinline__ void tc_cta(const CUtensorMap &xmap, const TcArgs &a, unsigned cta) {
    ptx::pdl_launch_dependents();
    constexpr bool F32 = sizeof(T) == 4;
    constexpr int NS = TcCfg<T>::NS;
    constexpr int NISS = TcCfg<T>::NISS;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *base =
        reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(base + a.bar_off);
    uint64_t *empty = full + NS;
    uint64_t *split = empty + NS;    // fp32: the stage's high/low parts are ready
    uint64_t *done = split + NS;     // every MMA completed
    uint64_t *rbar = done + 1;       // task record landed
    int *misc = reinterpret_cast<int *>(base + a.misc_off);   // [0] abort flag, [1] TMEM address
    int *itab = misc + 4;                                     // per item: row p0 p1 slot - len
    unsigned char *W_s = base + a.w_off;
    int32_t *I_s = reinterpret_cast<int32_t *>(base + a.trec_smem);   // the task record
    float *B_s = reinterpret_cast<float *>(base + a.bias_off);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int task = (int)(cta % a.n_tasks);
    const int64_t n0 = (int64_t)(cta / a.n_tasks) * TN;
    const int32_t *trec = a.trec + __ldg(a.trec_off + task);
    const int g_count = __ldg(trec + 1);
    const int C = a.C, nch = a.nchunks;
    const int items_at = 4 + pad4(nch + 1);   // record layout: header, chunk starts, items, entries

    if (threadIdx.x == 0) {
        for (int s = 0; s < NS; s++) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], NISS);
            ptx::mbar_init(&split[s], 1);
        }
        ptx::mbar_init(done, NISS);
        ptx::mbar_init(rbar, 1);
        misc[0] = 0;
        ptx::fence_barrier_init();
    }
    if ((int)threadIdx.x < g_count) {
        const int g = threadIdx.x;
        const int4 it = __ldg(reinterpret_cast<const int4 *>(trec + items_at) + g);   // row, p0, p1, slot
        itab[6 * g + 0] = it.x;
        itab[6 * g + 1] = it.y;
        itab[6 * g + 2] = it.z;
        itab[6 * g + 3] = it.w;
        itab[6 * g + 4] = 0;
        itab[6 * g + 5] = it.z - it.y;
    }
    if (warp == 1) tc5::alloc(reinterpret_cast<uint32_t *>(&misc[1]), a.tmem_cols);
    tc5::fence_before();
    __syncthreads();
    tc5::fence_after();
    const uint32_t tmem = (uint32_t)misc[1];
    const uint32_t wblock = (uint32_t)R * C * (F32 ? 8 : 2);   // bytes of one block's B operand(s)

    if (warp == 0) {
        // ---------------- producer
        if (lane == 0) {
            ptx::prefetch_tensormap(&xmap);
            const int n_ent = __ldg(trec + 4 + nch);
            const uint32_t rec_bytes = (uint32_t)(items_at + 4 * g_count + pad4(n_ent)) * 4;
            ptx::mbar_arrive_expect_tx(rbar, rec_bytes);
            ptx::bulk_load(I_s, trec, rec_bytes, rbar);
            ptx::pdl_wait();   // X may be an earlier kernel's output
            const unsigned char *wsrc = static_cast<const unsigned char *>(a.wpk);
            int k = 0;          // ring slots used (chunks with work, in order)
            int stalled = -1;   // test hook: the slot left empty
            bool ok = ptx::mbar_wait_bounded(rbar, 0, a.wait_ns);   // chunk starts, from shared memory
            const int64_t wfirst = ok ? I_s[0] : 0;                   // the task's first packed block
            for (int c = 0; ok && c < nch; c++) {
                const int lo = I_s[4 + c], hi = I_s[5 + c];
                if (lo == hi) continue;   // no block of this task in chunk c
                const int s = k % NS;
                if (k >= NS && !ptx::mbar_wait_bounded(&empty[s], ((k / NS) - 1) & 1, a.wait_ns)) {
                    ok = false;
                    break;
                }
                if (aborted(misc)) { ok = false; break; }
                if (c == a.stall_chunk) {   // never loaded: its consumer times out
                    stalled = k++;
                    continue;
                }
                // the X chunk and, beside it, the task's block values for this chunk
                const uint32_t wbytes = (uint32_t)(hi - lo) * wblock;
                ptx::mbar_arrive_expect_tx(&full[s], kStageBytes + wbytes);
                ptx::tma_load_2d(base + s * kStageBytes, &xmap, c * TcCfg<T>::KC, (int32_t)n0, &full[s]);
                ptx::bulk_load(W_s + s * a.wstage, wsrc + (wfirst + lo) * wblock, wbytes, &full[s]);
                k++;
            }
            if (!ok) {
                set_status(a.status, DEV_TIMEOUT);
                atomicExch(&misc[0], 1);
            }
            for (int d = max(0, k - NS); d < k; d++)
                if (d != stalled) ptx::mbar_wait_bounded(&full[d % NS], (d / NS) & 1, kDrainNs);
            ptx::mbar_wait_bounded(rbar, 0, kDrainNs);
        }
    } else if (warp <= NISS) {
        // ---------------- MMA issuers: lane 0 of warps 1..NISS, each over a
        // contiguous range of the task's items (its accumulators), ranges
        // balanced by block count; every issuer walks every chunk and
        // commits the stage, so `empty` and `done` count NISS arrivals
        if (lane == 0) {
            const int q = warp - 1;
            int i0 = 0, i1 = 0;
            {
                int total = 0;
                for (int g = 0; g < g_count; g++) total += itab[6 * g + 5];
                int acc = 0;
                i0 = g_count;
                for (int g = 0; g < g_count; g++) {
                    const int len = itab[6 * g + 5];
                    const int owner =
                        total > 0 ? min(NISS - 1, (int)((int64_t)(2 * acc + len) * NISS / (2 * (int64_t)total))) : 0;
                    acc += len;
                    if (owner == q) {
                        i0 = min(i0, g);
                        i1 = g + 1;
                    }
                }
                if (i1 == 0) i0 = 0;
            }
            const uint32_t ufirst = (uint32_t)i0, ucnt = (uint32_t)(i1 - i0);
            bool ok = ptx::mbar_wait_bounded(rbar, 0, a.wait_ns) && !aborted(misc);
            const int32_t *ent = I_s + items_at + 4 * g_count;
            int k = 0;   // chunks consumed
            for (int c = 0; ok && c < nch; c++) {
                const int lo = I_s[4 + c], hi = I_s[5 + c];
                if (lo == hi) continue;
                const int s = k % NS;
                // fp32: wait for the split parts (the split warps waited for the copy)
                if (!ptx::mbar_wait_bounded(F32 ? &split[s] : &full[s], (k / NS) & 1, a.wait_ns) || aborted(misc)) {
                    ok = false;
                    break;
                }
                tc5::fence_after();
                const uint32_t stage = ptx::smem_addr(base + s * kStageBytes);
                const uint32_t w_stage = ptx::smem_addr(W_s + s * a.wstage);
                // descriptors of the stage's first A row and first B block: an
                // operand's descriptor is these plus its byte offset / 16 in the
                // address field (no carry out: shared addresses stay below 256 KB)
                const uint64_t a0 = tc5::desc_sw128(stage), b0 = tc5::desc(w_stage, 128, 256);
                const uint32_t wb16 = wblock >> 4;
                int e = lo;
                if constexpr (!F32 && NISS == 1) {
                    if (C == 16) {
                        // one issuer, one MMA per block: read and decode 4
                        // entries, then issue their MMAs back to back (one
                        // thread issues, so the decoding would otherwise sit
                        // between MMAs)
                        constexpr uint32_t idesc = tc5::idesc(false, TN, R);
                        for (; e + 4 <= hi; e += 4) {
                            const uint32_t vv[4] = {(uint32_t)ent[e], (uint32_t)ent[e + 1], (uint32_t)ent[e + 2],
                                                    (uint32_t)ent[e + 3]};
                            uint64_t adv[4], bdv[4];
                            uint32_t dv[4], acc[4];
#pragma unroll
                            for (int jj = 0; jj < 4; jj++) {
                                adv[jj] = a0 + (uint64_t)((vv[jj] & 3u) * 2u);
                                bdv[jj] = b0 + (uint64_t)((uint32_t)(e + jj - lo) * wb16);
                                dv[jj] = tmem + ((vv[jj] >> 2) & 31u) * R;
                                acc[jj] = ((vv[jj] >> 7) & 1u) == 0u;
                            }
#pragma unroll
                            for (int jj = 0; jj < 4; jj++) tc5::mma_ss<false>(dv[jj], adv[jj], bdv[jj], idesc, acc[jj]);
                        }
                    }
                }
                for (; ucnt > 0 && e < hi; e++) {
                    const uint32_t v = (uint32_t)ent[e];
                    const uint32_t g = (v >> 2) & 31u, first = (v >> 7) & 1u;
                    const uint64_t ad = a0 + (uint64_t)((v & 3u) * 2u);             // + (v & 3) * 32 bytes
                    const uint64_t bd = b0 + (uint64_t)((uint32_t)(e - lo) * wb16);
                    if constexpr (!F32) {
                        if ((v >> 9) & 1u) continue;   // a stack member: its rows are in its head's MMAs
                        if ((v >> 8) & 1u) {
                            // a stack head: the B operand of all g_count items'
                            // blocks; this issuer's items are rows ufirst*R ..
                            // of it, into their adjacent accumulators
                            const uint32_t ns = (uint32_t)(g_count * R);
                            const uint32_t idesc_s = tc5::idesc(false, TN, (int)(ucnt * R));
                            const uint64_t bs = bd + (uint64_t)(ufirst * R * 2);   // ufirst * R rows of 32 bytes
#pragma unroll 4
                            for (int sl = 0; sl < C / 16; sl++)
                                tc5::mma_ss<false>(tmem + ufirst * R, ad + (uint64_t)(sl * 2), bs + (uint64_t)(sl * ns * 2),
                                         idesc_s, (first == 0u) | (sl > 0));
                            continue;
                        }
                    }
                    if (g - ufirst >= ucnt) continue;   // another issuer's item
                    const uint32_t d = tmem + g * R;
                    if constexpr (F32) {
                        // 3xTF32: high x high + high x low + low x high, K = 8 per MMA
                        constexpr uint32_t idesc = tc5::idesc(true, TN, R);
                        const uint64_t adl = ad + (uint64_t)(NS * kStageBytes >> 4), bdl = bd + (uint64_t)((uint32_t)R * C * 4 >> 4);
#pragma unroll 2
                        for (int sl = 0; sl < C / 8; sl++) {
                            const uint64_t ka = (uint64_t)(sl * 2), kb = (uint64_t)(sl * (R * 2));   // 32 and R*32 bytes
                            tc5::mma_ss<true>(d, ad + ka, bd + kb, idesc, (first == 0u) | (sl > 0));
                            tc5::mma_ss<true>(d, ad + ka, bdl + kb, idesc, 1u);
                            tc5::mma_ss<true>(d, adl + ka, bd + kb, idesc, 1u);
                        }
                    } else {
                        constexpr uint32_t idesc = tc5::idesc(false, TN, R);
#pragma unroll 4
                        for (int sl = 0; sl < C / 16; sl++)
                            tc5::mma_ss<false>(d, ad + (uint64_t)(sl * 2), bd + (uint64_t)(sl * (R * 2)), idesc,
                                     (first == 0u) | (sl > 0));
                    }
                }
                tc5::commit(&empty[s]);   // the stage is free once every issuer's MMAs completed
                k++;
            }
            if (!ok) {
                set_status(a.status, DEV_TIMEOUT);
                atomicExch(&misc[0], 1);
            }
            tc5::commit(done);   // every MMA this issuer issued completes before its `done` arrival
        }
    } else {
        // ---------------- the last four warps: fp32 split during the main
        // loop, then the epilogue; TMEM lane quarter = warp % 4
        const int et = threadIdx.x - 32 * (1 + NISS);   // 0..127
        ptx::pdl_wait();   // the bias, Y and the workspace may be an earlier kernel's
        for (int e = et; e < g_count * R; e += 128) {
            const int g = e / R, r = e - g * R;
            B_s[e] = a.bias ? __ldg(a.bias + (int64_t)itab[6 * g + 0] * R + r) : 0.f;
        }
        bool split_ok = true;
        if constexpr (F32) {
            // x = high + low per element of every loaded stage: the low part
            // into the stage's twin buffer (same swizzled layout); the high
            // part is the stage itself, since kind::tf32 MMAs use only the
            // top 19 bits of each fp32 element (round-to-nearest would leave
            // about 2^-11 relative error per product, far outside the fp32
            // tolerance the parity tests check)
            split_ok = ptx::mbar_wait_bounded(rbar, 0, a.wait_ns);
            int k = 0;
            for (int c = 0; split_ok && c < nch; c++) {
                if (I_s[4 + c] == I_s[5 + c]) continue;
                const int s = k % NS;
                const bool got = ptx::mbar_wait_bounded(&full[s], (k / NS) & 1, a.wait_ns) && !aborted(misc);
                if (ptx::named_barrier_or(2, 128, !got)) { split_ok = false; break; }
                float4 *hi4 = reinterpret_cast<float4 *>(base + s * kStageBytes);
                float4 *lo4 = reinterpret_cast<float4 *>(base + (NS + s) * kStageBytes);
#pragma unroll
                for (int j = 0; j < (int)(kStageBytes / 16 / 128); j++) {
                    const int q4 = et + 128 * j;
                    const float4 x = hi4[q4];
                    const float4 h = tf32_high(x);
                    lo4[q4] = make_float4(x.x - h.x, x.y - h.y, x.z - h.z, x.w - h.w);
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // visible to the tensor cores
                ptx::named_barrier(2, 128);
                if (et == 0) ptx::mbar_arrive(&split[s]);
                k++;
            }
            if (!split_ok && et == 0) {
                set_status(a.status, DEV_TIMEOUT);
                atomicExch(&misc[0], 1);
            }
        }
        ptx::named_barrier(1, 128);
        // the last commit fires after the whole main loop: allow it every chunk's bound
        const uint64_t limit = a.wait_ns * (uint64_t)(nch + 2);
        const bool got = ptx::mbar_wait_bounded_idle(done, 0, limit);   // the whole main loop: sleep while waiting
        tc5::fence_after();
        const bool stop = ptx::named_barrier_or(1, 128, !got || !split_ok || aborted(misc));
        if (!got && et == 0) set_status(a.status, DEV_TIMEOUT);
        const int q = warp & 3;
        const int t = 32 * q + lane;   // this thread's token row in the tile
        const int64_t n = n0 + t;
        const uint32_t lane_base = tmem + ((uint32_t)(32 * q) << 16);
        // Every MMA has completed, so the X ring is idle: it stages Y in
        // 16-column groups [128 tokens x 16 columns] that one thread stores by
        // TMA (rows past N are not written), rounds of 64 accumulator columns
        // alternating between two buffers. Split items write their fp32
        // partials to the workspace directly.
        constexpr uint32_t kGroupBytes = TN * 16 * sizeof(T);
        constexpr uint32_t kRoundBytes = 4 * kGroupBytes;
        static_assert(2 * kRoundBytes <= (F32 ? 2 : 1) * NS * kStageBytes, "Y staging exceeds the X ring");
        int round = 0;
        for (int c0 = 0; c0 < g_count * R && !stop; c0 += 64, round++) {
            unsigned char *buf = base + (round & 1) * kRoundBytes;
            if (round >= 2) {   // the stores issued from this buffer two rounds ago have read it
                if (et == 0) ptx::bulk_wait_group_read<1>();
                ptx::named_barrier(1, 128);
            }
            uint32_t r0[32], r1[32];
            tc5::ld32(lane_base + c0, r0);
            if (c0 + 32 < g_count * R) tc5::ld32(lane_base + c0 + 32, r1);
            tc5::ld_wait();
#pragma unroll
            for (int h = 0; h < 64; h += 16) {
                const int col = c0 + h;
                if (col >= g_count * R) break;
                const int g = col / R, hr = col - g * R;
                const int len = itab[6 * g + 5], slot = itab[6 * g + 3];
                float v[16];
#pragma unroll
                for (int j = 0; j < 16; j++) v[j] = len > 0 ? __uint_as_float(h < 32 ? r0[h + j] : r1[h - 32 + j]) : 0.f;
                if (slot < 0) {
                    // staged rows in the Y map's swizzled order (64-byte fp32 rows:
                    // 16-byte group j of row t at j ^ ((t / 2) % 4); 32-byte bf16
                    // rows: j ^ ((t / 4) % 2)), so a warp's stores spread over
                    // all banks; the TMA store writes Y's rows in plain order
                    unsigned char *row = buf + (h / 16) * kGroupBytes + t * 16 * (int)sizeof(T);
                    if constexpr (F32) {
                        float4 *dst = reinterpret_cast<float4 *>(row);
                        const int sw = (t >> 1) & 3;
#pragma unroll
                        for (int j = 0; j < 4; j++)
                            dst[j ^ sw] = make_float4(v[4 * j] + B_s[col + 4 * j], v[4 * j + 1] + B_s[col + 4 * j + 1],
                                                 v[4 * j + 2] + B_s[col + 4 * j + 2], v[4 * j + 3] + B_s[col + 4 * j + 3]);
                    } else {
                        uint32_t pk[8];
#pragma unroll
                        for (int j = 0; j < 8; j++) {
                            const float lo = v[2 * j] + B_s[col + 2 * j];
                            const float hi = v[2 * j + 1] + B_s[col + 2 * j + 1];
                            pk[j] = (uint32_t)from_f32<uint16_t>(lo) | ((uint32_t)from_f32<uint16_t>(hi) << 16);
                        }
                        uint4 *dst = reinterpret_cast<uint4 *>(row);
                        const int sw = (t >> 2) & 1;
                        dst[sw] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                        dst[1 ^ sw] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
                    }
                } else if (n < a.N) {
                    float4 *dst = reinterpret_cast<float4 *>(a.ws + ((int64_t)slot * a.N + n) * R + hr);
#pragma unroll
                    for (int j = 0; j < 4; j++) dst[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                }
            }
            ptx::fence_proxy_async_smem();   // the staged rows, visible to the TMA unit
            ptx::named_barrier(1, 128);
            if (et == 0) {
                for (int h = 0; h < 64; h += 16) {
                    const int col = c0 + h;
                    if (col >= g_count * R) break;
                    const int g = col / R, hr = col - g * R;
                    if (itab[6 * g + 3] >= 0) continue;
                    ptx::tma_store_2d(&a.ymap, buf + (h / 16) * kGroupBytes, itab[6 * g + 0] * R + hr, (int32_t)n0);
                }
                ptx::bulk_commit_group();
            }
        }
        if (et == 0) ptx::bulk_wait_group_all();   // no store outlives the CTA's shared memory
    }
    // ---------------- teardown: every MMA completed (the epilogue waited for
    // `done`, or the issuer never started), then free the tensor memory
    tc5::fence_before();
    __syncthreads();
    if (warp == 1) {
        tc5::fence_after();
        tc5::dealloc(tmem, a.tmem_cols);
    }
}

template <typename T, int R>
__global__ void __launch_bounds__(TcCfg<T>::NTHREADS, 2)
k_tc(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ TcArgs a) {
    tc_cta<T, R>(xmap, a, blockIdx.x);
}

// Several products sharing X in one grid: product h owns CTAs start[h] ..
// start[h+1]-1, with its own arguments (the launch gives every CTA the
// largest shared memory of the group).
struct TcBatch {
    int n;
    unsigned start[kTcBatchMax + 1];
    TcArgs args[kTcBatchMax];
};

template <typename T, int R>
__global__ void __launch_bounds__(TcCfg<T>::NTHREADS, 2)
k_tc_batch(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ TcBatch b) {
    int h = 0;
    while (h + 1 < b.n && blockIdx.x >= b.start[h + 1]) h++;
    tc_cta<T, R>(xmap, b.args[h], blockIdx.x - b.start[h]);
}

// Block values into the MMA's B operand layout (K-major, no swizzle): for each
// K-slice of 16 columns, 8-row x 16-byte core matrices, 128 bytes apart along
// K and 256 bytes apart along the rows.
// Packed block i holds stored block order[i]; stack[i] = (g << 16) | m puts it
// at rows g*R .. g*R+R-1 of an operand of m*R rows that starts at packed
// block i - g (m = 1: a block of its own).
__global__ void k_pack_tc(const uint16_t *__restrict__ data, const int32_t *__restrict__ order,
                          const int32_t *__restrict__ stack, uint16_t *__restrict__ out, int64_t n, int R, int C) {
    const int64_t total = n * R * C;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = e / ((int64_t)R * C);
        const int rc = (int)(e - p * R * C);
        const int n0 = rc / C, k = rc - n0 * C;
        const int sw = stack[p], g = sw >> 16, m = sw & 0xffff;
        const int RS = m * R, n_ = g * R + n0;   // rows of the operand, this row in it
        const int64_t dst =
            (p - g) * R * C + (k >> 4) * (RS * 16) + (n_ >> 3) * 128 + ((k & 15) >> 3) * 64 + (n_ & 7) * 8 + (k & 7);
        out[dst] = data[(int64_t)order[p] * R * C + rc];
    }
}

// fp32 block values as two tf32 B operands, high part then low part, each in
// the layout above with 8-column K-slices of 8-row x 16-byte core matrices.
__global__ void k_pack_tc_f32(const float *__restrict__ data, const int32_t *__restrict__ order,
                              float *__restrict__ out, int64_t n, int R, int C) {
    const int64_t total = n * R * C;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = e / ((int64_t)R * C);
        const int rc = (int)(e - p * R * C);
        const int n_ = rc / C, k = rc - n_ * C;
        const int64_t at = p * R * C * 2 + (k >> 3) * (R * 8) + (n_ >> 3) * 64 + ((k & 7) >> 2) * 32 + (n_ & 7) * 4 + (k & 3);
        const float w = data[(int64_t)order[p] * R * C + rc];
        const float h = __uint_as_float(__float_as_uint(w) & 0xffffe000u);
        out[at] = h;
        out[at + (int64_t)R * C] = w - h;
    }
}

// Narrow bf16 blocks into zero-filled R x 64 tiles: element (r, c) of stored
// block p goes to tile vmap[p] / 64, row r, column vmap[p] % 64 + c.
__global__ void k_reblock(const uint16_t *__restrict__ data, const int32_t *__restrict__ vmap, int64_t nnzb, int R,
                          int C, uint16_t *__restrict__ tiles) {
    const int64_t total = nnzb * R * C;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = e / ((int64_t)R * C);
        const int rc = (int)(e - p * R * C);
        const int r = rc / C, c = rc - r * C;
        tiles[(int64_t)vmap[p] + r * 64 + c] = data[e];   // vmap: offset of the block's (0, 0) in the tiles
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

// Y [N, M] for the epilogue's TMA stores: boxes of 16 columns x 128 token rows,
// with the swizzle of the row size (64 bytes fp32, 32 bytes bf16) in which
// the epilogue stages them.
template <typename T>
cudaError_t encode_y(void *Y, int64_t N, int64_t M, CUtensorMap *map) {
    auto enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const cuuint64_t dims[2] = {(cuuint64_t)M, (cuuint64_t)N};
    const cuuint64_t strides[1] = {(cuuint64_t)M * sizeof(T)};
    const cuuint32_t box[2] = {16, (cuuint32_t)TN};
    const cuuint32_t estr[2] = {1, 1};
    if (enc(map, sizeof(T) == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, Y, dims,
            strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            sizeof(T) == 4 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    return cudaSuccess;
}

uint32_t tmem_cols_for(int cols) {
    uint32_t n = 32;
    while ((int)n < cols) n <<= 1;
    return n;
}

// Kernel arguments and dynamic shared-memory bytes of one product at task
// size G (nothing to launch: smem = 0).
template <typename T, int R>
cudaError_t make_tc_args(const LaunchArgs &la, int G, TcArgs &a, uint32_t &smem) {
    constexpr int NS = TcCfg<T>::NS, KC = TcCfg<T>::KC;
    const Schedule &sc = *la.sc;
    const int n_items = (int)sc.items.size();
    smem = 0;
    if (n_items == 0 || la.N == 0) return cudaSuccess;
    const int gidx = tc_g_index(G);
    a.G = G;
    a.n_tasks = (int)sc.tc.rec_off[gidx].size();
    a.trec = sc.tc.d_rec[gidx];
    a.trec_off = sc.tc.d_rec_off[gidx];
    if (sc.tc.w_off[gidx] < 0) return cudaErrorInvalidConfiguration;
    a.wpk = static_cast<const unsigned char *>(la.data) + sc.tc.w_off[gidx];
    a.wstage = (uint32_t)sc.tc.task_wbytes[gidx];
    a.bias = la.bias;
    a.Y = la.Y;
    a.ws = la.ws;
    a.status = la.status;
    a.N = la.N;
    a.K = sc.K;
    a.M = sc.M;
    a.C = sc.ex_C;   // the execution block width (64 for re-blocked narrow blocks)
    a.nchunks = (int)((sc.K + KC - 1) / KC);
    a.w_off = (sizeof(T) == 4 ? 2 : 1) * NS * kStageBytes;
    a.trec_smem = a.w_off + NS * a.wstage;
    a.bias_off = a.trec_smem + (uint32_t)((sc.tc.task_ibytes[gidx] + 15) & ~size_t(15));
    a.bar_off = a.bias_off + (uint32_t)(((size_t)G * R * 4 + 15) & ~size_t(15));
    a.misc_off = a.bar_off + (3 * NS + 2) * 8;
    a.tmem_cols = tmem_cols_for(G * R);
    a.wait_ns = la.wait_ns;
    a.stall_chunk = la.stall_chunk;
    smem = a.misc_off + (4 + 6 * 32) * 4 + 1024;
    if (smem > (uint32_t)kTcMaxSmem || G * R > kTcTmemCols) return cudaErrorInvalidConfiguration;
    return encode_y<T>(la.Y, la.N, sc.M, &a.ymap);
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

template <typename T>
cudaError_t encode_x(const void *X, int64_t N, int64_t K, CUtensorMap *map) {
    auto enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)N};
    const cuuint64_t strides[1] = {(cuuint64_t)K * sizeof(T)};
    const cuuint32_t box[2] = {(cuuint32_t)TcCfg<T>::KC, (cuuint32_t)TN};
    const cuuint32_t estr[2] = {1, 1};
    if (enc(map, sizeof(T) == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
            const_cast<void *>(X), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) !=
        CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    return cudaSuccess;
}

// n products sharing X (same dtype, R, K, N and stream): n == 1 the plain
// launch, n > 1 one fused grid.
template <typename T, int R>
cudaError_t launch_r(const LaunchArgs *las, const int *Gs, int n) {
    const int64_t n_tiles = (las[0].N + TN - 1) / TN;
    CUtensorMap map;
    if (n == 1) {
        TcArgs a;
        uint32_t smem = 0;
        cudaError_t e = make_tc_args<T, R>(las[0], Gs[0], a, smem);
        if (e != cudaSuccess || smem == 0) return e;
        static std::atomic<uint64_t> attr_set{0};
        if ((e = allow_smem(k_tc<T, R>, attr_set)) != cudaSuccess) return e;
        if ((e = encode_x<T>(las[0].X, las[0].N, las[0].sc->K, &map)) != cudaSuccess) return e;
        const int64_t grid = n_tiles * a.n_tasks;   // task-fastest order
        if (grid > INT32_MAX) return cudaErrorInvalidConfiguration;
        return launch_kernel(k_tc<T, R>, dim3((unsigned)grid), dim3(TcCfg<T>::NTHREADS), smem, las[0].stream, map, a);
    }
    if (n > kTcBatchMax) return cudaErrorInvalidValue;
    TcBatch b;
    b.n = 0;
    uint32_t smem_max = 0;
    int64_t grid = 0;
    for (int i = 0; i < n; i++) {
        uint32_t smem = 0;
        cudaError_t e = make_tc_args<T, R>(las[i], Gs[i], b.args[b.n], smem);
        if (e != cudaSuccess) return e;
        if (smem == 0) continue;
        b.start[b.n] = (unsigned)grid;
        grid += n_tiles * b.args[b.n].n_tasks;
        smem_max = std::max(smem_max, smem);
        b.n++;
    }
    if (b.n == 0) return cudaSuccess;
    if (grid > INT32_MAX) return cudaErrorInvalidConfiguration;
    b.start[b.n] = (unsigned)grid;
    static std::atomic<uint64_t> attr_set_b{0};
    cudaError_t e = allow_smem(k_tc_batch<T, R>, attr_set_b);
    if (e != cudaSuccess) return e;
    if ((e = encode_x<T>(las[0].X, las[0].N, las[0].sc->K, &map)) != cudaSuccess) return e;
    return launch_kernel(k_tc_batch<T, R>, dim3((unsigned)grid), dim3(TcCfg<T>::NTHREADS), smem_max, las[0].stream, map, b);
}

}  // namespace

bool tc_supports(int R, int C, bsr_dtype_t dt, int64_t K, int64_t MK) {
    const bool r_ok = R == 16 || R == 32 || R == 64 || R == 128;
    if (dt == BSR_BF16) return r_ok && (C == 16 || C == 32 || C == 64) && K % 8 == 0 && K > 0;
    // fp32 as 3xTF32; a block lies inside one 32-column stage. Blocks of 32
    // or more rows always; 16-row blocks on weights of at least 2^20
    // elements, where a call carries enough work to pay for the split stages
    // (measured: 1024 x 1024 at 90% and 16384 tokens, 117 us against the
    // SIMT kernel's 180 us; 768 x 768 at 80% and 1024 tokens, 28 us against
    // 25 us). BSR_TC_F32_R16=1 takes every 16-row weight, =0 none.
    static const int r16 = [] {
        const char *v = getenv("BSR_TC_F32_R16");
        return v && *v ? atoi(v) : -1;
    }();
    const bool r16_ok = r16 == 1 || (r16 != 0 && MK >= ((int64_t)1 << 20));
    return ((R >= 32 || (R == 16 && r16_ok)) && r_ok) && (C == 16 || C == 32) && K % 4 == 0 && K > 0;
}

int tc_g_index(int G) {
    for (int i = 0; i < kTcTaskSizes; i++)
        if (kTcG[i] == G) return i;
    return 0;
}

size_t tc_smem_bytes(int R, int G, size_t wstage, size_t ibytes, bsr_dtype_t dt) {
    const size_t ring = dt == BSR_F32 ? (size_t)2 * kTcStagesF32 * kStageBytes : (size_t)kTcStages * kStageBytes;
    const int ns = dt == BSR_F32 ? kTcStagesF32 : kTcStages;
    return ring + ns * ((wstage + 15) & ~size_t(15)) + ((ibytes + 15) & ~size_t(15)) +
           (((size_t)G * R * 4 + 15) & ~size_t(15)) + (3 * ns + 2) * 8 + (4 + 6 * 32) * 4 + 1024;
}

int tc_ctas_per_sm(int R, int G, size_t wbytes, size_t ibytes, bsr_dtype_t dt) {
    constexpr size_t kSmemPerSm = 233472;   // 228 KB, of which 1 KB is reserved per CTA
    const size_t per_cta = tc_smem_bytes(R, G, wbytes, ibytes, dt) + 1024;
    const int by_smem = (int)(kSmemPerSm / per_cta);
    const int by_tmem = kTcTmemCols / (int)tmem_cols_for(G * R);
    const int bound = 2;   // the kernel's __launch_bounds__
    return std::max(1, std::min(bound, std::min(by_smem, by_tmem)));
}

cudaError_t pack_tc_data(const void *data, bsr_dtype_t dt, const int32_t *order, const int32_t *stack, int64_t n,
                         int R, int C, void *out, cudaStream_t s) {
    const int64_t total = n * R * C;
    if (total == 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>((total + 255) / 256, 1 << 20);
    if (dt == BSR_F32)
        k_pack_tc_f32<<<grid, 256, 0, s>>>(static_cast<const float *>(data), order, static_cast<float *>(out), n, R, C);
    else
        k_pack_tc<<<grid, 256, 0, s>>>(static_cast<const uint16_t *>(data), order, stack, static_cast<uint16_t *>(out), n,
                                       R, C);
    return cudaGetLastError();
}

cudaError_t reblock_tc_data(const uint16_t *data, const int32_t *vmap, int64_t nnzb, int R, int C, uint16_t *tiles,
                            cudaStream_t s) {
    const int64_t total = nnzb * R * C;
    if (total == 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>((total + 255) / 256, 1 << 20);
    k_reblock<<<grid, 256, 0, s>>>(data, vmap, nnzb, R, C, tiles);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_tc_t(const LaunchArgs *las, const int *Gs, int n) {
    switch (las[0].sc->ex_R) {
        case 16: return launch_r<T, 16>(las, Gs, n);
        case 32: return launch_r<T, 32>(las, Gs, n);
        case 64: return launch_r<T, 64>(las, Gs, n);
        case 128: return launch_r<T, 128>(las, Gs, n);
    }
    return cudaErrorNotSupported;
}

cudaError_t launch_tc(const LaunchArgs &la, int G) {
    return la.sc->dt == BSR_F32 ? launch_tc_t<float>(&la, &G, 1) : launch_tc_t<uint16_t>(&la, &G, 1);
}

cudaError_t tc_encode_x(bsr_dtype_t dt, const void *X, int64_t N, int64_t K, CUtensorMap *map) {
    return dt == BSR_F32 ? encode_x<float>(X, N, K, map) : encode_x<uint16_t>(X, N, K, map);
}

int tc_fusion_key(const Schedule &sc) { return (int)sc.dt * 1024 + sc.ex_R; }

cudaError_t launch_tc_batch(const LaunchArgs *las, const int *Gs, int n) {
    if (n <= 0) return cudaSuccess;
    if (n > kTcBatchMax) return cudaErrorInvalidValue;
    return las[0].sc->dt == BSR_F32 ? launch_tc_t<float>(las, Gs, n) : launch_tc_t<uint16_t>(las, Gs, n);
}

}  // namespace bsr
