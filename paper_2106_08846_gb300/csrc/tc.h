// Parameters shared by the tcgen05 kernel and the schedule that feeds it.
#pragma once

#include <cuda.h>

#include <cstddef>
#include <cstdint>
#include <vector>

#include "bsr.h"

namespace bsr {

constexpr int kTcTokens = 128;         // tokens per CTA = MMA M = TMEM lanes
constexpr int kTcChunk = 64;           // K columns per ring stage (one 128-byte swizzle row of bf16)
constexpr int kTcStages = 3;           // ring depth (bf16; two CTAs per SM)
constexpr int kTcStagesF32 = 2;        // ring depth (fp32: each stage has a twin for the low parts; two
                                       // stages let two CTAs share an SM and overlap their stage latencies)
constexpr int kTcMaxSmem = 232448;     // 227 KB
constexpr int kTcpIssuers = 4;         // MMA-issuing threads of the persistent kernel (one per warp)
constexpr int kTcpProgHeader = 16;     // ints before a stage program's MMAs: per issuer its first MMA, and the end
// Warps issuing MMAs in the tc kernel: the issue rate grows with the issuing
// warps, which pays for fp32 (three MMAs per K slice); bf16 keeps one issuer
// (measured faster on 16 x 16 blocks, where a second issuer's entry scans
// cost more than its MMAs save).
constexpr int tc_issuers(bool f32) { return f32 ? 4 : 1; }
constexpr int tc_threads(bool f32) { return 32 * (1 + tc_issuers(f32) + 4); }   // producer, issuers, split/epilogue
constexpr int kTcBatchMax = 64;        // products in one fused launch (bsr_spmm_batch)
constexpr int kTcpStagesMax = 8;       // ring stages of the persistent kernel (fewer when they do not fit)
constexpr int kTcTmemCols = 512;       // accumulator columns per SM
constexpr int kTcTaskSizes = 6;
constexpr int kTcG[kTcTaskSizes] = {1, 2, 4, 8, 16, 32};

// Per task size G: the task records the kernel bulk-copies (see below), the
// W stage (largest block-value footprint of one task's chunk) and record
// footprints, and the order in which the block values of all tasks are
// packed for G: task by task, chunk by chunk, in entry order, so that the
// values one chunk of one task needs are one contiguous range (streamed
// through a ring beside X instead of held for the whole kernel).
struct TcPlan {
    size_t task_wbytes[kTcTaskSizes] = {};   // W ring stage bytes
    size_t task_ibytes[kTcTaskSizes] = {};
    int64_t task_cost_max[kTcTaskSizes] = {};     // MMA cost of the most loaded task (units: one N <= 64 MMA)
    int64_t stacks[kTcTaskSizes] = {};            // stacked chunks over all tasks
    std::vector<int32_t> rec[kTcTaskSizes];       // all task records of this G
    std::vector<int32_t> rec_off[kTcTaskSizes];   // per task: offset (ints, multiple of 4)
    std::vector<int32_t> worder[kTcTaskSizes];    // per packed block: the (execution) block it holds
    std::vector<int32_t> wstack[kTcTaskSizes];    // per packed block: (its row group in a stack << 16) | stack size
    int64_t w_off[kTcTaskSizes] = {};             // byte offset of G's packed values (-1: G not usable)
    size_t tcp_wbytes[kTcTaskSizes] = {};         // largest block-value footprint of one task's persistent-kernel
                                                  // stage (tcp_stage_chunks consecutive chunks)
    // Persistent kernel: per task and stage a program of ready MMAs (see
    // tcp_plan); per task, per stage (program offset / 16, program bytes)
    std::vector<uint32_t> prog[kTcTaskSizes];
    std::vector<int32_t> stab[kTcTaskSizes];
    int stab_ints = 0;                            // ints of one task's stage table (a multiple of 4)
    size_t tcp_pbytes[kTcTaskSizes] = {};         // largest stage program
    uint32_t *d_prog[kTcTaskSizes] = {};
    int32_t *d_stab[kTcTaskSizes] = {};
    int32_t *d_rec[kTcTaskSizes] = {};
    int32_t *d_rec_off[kTcTaskSizes] = {};
    int32_t *d_worder[kTcTaskSizes] = {};
    int32_t *d_wstack[kTcTaskSizes] = {};
};

// A task record (int32): [ the task's first packed block, its item count g,
// 0, 0 | per K chunk c = 0..nchunks the index of the chunk's first entry,
// padded to 4 | per item (row, p0, p1, slot) | one entry per MMA-block,
// chunk by chunk, padded to 4 ]. Entry e uses packed block (first + e).
// Entry bits: [0,2) stage column offset / 32 bytes, [2,7) item in the task,
// 7 first block of its item, 8 stack head, 9 stack member. A stack is a chunk
// in which every item of the task has exactly one block, at the same column
// offset, all first or all not first (bf16 blocks of 32 or more columns): its
// g blocks are packed as one B operand of g * R rows, and the head's MMAs
// (N = g * R, into the accumulators of items 0..g-1, which are adjacent)
// replace the members'.
inline int64_t tc_pad4(int64_t n) { return (n + 3) & ~int64_t(3); }

// Block shapes the tensor-core kernels run; MK: the weight's elements (M K).
bool tc_supports(int R, int C, bsr_dtype_t dt, int64_t K, int64_t MK);
int tc_g_index(int G);
size_t tc_smem_bytes(int R, int G, size_t wbytes, size_t ibytes, bsr_dtype_t dt);
// CTAs of the tensor-core kernel that fit one SM at once (shared memory,
// tensor memory and the kernel's launch bound), for a task size's footprint.
int tc_ctas_per_sm(int R, int G, size_t wbytes, size_t ibytes, bsr_dtype_t dt);
// Chunks per stage of the persistent kernel: 128 bf16 or 64 fp32 columns
// (an fp32 stage fills 128 tensor-memory columns with its high and low
// parts).
constexpr int kTcpStageChunks = 2;
inline int tcp_stage_chunks(bsr_dtype_t) { return kTcpStageChunks; }
// K columns per ring stage: one 128-byte swizzle row (64 bf16 or 32 fp32)
inline int tc_chunk_cols(bsr_dtype_t dt) { return dt == BSR_F32 ? 32 : 64; }
// bytes of one block's B operand(s): bf16, or fp32 high and low tf32 parts
// Stage programs of the persistent kernel, built from the task records for
// every usable task size: per stage a header of kTcpProgHeader ints (issuer
// q's MMAs are [h[q], h[q + 1])), then one 16-byte word per MMA: B offset in
// the stage's block values / 16, accumulator column, A operand (bit 31:
// accumulate; fp32: column in the stage's A slot in tensor memory; bf16:
// descriptor offset / 16 in the stage's X buffer), instruction descriptor. Issuer q owns a contiguous
// range of the task's items, balanced by block count.
void plan_tcp(struct Schedule &sc);
// The tensor map of X [N, K] both tensor-core kernels load from: boxes of
// 128 bytes x 128 token rows, 128-byte swizzle.
cudaError_t tc_encode_x(bsr_dtype_t dt, const void *X, int64_t N, int64_t K, CUtensorMap *map);
inline size_t tc_block_bytes(int R, int C, bsr_dtype_t dt) { return (size_t)R * C * (dt == BSR_F32 ? 8 : 2); }

}  // namespace bsr
