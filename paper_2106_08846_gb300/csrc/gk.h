// Parameters shared by the gathered-K tensor-core kernel ("gk") and the
// schedule that feeds it.
#pragma once

#include <algorithm>
#include <cstddef>
#include <cstdint>
#include <vector>

#include "bsr.h"

namespace bsr {

constexpr int kGkTokens = 128;         // tokens per CTA = MMA M = tensor-memory lanes
constexpr int kGkStages = 4;           // most X / W ring stages (fewer when they do not fit)
constexpr int kGkASlotsMax = 8;        // A operand buffers in tensor memory (batches in flight)
constexpr int kGkMaxSmem = 232448;     // 227 KB
constexpr int kGkTmemCols = 512;
constexpr int kGkTaskSizes = 5;
constexpr int kGkG[kGkTaskSizes] = {1, 2, 4, 8, 16};
constexpr int kGkEntryInts = 8;        // ints per (chunk, item) entry
constexpr int kGkIssuers = 4;          // MMA-issuing threads (one per warp): the issue rate grows with them

// K columns of X per ring stage: 32 KB of fp32 (64 columns) or bf16 (128).
inline int gk_chunk_cols(bsr_dtype_t dt) { return dt == BSR_F32 ? 64 : 128; }
// K of one MMA: 8 (tf32) or 16 (bf16).
inline int gk_kslice(bsr_dtype_t dt) { return dt == BSR_F32 ? 8 : 16; }

// Block shapes the kernel runs: R a multiple of 16 up to 128 (the MMA's N),
// C dividing the chunk (blocks never straddle a stage).
bool gk_supports(int R, int C, bsr_dtype_t dt, int64_t K);

// Per task size G (index gi): tasks of at most G block rows, balanced by
// work; per task a record, and the task's gathered block values chunk by
// chunk in the MMA's B layout.
//
// Record (int32): [ n_items, n_batches, first value byte / 16, record bytes |
// per chunk c = 0..nchunks: its first batch, padded to 4 | per chunk: its
// values' byte offset / 16 from the task's first, padded to 4 | per chunk:
// its MMA program's offset / 16 in the programs and its bytes, padded to 4
// | per batch
// b = 0..n_batches: its first entry, padded to 4 | per item (row, len, 0, 0)
// | entries, kGkEntryInts each: (item, first, A column in the batch's
// buffer, K slices, B byte offset in the chunk's values / 16, blocks, first
// column-list index, 0) | column list: per block of an entry, the byte offset
// of its first column in a stage at token row 0 (before the swizzle), padded
// to 4 ]. An entry gathers its item's blocks of one chunk into K = blocks x C
// columns, zero-padded to a multiple of the MMA's K; fp32 entries hold high
// then low tf32 parts (2 K columns of tensor memory), bf16 entries K / 2
// (pairs); an item's blocks in a chunk that need more A columns than one
// buffer holds are split into several entries (pieces). A batch is a run of
// one chunk's entries whose A columns fit one A buffer.
//
// A chunk's MMA program: per batch of the chunk and issuer q the start of
// its MMAs, then the end (padded to 4 ints), then one 16-byte word per MMA
// (batch-major, issuer-minor): B offset in the chunk's values / 16,
// accumulator column, A column in the batch's A buffer (bit 31:
// accumulate), instruction descriptor. Issuer q owns a contiguous range of
// the task's items, balanced by work.
struct GkPlan {
    bool ok = false;
    int64_t off[kGkTaskSizes] = {-1, -1, -1, -1, -1};    // byte offset of G's values in the packed buffer (-1: unusable)
    int64_t total_bytes = 0;                           // end of the gk region in the packed buffer
    int n_tasks[kGkTaskSizes] = {};
    uint32_t wstage[kGkTaskSizes] = {};                // bytes of one W stage (largest chunk of any task)
    uint32_t ibytes[kGkTaskSizes] = {};                // largest record
    uint32_t acols[kGkTaskSizes] = {};                 // tensor-memory columns of one A buffer (gk_slot_cols)
    int64_t cost_max[kGkTaskSizes] = {};               // MMAs of the most loaded task
    std::vector<int32_t> rec[kGkTaskSizes];
    std::vector<int32_t> rec_off[kGkTaskSizes];
    std::vector<int32_t> wsrc[kGkTaskSizes];           // per packed block slot: stored block (-1: zero padding)
    std::vector<int32_t> wslot[kGkTaskSizes];          // per packed block slot: (K row of its first column in
                                                       // its entry) | (entry K rows << 16), in packing order
    std::vector<int64_t> wbase[kGkTaskSizes];          // per packed block slot: byte offset of its entry's B operand
    std::vector<uint32_t> prog[kGkTaskSizes];          // chunk MMA programs of all tasks
    uint32_t pstage[kGkTaskSizes] = {};                // largest chunk program (bytes)
    int32_t *d_rec[kGkTaskSizes] = {};
    int32_t *d_rec_off[kGkTaskSizes] = {};
    int32_t *d_wsrc[kGkTaskSizes] = {};
    int32_t *d_wslot[kGkTaskSizes] = {};
    int64_t *d_wbase[kGkTaskSizes] = {};
    uint32_t *d_prog[kGkTaskSizes] = {};
};

// Shared memory of one CTA with the smallest ring (more than kGkMaxSmem: does not fit).
size_t gk_smem_bytes(bsr_dtype_t dt, size_t wstage, size_t ibytes, int G, int R);   // wstage: values + program
// Tensor-memory columns of one A buffer: room for one piece of an entry of
// at least 32 K columns of fp32 (high and low parts: 64 columns) or 128 of
// bf16 (pairs: 64 columns), and at least one whole block (C columns). The
// buffers fill the 512 columns after the G R accumulator columns, at most
// kGkASlotsMax of them; 0 if fewer than two fit.
inline int64_t gk_slot_cols(int R, int C, bool f32, int G) {
    const int64_t slot = std::max<int64_t>(64, f32 ? 2 * C : C / 2);
    const int64_t left = kGkTmemCols - (int64_t)G * R;
    return left / slot >= 2 ? slot : 0;
}
inline int gk_slots(int R, int C, bool f32, int G) {
    const int64_t slot = gk_slot_cols(R, C, f32, G);
    return slot ? (int)std::min<int64_t>(kGkASlotsMax, (kGkTmemCols - (int64_t)G * R) / slot) : 0;
}

}  // namespace bsr
