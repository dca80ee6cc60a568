// Parameters shared by the xstage kernel and the schedule that feeds it.
#pragma once

#include <cstddef>
#include <cstdint>

#include "bsr.h"

namespace bsr {

constexpr int kXsTokens = 64;          // tokens per CTA
constexpr int kXsChunk = 128;          // K columns per ring stage
constexpr int kXsStages = 3;           // ring depth
constexpr int kXsConsumerWarps = 14;   // + 1 producer warp, up to 136 registers a thread
constexpr int kXsConsumerWarpsR1 = 24; // one-row blocks (small tiles): + 1 producer warp, 80 registers a thread
constexpr int kXsMaxSmem = 232448;     // 227 KB, the per-CTA opt-in limit
constexpr int kXsWDup = 1;             // copies of each packed block value
constexpr int kXsBatchMax = 64;        // products in one fused launch (bsr_spmm_batch)

// Task sizes G (items per CTA): up to the consumer warps NW, NW/G (rounded
// down) warps per item, the rest idle; one-row blocks (NW = 24) take only
// sizes dividing 24, and also G = 48 and 96, two or four items per warp.
// Multi-row blocks run fourteen consumer warps: more warps hide more of the
// multiply-add loop's latency, and fourteen measured faster than twelve even
// where two of them idle (BERT-large 32x1 fp32: 7-item tasks 139.1 us against
// 6-item tasks on twelve warps 141.2 us; block-shape sweep 154 against 157
// us), fifteen slower (146 us: 5-item tasks).
constexpr int kXsTaskSizes = 11;
constexpr int kXsG[kXsTaskSizes] = {1, 2, 3, 4, 6, 7, 12, 14, 24, 48, 96};

constexpr int kXsItab = 12;   // ints per item in a task's item table

// Per task size (index into kXsG): the largest shared-memory footprint of
// block values / indices over all tasks of G consecutive items.
//
// Everything one task needs is one contiguous "blob" in device memory, at a
// fixed stride per task size, so a CTA fetches it in one round trip without
// first reading any table: [ item table: G x kXsItab ints (row, p0, p1,
// slot, -, len, -, woff, roff, -, -, -) | records (task_ibytes, 16-byte
// padded) | block values (task_wbytes, 16-byte padded) ]. woff (floats) and
// roff (ints) locate an item's values and record inside their regions.
struct XsPlan {
    size_t task_wbytes[kXsTaskSizes] = {};
    size_t task_ibytes[kXsTaskSizes] = {};   // item records (see xstage_record_ints)
};

// Per item, the task blob holds one "record" of int32:
//   [ per block: its X offset inside a ring stage (C == 1) or its block
//     column (C > 1) -- for 1x1 blocks followed by its weight --, padded to
//     4 ints | per K chunk c = 0..nchunks: the first item-local block of
//     chunk c, padded to 4 ints ]
#ifdef __CUDACC__
#define XS_HD __host__ __device__
#else
#define XS_HD
#endif
XS_HD inline int64_t xstage_pad4(int64_t n) { return (n + 3) & ~int64_t(3); }
// ints per block in a record: 1x1 blocks carry (X offset, weight) pairs, so
// one 8-byte load gives a block's whole operand description; others one int
// (their values live in the blob's value region)
XS_HD inline int xstage_block_ints(int R, int C) { return R == 1 && C == 1 ? 2 : 1; }
XS_HD inline int64_t xstage_record_ints(int64_t len, int64_t nchunks, int bi = 1) {
    return xstage_pad4(bi * len) + xstage_pad4(nchunks + 1);
}
// Tile slots, written by the consumer warps after the main loop (in the
// ring, then free): token-major, [t][slot][r], so that the output pass reads
// consecutive outputs of one token from consecutive banks. The token pitch
// (floats) is padded so that eight consecutive tokens of one slot land in
// distinct 16-byte bank groups (one-row and two-row tiles: distinct banks).
constexpr int xstage_slot_pitch(int R, int nslot) {
    const int base = nslot * R;
    if (R == 1) return base % 2 == 0 ? base + 1 : base;
    if (R == 2) return (base / 2) % 2 == 0 ? base + 2 : base;
    return base % 8 == 4 ? base : base + (12 - base % 8) % 8;
}
// Byte offset of chunk column kk inside a ring stage, token row 0.
uint32_t xstage_stage_offset(bsr_dtype_t dt, int kk);

int g_index(int G);
bool xstage_task_size_ok(int R, int G);   // G > 14 needs one-row blocks
bool xstage_supports(int R, int C, bsr_dtype_t dt, int64_t K);

// Dynamic shared memory of one CTA: ring (reused for the epilogue's partial
// tiles), block values, indices, chunk table, barriers and item table.
size_t xstage_smem_bytes(bsr_dtype_t dt, int R, int64_t K, int G, size_t wbytes, size_t ibytes);
// Shared memory left for block values + indices of one task.
size_t xstage_task_budget(bsr_dtype_t dt, int R, int64_t K);

}  // namespace bsr
