// Parameters shared by the persistent SIMT kernel for tall blocks ("xrow")
// and the schedule that feeds it.
#pragma once

#include <cstddef>
#include <cstdint>
#include <vector>

#include "bsr.h"

namespace bsr {

constexpr int kXrWarps = 12;          // consumer warps; + 1 producer warp
constexpr int kXrStages = 3;          // X ring depth
constexpr int kXrMaxSmem = 232448;    // 227 KB, the per-CTA opt-in limit
constexpr int kXrItab = 8;            // ints per item in a task's item table
constexpr int kXrConfigs = 2;         // S = 2 (64 tokens, 6 items per task), S = 4 (128 tokens, 3 items)

// Configuration s (0 or 1): S = 2 << s warps per item, each on its own
// 32-token subtile; a task holds kXrWarps / S items and a unit (one CTA's
// turn) covers 32 S tokens; a ring stage holds 4096 / (32 S) columns of X
// (32 KB of fp32).
inline int xrow_S(int s) { return 2 << s; }
inline int xrow_G(int s) { return kXrWarps / xrow_S(s); }
inline int xrow_tokens(int s) { return 32 * xrow_S(s); }
inline int xrow_chunk(int s) { return 256 / xrow_S(s); }

// Block shapes the kernel runs: 16 or 32 rows, one column or 16 / 32 columns.
bool xrow_supports(int R, int C, bsr_dtype_t dt, int64_t K);

// Values of one stored block in a task blob (floats): one-column blocks take
// R + 4 (padding that moves consecutive blocks four banks apart), wider
// blocks C * R (their 16-byte row groups permuted per column, see the packer).
inline int64_t xrow_block_floats(int R, int C) { return C == 1 ? R + 4 : (int64_t)C * R; }

// Byte offset of chunk column kk in a ring stage at token row 0, before the
// 128-byte swizzle: boxes of 128-byte rows (32 fp32 or 64 bf16 columns) by
// `tokens` rows, one after another.
inline uint32_t xrow_stage_offset(bsr_dtype_t dt, int tokens, int kk) {
    const int es = dt == BSR_F32 ? 4 : 2;
    const int box_cols = 128 / es;
    return (uint32_t)((kk / box_cols) * tokens * 128 + (kk % box_cols) * es);
}

// Per configuration: task blobs [ item table: G x kXrItab ints (row, slot,
// len, woff, roff, 0, 0, 0) | records (16-byte aligned) | block values
// (16-byte aligned) ] at a fixed stride, and the work per task (multiply-adds
// per token of its longest item, plus a fixed cost) as prefix sums, which the
// kernel uses to give every CTA a contiguous range of equal total work.
// Record of an item: [ per chunk c = 0..nchunks: its first block in chunk c,
// padded to 4 | per block: its X offset in a stage (one column) or its block
// column (wider), padded to 4 ].
struct XrPlan {
    bool ok[kXrConfigs] = {false, false};
    int n_tasks[kXrConfigs] = {0, 0};
    uint32_t stride[kXrConfigs] = {0, 0};   // blob bytes per task
    uint32_t ibytes[kXrConfigs] = {0, 0};   // record region bytes per task (16-byte padded)
    uint32_t wbytes[kXrConfigs] = {0, 0};   // value region bytes per task
    int64_t blob_off[kXrConfigs] = {-1, -1};   // byte offset of the blobs in the packed values
    int64_t cost_off[kXrConfigs] = {-1, -1};   // byte offset of the int64 task-cost prefix sums
    int64_t total_bytes = 0;
    std::vector<int32_t> blob;               // all configurations' blobs and prefix sums, values zero
    std::vector<int64_t> vdst;               // [cfg][item]: float offset of the item's values (-1: none)
    std::vector<int32_t> perm;               // [cfg][position]: stored block at each packed position
    int64_t *d_vdst = nullptr;
    int32_t *d_perm = nullptr;
};

size_t xrow_smem_bytes(int s, bsr_dtype_t dt, size_t stride);

}  // namespace bsr
