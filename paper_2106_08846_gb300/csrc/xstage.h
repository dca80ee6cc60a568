// Parameters shared by the xstage kernel and the schedule that feeds it.
#pragma once

#include <cstddef>
#include <cstdint>

#include "bsr.h"

namespace bsr {

constexpr int kXsTokens = 64;          // tokens per CTA
constexpr int kXsChunk = 128;          // K columns per ring stage
constexpr int kXsStages = 3;           // ring depth
constexpr int kXsConsumerWarps = 8;
constexpr int kXsMaxSmem = 232448;     // 227 KB, the per-CTA opt-in limit

// Per task size G in {1, 2, 4, 8} (index 0..3): the largest shared-memory
// footprint of block values / indices over all tasks of G consecutive items.
struct XsPlan {
    size_t task_wbytes[4] = {0, 0, 0, 0};
    size_t task_ibytes[4] = {0, 0, 0, 0};
};

int g_index(int G);
bool xstage_supports(int R, int C, bsr_dtype_t dt, int64_t K);

// Dynamic shared memory of one CTA: ring (reused for the epilogue's partial
// tiles), block values, indices, chunk table, barriers and item table.
size_t xstage_smem_bytes(bsr_dtype_t dt, int R, int64_t K, int G, size_t wbytes, size_t ibytes);
// Shared memory left for block values + indices of one task.
size_t xstage_task_budget(bsr_dtype_t dt, int R, int64_t K);

}  // namespace bsr
