// Parameters shared by the tcgen05 kernel and the schedule that feeds it.
#pragma once

#include <cstddef>
#include <cstdint>

#include "bsr.h"

namespace bsr {

constexpr int kTcTokens = 128;         // tokens per CTA = MMA M = TMEM lanes
constexpr int kTcChunk = 64;           // K columns per ring stage (one 128-byte swizzle row of bf16)
constexpr int kTcStages = 6;           // ring depth
constexpr int kTcMaxSmem = 232448;     // 227 KB
constexpr int kTcTmemCols = 512;       // accumulator columns per SM
constexpr int kTcTaskSizes = 6;
constexpr int kTcG[kTcTaskSizes] = {1, 2, 4, 8, 16, 32};

struct TcPlan {
    size_t task_wbytes[kTcTaskSizes] = {0, 0, 0, 0, 0, 0};
    size_t task_ibytes[kTcTaskSizes] = {0, 0, 0, 0, 0, 0};
};

bool tc_supports(int R, int C, bsr_dtype_t dt, int64_t K);
int tc_g_index(int G);
size_t tc_smem_bytes(int R, int G, size_t wbytes, size_t ibytes);
size_t tc_task_budget(int R);

}  // namespace bsr
