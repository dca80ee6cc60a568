// Planning and per-call choice of the gathered-K tensor-core kernel.
#pragma once

#include "bsr_internal.h"

namespace bsr {

// Builds sc.gk for a schedule whose structure is set (the caller's block
// rows): its packed values start at byte packed_end of the packed buffer.
void plan_gk(Schedule &sc, int64_t packed_end);

// The gk task size for a call of N tokens, or -1 for the schedule's own kernel.
int choose_gk(const Schedule &sc, int64_t N);

}  // namespace bsr
