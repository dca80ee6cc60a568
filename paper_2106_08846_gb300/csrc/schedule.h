// Schedule construction (work list, split rows, kernel choice) and dispatch.
#pragma once

#include "bsr_internal.h"

namespace bsr {

// Fills the plan of a Schedule whose key fields (device, dtype, R, C, M, K,
// indptr, indices) are set, and uploads its device arrays.
bsr_status_t build_schedule(Schedule &sc);

// Makes the handle's kernel-layout copy of the block values, if the chosen
// kernel wants one (else the borrowed array is used directly).
bsr_status_t pack_data(Handle &h);

// Launches every kernel of one bsr_spmm call on a.stream.
cudaError_t launch_spmm(const LaunchArgs &a);

// A product's fusion class at N: products with equal non-negative classes
// (same X, N and stream) can share one grid; -1: the generic kernel, which
// runs alone. *G receives the task size chosen for N.
int fusion_class(const Schedule &sc, int64_t N, int *G);

// Launches n products that share X, N and the stream: products whose kernels
// share a template (xstage, or tensor-core of one dtype and R) run as one
// grid, up to 64 at a time; generic-kernel products one after another.
cudaError_t launch_spmm_batch(const LaunchArgs *as, int n);

}  // namespace bsr
