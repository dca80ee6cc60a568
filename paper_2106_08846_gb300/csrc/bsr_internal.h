// Internal declarations shared by the host runtime (api.cpp) and the kernels.
#pragma once

#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <memory>
#include <mutex>
#include <string>
#include <vector>

#include "bsr.h"
#include "gk.h"
#include "tc.h"
#include "xstage.h"

namespace bsr {

// One unit of work: block row `row`, stored blocks [p0, p1). slot < 0 writes
// Y (+ bias) directly; slot >= 0 writes an fp32 partial tile to the workspace
// at [slot][N][R] and a reduce pass sums the slots of the row.
struct Item {
    int32_t row, p0, p1, slot;
};

// A row finished by the reduce pass: a block row split into pieces, slots
// [slot0, slot0 + nslot) in piece order, or an empty row (nslot 0: Y = bias).
struct Split {
    int32_t row, slot0, nslot, pad;
};

enum Variant : int {
    V_GENERIC = 0,   // any R x C, any dtype: one thread per output, global loads
    V_XSTAGE = 1,    // SIMT, X token tile staged in shared memory, register tiles
    V_TC = 2,        // tcgen05 tensor cores, bf16 square blocks
};

const char *variant_name(int v);

// Device-side status word values (first error wins).
enum : int { DEV_OK = 0, DEV_TIMEOUT = 1 };

// Everything derived from (device, dtype, R, C, M, K, indptr, indices): shared
// between handles whose structure is identical.
struct Schedule {
    int device = 0;
    bsr_dtype_t dt = BSR_F32;
    int R = 1, C = 1;
    int64_t M = 0, K = 0, MB = 0, KB = 0, nnzb = 0;
    std::vector<int32_t> indptr, indices;   // host copies (the key)
    uint64_t hash = 0;

    int variant = V_GENERIC;
    int tn = 0;            // tokens per CTA
    int threads = 256;     // threads per CTA
    int split_len = 0;     // max blocks per item (0: no splitting)
    int groups = 1;        // item groups per token tile
    size_t smem = 0;       // dynamic shared memory per CTA
    std::vector<Item> items;
    std::vector<Split> splits;
    std::vector<int32_t> group_begin;   // groups + 1 offsets into items
    XsPlan xs;                          // xstage task footprints
    TcPlan tc;                          // tcgen05 task footprints
    GkPlan gk;                          // gathered-K tensor-core kernel, alongside the variant's own
    int n_slots = 0;
    int64_t empty_rows = 0, max_row = 0;
    int sm_count = 148;

    Item *d_items = nullptr;
    Split *d_splits = nullptr;
    int32_t *d_group_begin = nullptr;
    std::vector<int32_t> xs_rec;        // xstage: per-item records (block offsets/columns, chunk starts)
    std::vector<int32_t> xs_rec_off;    // per item: record offset in ints (multiple of 4)
    std::vector<int32_t> xs_perm;       // per packed block position: the stored block it holds
    std::vector<int32_t> xs_blob;       // task blobs of every task size, block values left zero
    int64_t xs_blob_off[kXsTaskSizes] = {};      // byte offset of task size gi's blobs (-1: not usable)
    int64_t xs_blob_stride[kXsTaskSizes] = {};   // bytes per task
    std::vector<int64_t> xs_vdst;       // [gi][item]: float offset of the item's values in the blobs (-1: none)
    int32_t *d_xs_perm = nullptr;
    int64_t *d_xs_vdst = nullptr;
    int32_t *d_indptr = nullptr;        // owned copies of the structure
    int32_t *d_indices = nullptr;

    // Execution structure of the tensor-core kernel when it runs small bf16
    // blocks re-blocked into max(R, 16) x 64 tiles (ex_C = 64, ex_R; zeros for
    // absent blocks): the items and task lists refer to these tiles; vmap
    // gives every stored block the element offset of its first value in the
    // tile array.
    int ex_C = 1;
    int ex_R = 1;             // execution block height (16 for blocks of fewer rows re-blocked into tiles)
    int64_t ex_nnzb = 0;
    int64_t tc_w_total = 0;   // bytes of the tensor-core kernel's packed values (all task sizes)
    std::vector<int32_t> vmap;
    int32_t *d_vmap = nullptr;

    std::atomic<int64_t> reuse_count{0};
    ~Schedule();
};

struct Handle {
    int device = 0;
    bsr_dtype_t dt = BSR_F32;
    int R = 1, C = 1;
    int64_t M = 0, K = 0;
    const void *data = nullptr;         // borrowed
    void *data_packed = nullptr;        // owned, kernel layout
    std::shared_ptr<Schedule> sched;
    int *d_status = nullptr;
    float *ws = nullptr;                // split-row partials
    size_t ws_bytes = 0;
    void *stage_x = nullptr, *stage_y = nullptr;   // for host X / Y
    size_t stage_x_bytes = 0, stage_y_bytes = 0;
    bool cache_hit = false;
    uint64_t wait_ns = 1000000000ull;   // device wait bound (BSR_WAIT_LIMIT_NS at create)
    int stall_chunk = -1;               // test hook (BSR_TEST_STALL_CHUNK at create): never load this X chunk
};

inline size_t dtype_size(bsr_dtype_t dt) { return dt == BSR_F32 ? 4 : 2; }

// ---- builder (builder.cu)
cudaError_t launch_builder_count(const void *W, bsr_dtype_t dt, int64_t M, int64_t K, int R, int C,
                                 float thr, uint8_t *flags, int32_t *counts, int32_t *indptr,
                                 cudaStream_t s);
cudaError_t launch_builder_compact(const void *W, bsr_dtype_t dt, int64_t M, int64_t K, int R, int C,
                                   const uint8_t *flags, const int32_t *indptr, int32_t *indices,
                                   void *data, cudaStream_t s);

// ---- SpMM kernels (spmm_*.cu)
struct LaunchArgs {
    const Schedule *sc;
    const void *data;      // kernel-layout block values
    const void *X;
    const float *bias;
    void *Y;
    float *ws;
    int *status;
    int64_t N;
    cudaStream_t stream;
    uint64_t wait_ns;      // bound on every device-side wait
    int stall_chunk;       // test hook, -1 in normal use
};
cudaError_t launch_generic(const LaunchArgs &a);
cudaError_t launch_xstage(const LaunchArgs &a, int G);
// Products whose xstage launches can share one grid have equal keys (dtype,
// block shape class and kernel template at task size G).
int xstage_fusion_key(const Schedule &sc, int G);
// n products sharing X (equal fusion keys, same X, N, K and stream) in one grid.
cudaError_t launch_xstage_batch(const LaunchArgs *las, const int *Gs, int n);
cudaError_t launch_tc(const LaunchArgs &a, int G);
// Products whose tensor-core launches can share one grid have equal keys.
int tc_fusion_key(const Schedule &sc);
// n products sharing X (equal keys, same X, N, K and stream) in one grid.
cudaError_t launch_tc_batch(const LaunchArgs *las, const int *Gs, int n);
cudaError_t pack_tc_data(const void *data, bsr_dtype_t dt, const int32_t *order, const int32_t *stack, int64_t n,
                         int R, int C, void *out,
                         cudaStream_t s);
cudaError_t reblock_tc_data(const uint16_t *data, const int32_t *vmap, int64_t nnzb, int R, int C, uint16_t *tiles,
                            cudaStream_t s);
cudaError_t pack_xstage_data(const void *data, bsr_dtype_t dt, const Item *items, const int32_t *perm,
                             const int64_t *vdst, int64_t n_items, int R, int C, float *blobs, cudaStream_t s);
cudaError_t launch_reduce(const LaunchArgs &a);
// The persistent tensor-core kernel on the tc task records at task size G,
// and the task size it runs a call of N tokens at (-1: the tc kernel runs it).
cudaError_t launch_tcp(const LaunchArgs &a, int G);
int choose_tcp(const Schedule &sc, int64_t N);
// The gathered-K tensor-core kernel at task size G (gk.h).
cudaError_t launch_gk(const LaunchArgs &a, int G);
cudaError_t pack_gk_data(const void *data, bsr_dtype_t dt, const int32_t *wsrc, const int32_t *wslot,
                         const int64_t *wbase, int64_t n, int R, int C, void *out, cudaStream_t s);

int launches_per_call(const Schedule &sc, int64_t N = 0);   // N = 0: the schedule variant's own path

}  // namespace bsr

// The opaque handle of the C ABI.
struct bsr_handle_s : public bsr::Handle {};
