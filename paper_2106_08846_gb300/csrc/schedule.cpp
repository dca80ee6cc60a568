// Work list, load balancing and kernel selection: the GPU stand-in for the
// TVM task scheduler of Section 2.2, which tunes each BSR task for the
// hardware and groups tasks by their sparsity structure.
//
// A schedule turns the block rows into work items. Rows much longer than the
// mean are split into pieces whose fp32 partial tiles are summed by a reduce
// pass in a fixed order (so results do not depend on timing). Empty rows stay
// as items so that their outputs receive the bias. Items are ordered longest
// first, the classic LPT rule, so that the long ones start early.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <numeric>

#include "schedule.h"

namespace bsr {

namespace {

template <typename T>
cudaError_t upload(T **dst, const std::vector<T> &v) {
    *dst = nullptr;
    if (v.empty()) return cudaSuccess;
    cudaError_t e = cudaMalloc((void **)dst, v.size() * sizeof(T));
    if (e != cudaSuccess) return e;
    return cudaMemcpy(*dst, v.data(), v.size() * sizeof(T), cudaMemcpyHostToDevice);
}

// Splits rows longer than `limit` blocks into ceil(len/limit) near-equal pieces.
void make_items(Schedule &sc, int64_t limit) {
    sc.items.clear();
    sc.splits.clear();
    sc.n_slots = 0;
    sc.split_len = (int)std::min<int64_t>(limit, INT32_MAX);
    for (int64_t i = 0; i < sc.MB; i++) {
        int32_t p0 = sc.indptr[i], p1 = sc.indptr[i + 1];
        int64_t len = p1 - p0;
        if (limit <= 0 || len <= limit) {
            sc.items.push_back({(int32_t)i, p0, p1, -1});
            continue;
        }
        int64_t pieces = (len + limit - 1) / limit;
        Split s{(int32_t)i, sc.n_slots, (int32_t)pieces, 0};
        for (int64_t k = 0; k < pieces; k++) {
            int32_t a = (int32_t)(p0 + len * k / pieces), b = (int32_t)(p0 + len * (k + 1) / pieces);
            sc.items.push_back({(int32_t)i, a, b, sc.n_slots++});
        }
        sc.splits.push_back(s);
    }
    std::stable_sort(sc.items.begin(), sc.items.end(),
                     [](const Item &a, const Item &b) { return a.p1 - a.p0 > b.p1 - b.p0; });
}

void row_stats(Schedule &sc) {
    sc.empty_rows = 0;
    sc.max_row = 0;
    for (int64_t i = 0; i < sc.MB; i++) {
        int64_t len = sc.indptr[i + 1] - sc.indptr[i];
        sc.empty_rows += len == 0;
        sc.max_row = std::max(sc.max_row, len);
    }
}

// Rows longer than twice the mean non-empty row (and than 32 blocks) are
// split into pieces of at most that length.
int64_t split_limit(const Schedule &sc) {
    if (sc.MB == 0 || sc.nnzb == 0) return 0;
    const int64_t nonempty = sc.MB - sc.empty_rows;
    const double mean = (double)sc.nnzb / (double)std::max<int64_t>(nonempty, 1);
    const int64_t limit = std::max<int64_t>(32, (int64_t)std::ceil(2.0 * mean));
    return sc.max_row > limit ? limit : 0;
}

}  // namespace

bsr_status_t build_schedule(Schedule &sc) {
    row_stats(sc);
    sc.variant = V_GENERIC;
    sc.threads = 256;
    sc.tn = std::max(1, 256 / std::min(sc.R, 256));
    sc.groups = 1;
    sc.smem = 0;
    make_items(sc, split_limit(sc));
    sc.group_begin = {0, (int32_t)sc.items.size()};
    if (upload(&sc.d_items, sc.items) != cudaSuccess || upload(&sc.d_splits, sc.splits) != cudaSuccess ||
        upload(&sc.d_group_begin, sc.group_begin) != cudaSuccess ||
        upload(&sc.d_indptr, sc.indptr) != cudaSuccess || upload(&sc.d_indices, sc.indices) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_ALLOC;
    }
    return BSR_OK;
}

bsr_status_t pack_data(Handle &h) {
    h.data_packed = nullptr;
    return BSR_OK;
}

int launches_per_call(const Schedule &sc) { return 1 + (sc.splits.empty() ? 0 : 1); }

cudaError_t launch_spmm(const LaunchArgs &a) {
    cudaError_t e = launch_generic(a);
    if (e != cudaSuccess) return e;
    if (!a.sc->splits.empty()) e = launch_reduce(a);
    return e;
}

}  // namespace bsr
