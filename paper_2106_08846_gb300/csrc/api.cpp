// Host runtime behind include/bsr.h: argument validation, structure checks,
// the schedule (work list, split rows, kernel choice), the schedule cache and
// stream-ordered launches.
//
// The schedule cache stands in for the task buffer of Section 2.2: a BSR
// operator whose structure (shape, block shape, dtype, indptr, indices) is
// identical to one already scheduled reuses that schedule instead of
// building a new one.
#include <algorithm>
#include <cinttypes>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <unordered_map>
#include <vector>

#include "bsr_internal.h"
#include "schedule.h"

namespace bsr {

namespace {

struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) { ok = false; return; }
        if (prev != dev && cudaSetDevice(dev) != cudaSuccess) ok = false;
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

std::mutex g_cache_mu;
std::unordered_map<uint64_t, std::vector<std::weak_ptr<Schedule>>> g_cache;
std::atomic<int64_t> g_cache_hits{0}, g_cache_misses{0};

uint64_t fnv1a(uint64_t h, const void *p, size_t n) {
    const unsigned char *b = static_cast<const unsigned char *>(p);
    for (size_t i = 0; i < n; i++) { h ^= b[i]; h *= 0x100000001b3ull; }
    return h;
}

uint64_t structure_hash(int device, bsr_dtype_t dt, int R, int C, int64_t M, int64_t K,
                        const std::vector<int32_t> &indptr, const std::vector<int32_t> &indices) {
    uint64_t h = 0xcbf29ce484222325ull;
    int64_t key[6] = {device, (int64_t)dt, R, C, M, K};
    h = fnv1a(h, key, sizeof key);
    h = fnv1a(h, indptr.data(), indptr.size() * sizeof(int32_t));
    return fnv1a(h, indices.data(), indices.size() * sizeof(int32_t));
}

bool same_key(const Schedule &s, int device, bsr_dtype_t dt, int R, int C, int64_t M, int64_t K,
              const std::vector<int32_t> &indptr, const std::vector<int32_t> &indices) {
    return s.device == device && s.dt == dt && s.R == R && s.C == C && s.M == M && s.K == K &&
           s.indptr == indptr && s.indices == indices;
}

enum PtrKind { PK_DEVICE, PK_HOST, PK_BAD };

// Where a pointer lives, relative to the handle's device.
PtrKind classify(const void *p, int device) {
    cudaPointerAttributes at;
    cudaError_t e = cudaPointerGetAttributes(&at, p);
    if (e != cudaSuccess) { cudaGetLastError(); return PK_BAD; }
    switch (at.type) {
        case cudaMemoryTypeDevice: return at.device == device ? PK_DEVICE : PK_BAD;
        case cudaMemoryTypeManaged: return PK_DEVICE;
        case cudaMemoryTypeHost:
        case cudaMemoryTypeUnregistered: return PK_HOST;
        default: return PK_BAD;
    }
}

bool overlaps(const void *a, size_t na, const void *b, size_t nb) {
    uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
    return na && nb && x < y + nb && y < x + na;
}

bsr_status_t grow(void **buf, size_t *cap, size_t need) {
    if (need <= *cap) return BSR_OK;
    if (*buf) cudaFree(*buf);
    *buf = nullptr;
    *cap = 0;
    if (cudaMalloc(buf, need) != cudaSuccess) { cudaGetLastError(); *buf = nullptr; return BSR_ERR_ALLOC; }
    *cap = need;
    return BSR_OK;
}

bsr_status_t check_shape(int64_t M, int64_t K, int R, int C, bsr_dtype_t dt) {
    if (dt != BSR_F32 && dt != BSR_BF16) return BSR_ERR_UNSUPPORTED;
    if (M < 0 || K < 0 || R <= 0 || C <= 0) return BSR_ERR_INVALID_ARG;
    if ((int64_t)R * C > 4096) return BSR_ERR_UNSUPPORTED;
    if (M % R || K % C) return BSR_ERR_SHAPE;
    if (M / R + 1 > INT32_MAX || K / C > INT32_MAX) return BSR_ERR_SHAPE;
    return BSR_OK;
}

}  // namespace

const char *variant_name(int v) {
    switch (v) {
        case V_GENERIC: return "generic";
        case V_XSTAGE: return "xstage";
        case V_TC: return "tcgen05";
        default: return "?";
    }
}

Schedule::~Schedule() {
    DeviceGuard g(device);
    cudaFree(d_items);
    cudaFree(d_splits);
    cudaFree(d_group_begin);
    cudaFree(d_indptr);
    cudaFree(d_xs_perm);
    cudaFree(d_vmap);
    cudaFree(d_xs_vdst);
    for (int gi = 0; gi < kGkTaskSizes; gi++) {
        cudaFree(gk.d_rec[gi]);
        cudaFree(gk.d_rec_off[gi]);
        cudaFree(gk.d_wsrc[gi]);
        cudaFree(gk.d_wslot[gi]);
        cudaFree(gk.d_wbase[gi]);
        cudaFree(gk.d_prog[gi]);
    }
    for (int gi = 0; gi < kTcTaskSizes; gi++) {
        cudaFree(tc.d_rec[gi]);
        cudaFree(tc.d_rec_off[gi]);
        cudaFree(tc.d_worder[gi]);
        cudaFree(tc.d_wstack[gi]);
        cudaFree(tc.d_prog[gi]);
        cudaFree(tc.d_stab[gi]);
    }
    cudaFree(d_indices);
}

}  // namespace bsr

using namespace bsr;

// A captured product sequence (bsr_plan_create).
struct bsr_plan_s {
    int device = 0;
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    std::vector<int> order, call;   // execution order; library call of each executed product
    int n_kernels = 0;
    std::vector<float *> ws;        // owned split-row workspaces
    ~bsr_plan_s() {
        DeviceGuard g(device);
        if (exec) cudaGraphExecDestroy(exec);
        if (graph) cudaGraphDestroy(graph);
        for (float *p : ws) cudaFree(p);
    }
};

namespace {

// The execution order and call grouping of a plan: `calls` lists, per library
// call, the products it runs.
void plan_order(const bsr_handle_t *handles, const void *const *X, const int64_t *N, int n, bool independent,
                std::vector<std::vector<int>> &calls) {
    calls.clear();
    if (!independent) {
        for (int i = 0; i < n; i++)
            if (N[i] > 0) calls.push_back({i});
        return;
    }
    // groups of products sharing (X, N, dtype, K), in first-appearance order
    std::vector<std::vector<int>> groups;
    for (int i = 0; i < n; i++) {
        if (N[i] == 0) continue;
        const Handle *h = handles[i];
        size_t g = 0;
        for (; g < groups.size(); g++) {
            const int j = groups[g][0];
            if (X[j] == X[i] && N[j] == N[i] && handles[j]->dt == h->dt && handles[j]->K == h->K) break;
        }
        if (g == groups.size()) groups.emplace_back();
        groups[g].push_back(i);
    }
    for (std::vector<int> &grp : groups) {
        // kernels that share a template next to each other (generic last),
        // handles that share a schedule adjacent, then the given order
        std::vector<const Schedule *> first_seen;
        auto sched_rank = [&](const Schedule *sc) {
            for (size_t k = 0; k < first_seen.size(); k++)
                if (first_seen[k] == sc) return (int)k;
            first_seen.push_back(sc);
            return (int)first_seen.size() - 1;
        };
        std::vector<std::pair<std::pair<int, int>, int>> keyed;
        for (int i : grp) {
            int G = 0;
            const int fc = fusion_class(*handles[i]->sched, N[i], &G);
            keyed.push_back({{fc < 0 ? INT32_MAX : fc, sched_rank(handles[i]->sched.get())}, i});
        }
        std::stable_sort(keyed.begin(), keyed.end(),
                         [](const auto &a, const auto &b) { return a.first < b.first; });
        // a handle may run once per call (its status word and schedule state)
        std::vector<int> cur;
        for (const auto &kv : keyed) {
            const int i = kv.second;
            bool repeat = false;
            for (int j : cur) repeat |= handles[j] == handles[i];
            if (repeat) {
                calls.push_back(cur);
                cur.clear();
            }
            cur.push_back(i);
        }
        if (!cur.empty()) calls.push_back(cur);
    }
}

}  // namespace

extern "C" {

const char *bsr_status_str(bsr_status_t s) {
    switch (s) {
        case BSR_OK: return "BSR_OK";
        case BSR_ERR_INVALID_ARG: return "BSR_ERR_INVALID_ARG";
        case BSR_ERR_SHAPE: return "BSR_ERR_SHAPE";
        case BSR_ERR_UNSUPPORTED: return "BSR_ERR_UNSUPPORTED";
        case BSR_ERR_CAPACITY: return "BSR_ERR_CAPACITY";
        case BSR_ERR_STRUCTURE: return "BSR_ERR_STRUCTURE";
        case BSR_ERR_ALIGNMENT: return "BSR_ERR_ALIGNMENT";
        case BSR_ERR_CUDA: return "BSR_ERR_CUDA";
        case BSR_ERR_TIMEOUT: return "BSR_ERR_TIMEOUT";
        case BSR_ERR_ALLOC: return "BSR_ERR_ALLOC";
    }
    return "BSR_ERR_UNKNOWN";
}

bsr_status_t bsr_from_dense(const void *W, int64_t M, int64_t K, int R, int C, float threshold,
                            bsr_dtype_t dt, int32_t *indptr, int32_t *indices, void *data,
                            int64_t capacity_blocks, int64_t *nnzb_out, void *stream) {
    bsr_status_t st = check_shape(M, K, R, C, dt);
    if (st != BSR_OK) return st;
    if (!indptr || capacity_blocks < 0 || std::isnan(threshold) || threshold < 0.0f)
        return BSR_ERR_INVALID_ARG;
    if (M * K > 0 && !W) return BSR_ERR_INVALID_ARG;
    if (capacity_blocks > 0 && (!indices || !data)) return BSR_ERR_INVALID_ARG;
    const int64_t MB = M / R, KB = K / C;
    if (MB * KB > (int64_t)1 << 40) return BSR_ERR_SHAPE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);

    uint8_t *flags = nullptr;
    int32_t *counts = nullptr;
    size_t nflags = (size_t)std::max<int64_t>(MB * KB, 1);
    if (cudaMallocAsync((void **)&flags, nflags, s) != cudaSuccess ||
        cudaMallocAsync((void **)&counts, (size_t)std::max<int64_t>(MB, 1) * 4, s) != cudaSuccess) {
        cudaGetLastError();
        if (flags) cudaFreeAsync(flags, s);
        return BSR_ERR_ALLOC;
    }
    int64_t nnzb = 0;
    int32_t last = 0;
    st = BSR_OK;
    if (launch_builder_count(W, dt, M, K, R, C, threshold, flags, counts, indptr, s) != cudaSuccess ||
        cudaMemcpyAsync(&last, indptr + MB, sizeof last, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess) {
        cudaGetLastError();
        st = BSR_ERR_CUDA;
    }
    nnzb = last;
    if (st == BSR_OK && last < 0) st = BSR_ERR_SHAPE;   // more than 2^31-1 kept blocks
    if (st == BSR_OK && nnzb_out) *nnzb_out = nnzb;
    const bool query = !indices && !data && capacity_blocks == 0;
    if (st == BSR_OK && !query) {
        if (capacity_blocks < nnzb) {
            st = BSR_ERR_CAPACITY;
        } else if (nnzb > 0 &&
                   launch_builder_compact(W, dt, M, K, R, C, flags, indptr, indices, data, s) != cudaSuccess) {
            cudaGetLastError();
            st = BSR_ERR_CUDA;
        }
    }
    cudaFreeAsync(flags, s);
    cudaFreeAsync(counts, s);
    return st;
}

bsr_status_t bsr_create(const int32_t *indptr, const int32_t *indices, const void *data, int R,
                        int C, int64_t M, int64_t K, bsr_dtype_t dt, bsr_handle_t *out) {
    if (!out) return BSR_ERR_INVALID_ARG;
    *out = nullptr;
    bsr_status_t st = check_shape(M, K, R, C, dt);
    if (st != BSR_OK) return st;
    if (!indptr) return BSR_ERR_INVALID_ARG;
    int device = 0;
    if (cudaGetDevice(&device) != cudaSuccess) { cudaGetLastError(); return BSR_ERR_CUDA; }
    const int64_t MB = M / R, KB = K / C;
    if (classify(indptr, device) != PK_DEVICE) return BSR_ERR_INVALID_ARG;

    std::vector<int32_t> hp((size_t)MB + 1);
    if (cudaMemcpy(hp.data(), indptr, hp.size() * 4, cudaMemcpyDeviceToHost) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    if (hp[0] != 0) return BSR_ERR_STRUCTURE;
    for (int64_t i = 0; i < MB; i++)
        if (hp[i + 1] < hp[i]) return BSR_ERR_STRUCTURE;
    const int64_t nnzb = hp[MB];
    if (nnzb > 0 && (!indices || !data)) return BSR_ERR_INVALID_ARG;
    if (nnzb > 0 && (classify(indices, device) != PK_DEVICE || classify(data, device) != PK_DEVICE))
        return BSR_ERR_INVALID_ARG;
    if (nnzb > 0 && ((uintptr_t)data % dtype_size(dt) || (uintptr_t)indices % 4))
        return BSR_ERR_ALIGNMENT;
    std::vector<int32_t> hi((size_t)nnzb);
    if (nnzb > 0 && cudaMemcpy(hi.data(), indices, (size_t)nnzb * 4, cudaMemcpyDeviceToHost) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    for (int64_t i = 0; i < MB; i++)
        for (int64_t p = hp[i]; p < hp[i + 1]; p++) {
            if (hi[p] < 0 || hi[p] >= KB) return BSR_ERR_STRUCTURE;
            if (p > hp[i] && hi[p] <= hi[p - 1]) return BSR_ERR_STRUCTURE;
        }

    bsr_handle_s *h = new (std::nothrow) bsr_handle_s;
    if (!h) return BSR_ERR_ALLOC;
    h->device = device;
    h->dt = dt;
    h->R = R;
    h->C = C;
    h->M = M;
    h->K = K;
    h->data = data;
    if (const char *w = getenv("BSR_WAIT_LIMIT_NS")) h->wait_ns = strtoull(w, nullptr, 10);
    if (const char *w = getenv("BSR_TEST_STALL_CHUNK")) h->stall_chunk = atoi(w);

    uint64_t hash = structure_hash(device, dt, R, C, M, K, hp, hi);
    {
        std::lock_guard<std::mutex> lk(g_cache_mu);
        auto &bucket = g_cache[hash];
        for (auto it = bucket.begin(); it != bucket.end();) {
            auto sp = it->lock();
            if (!sp) { it = bucket.erase(it); continue; }
            if (same_key(*sp, device, dt, R, C, M, K, hp, hi)) { h->sched = sp; break; }
            ++it;
        }
        if (h->sched) {
            h->cache_hit = true;
            h->sched->reuse_count++;
            g_cache_hits++;
        } else {
            auto sc = std::make_shared<Schedule>();
            sc->device = device;
            sc->dt = dt;
            sc->R = R;
            sc->C = C;
            sc->M = M;
            sc->K = K;
            sc->MB = MB;
            sc->KB = KB;
            sc->nnzb = nnzb;
            sc->indptr = std::move(hp);
            sc->indices = std::move(hi);
            sc->hash = hash;
            st = build_schedule(*sc);
            if (st != BSR_OK) { delete h; return st; }
            bucket.push_back(sc);
            h->sched = sc;
            g_cache_misses++;
        }
    }
    st = pack_data(*h);
    if (st == BSR_OK && cudaMalloc((void **)&h->d_status, sizeof(int)) != cudaSuccess) st = BSR_ERR_ALLOC;
    if (st == BSR_OK && cudaMemset(h->d_status, 0, sizeof(int)) != cudaSuccess) st = BSR_ERR_CUDA;
    if (st != BSR_OK) {
        cudaGetLastError();
        bsr_destroy(h);
        return st;
    }
    *out = h;
    return BSR_OK;
}

static bsr_status_t reserve_ws(Handle *h, int64_t N, bool host_io) {
    const Schedule &sc = *h->sched;
    size_t es = dtype_size(h->dt);
    bsr_status_t st = grow((void **)&h->ws, &h->ws_bytes, (size_t)sc.n_slots * (size_t)N * sc.ex_R * 4);
    if (st == BSR_OK && host_io) {
        st = grow(&h->stage_x, &h->stage_x_bytes, (size_t)N * h->K * es);
        if (st == BSR_OK) st = grow(&h->stage_y, &h->stage_y_bytes, (size_t)N * h->M * es);
    }
    return st;
}

bsr_status_t bsr_reserve(bsr_handle_t h, int64_t N_max) {
    if (!h || N_max < 0) return BSR_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    if (!g.ok) return BSR_ERR_CUDA;
    if (cudaDeviceSynchronize() != cudaSuccess) { cudaGetLastError(); return BSR_ERR_CUDA; }
    return reserve_ws(h, N_max, false);
}

bsr_status_t bsr_spmm(bsr_handle_t h, const void *X, const float *bias, void *Y, int64_t N,
                      void *stream) {
    if (!h || N < 0) return BSR_ERR_INVALID_ARG;
    if (N == 0) return BSR_OK;
    if (!X || !Y) return BSR_ERR_INVALID_ARG;
    const size_t es = dtype_size(h->dt);
    const size_t xbytes = (size_t)N * h->K * es, ybytes = (size_t)N * h->M * es;
    if ((uintptr_t)X % 16 || (uintptr_t)Y % 16 || (uintptr_t)bias % 4) return BSR_ERR_ALIGNMENT;
    if (overlaps(X, xbytes, Y, ybytes) || (bias && overlaps(bias, (size_t)h->M * 4, Y, ybytes)))
        return BSR_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    if (!g.ok) return BSR_ERR_CUDA;
    PtrKind kx = xbytes ? classify(X, h->device) : PK_DEVICE;
    PtrKind ky = ybytes ? classify(Y, h->device) : PK_DEVICE;
    if (kx == PK_BAD || ky == PK_BAD || kx != ky) return BSR_ERR_INVALID_ARG;
    if (bias && classify(bias, h->device) != PK_DEVICE) return BSR_ERR_INVALID_ARG;
    const bool host_io = kx == PK_HOST;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const Schedule &sc = *h->sched;

    bool need_grow = (size_t)sc.n_slots * (size_t)N * sc.ex_R * 4 > h->ws_bytes ||
                     (host_io && (xbytes > h->stage_x_bytes || ybytes > h->stage_y_bytes));
    if (need_grow) {
        if (cudaStreamSynchronize(s) != cudaSuccess) { cudaGetLastError(); return BSR_ERR_CUDA; }
        bsr_status_t st = reserve_ws(h, N, host_io);
        if (st != BSR_OK) return st;
    }
    const void *Xd = X;
    void *Yd = Y;
    if (host_io) {
        if (cudaMemcpyAsync(h->stage_x, X, xbytes, cudaMemcpyHostToDevice, s) != cudaSuccess) {
            cudaGetLastError();
            return BSR_ERR_CUDA;
        }
        Xd = h->stage_x;
        Yd = h->stage_y;
    }
    LaunchArgs a{&sc, h->data_packed ? h->data_packed : h->data, Xd, bias, Yd, h->ws, h->d_status, N, s,
                 h->wait_ns, h->stall_chunk};
    if (launch_spmm(a) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    if (host_io && cudaMemcpyAsync(Y, h->stage_y, ybytes, cudaMemcpyDeviceToHost, s) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    return BSR_OK;
}

bsr_status_t bsr_spmm_batch(const bsr_handle_t *handles, int n, const void *X, const float *const *biases,
                            void *const *Ys, int64_t N, void *stream) {
    if (n < 0 || N < 0) return BSR_ERR_INVALID_ARG;
    if (n == 0 || N == 0) return BSR_OK;
    if (!handles || !X || !Ys) return BSR_ERR_INVALID_ARG;
    for (int i = 0; i < n; i++) {
        if (!handles[i] || !Ys[i]) return BSR_ERR_INVALID_ARG;
        for (int j = 0; j < i; j++)
            if (handles[j] == handles[i]) return BSR_ERR_INVALID_ARG;   // one workspace per handle and call
    }
    const Handle *h0 = handles[0];
    for (int i = 1; i < n; i++)
        if (handles[i]->device != h0->device || handles[i]->dt != h0->dt) return BSR_ERR_INVALID_ARG;
    for (int i = 0; i < n; i++)
        if (handles[i]->K != h0->K) return BSR_ERR_SHAPE;
    const size_t es = dtype_size(h0->dt);
    const size_t xbytes = (size_t)N * h0->K * es;
    if ((uintptr_t)X % 16) return BSR_ERR_ALIGNMENT;
    for (int i = 0; i < n; i++) {
        if ((uintptr_t)Ys[i] % 16) return BSR_ERR_ALIGNMENT;
        if (biases && (uintptr_t)biases[i] % 4) return BSR_ERR_ALIGNMENT;
    }
    // no output may overlap X, a bias or another output
    for (int i = 0; i < n; i++) {
        const size_t yb = (size_t)N * handles[i]->M * es;
        if (overlaps(X, xbytes, Ys[i], yb)) return BSR_ERR_INVALID_ARG;
        for (int j = 0; j < n; j++) {
            if (biases && biases[j] && overlaps(biases[j], (size_t)handles[j]->M * 4, Ys[i], yb))
                return BSR_ERR_INVALID_ARG;
            if (j < i && overlaps(Ys[j], (size_t)N * handles[j]->M * es, Ys[i], yb)) return BSR_ERR_INVALID_ARG;
        }
    }
    DeviceGuard g(h0->device);
    if (!g.ok) return BSR_ERR_CUDA;
    if (classify(X, h0->device) != PK_DEVICE) return BSR_ERR_INVALID_ARG;   // device buffers only
    for (int i = 0; i < n; i++) {
        if (classify(Ys[i], h0->device) != PK_DEVICE) return BSR_ERR_INVALID_ARG;
        if (biases && biases[i] && classify(biases[i], h0->device) != PK_DEVICE) return BSR_ERR_INVALID_ARG;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    bool synced = false;
    for (int i = 0; i < n; i++) {
        Handle *h = handles[i];
        if ((size_t)h->sched->n_slots * (size_t)N * h->sched->ex_R * 4 <= h->ws_bytes) continue;
        if (!synced) {
            if (cudaStreamSynchronize(s) != cudaSuccess) { cudaGetLastError(); return BSR_ERR_CUDA; }
            synced = true;
        }
        bsr_status_t st = reserve_ws(h, N, false);
        if (st != BSR_OK) return st;
    }
    std::vector<LaunchArgs> as;
    as.reserve((size_t)n);
    for (int i = 0; i < n; i++) {
        Handle *h = handles[i];
        as.push_back(LaunchArgs{h->sched.get(), h->data_packed ? h->data_packed : h->data, X,
                                biases ? biases[i] : nullptr, Ys[i], h->ws, h->d_status, N, s, h->wait_ns,
                                h->stall_chunk});
    }
    if (launch_spmm_batch(as.data(), n) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    return BSR_OK;
}

bsr_status_t bsr_plan_create(const bsr_handle_t *handles, const void *const *X, const float *const *biases,
                             void *const *Y, const int64_t *N, int n, int independent, bsr_plan_t *out) {
    if (!out || n < 0) return BSR_ERR_INVALID_ARG;
    *out = nullptr;
    if (n > 0 && (!handles || !X || !Y || !N)) return BSR_ERR_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) { cudaGetLastError(); return BSR_ERR_CUDA; }
    std::vector<size_t> xb((size_t)n), yb((size_t)n);
    for (int i = 0; i < n; i++) {
        const Handle *h = handles[i];
        if (!h || N[i] < 0 || h->device != dev) return BSR_ERR_INVALID_ARG;
        if (N[i] == 0) continue;
        const float *b = biases ? biases[i] : nullptr;
        if (!X[i] || !Y[i]) return BSR_ERR_INVALID_ARG;
        if ((uintptr_t)X[i] % 16 || (uintptr_t)Y[i] % 16 || (uintptr_t)b % 4) return BSR_ERR_ALIGNMENT;
        const size_t es = dtype_size(h->dt);
        xb[(size_t)i] = (size_t)N[i] * h->K * es;
        yb[(size_t)i] = (size_t)N[i] * h->M * es;
        if (overlaps(X[i], xb[(size_t)i], Y[i], yb[(size_t)i]) || (b && overlaps(b, (size_t)h->M * 4, Y[i], yb[(size_t)i])))
            return BSR_ERR_INVALID_ARG;
        if ((xb[(size_t)i] && classify(X[i], dev) != PK_DEVICE) || (yb[(size_t)i] && classify(Y[i], dev) != PK_DEVICE) ||
            (b && classify(b, dev) != PK_DEVICE))
            return BSR_ERR_INVALID_ARG;
    }
    if (independent) {
        // no product may write what another reads or writes
        for (int i = 0; i < n; i++) {
            if (N[i] == 0) continue;
            for (int j = 0; j < n; j++) {
                if (j == i || N[j] == 0) continue;
                const float *bj = biases ? biases[j] : nullptr;
                if (overlaps(Y[i], yb[(size_t)i], X[j], xb[(size_t)j]) ||
                    (bj && overlaps(Y[i], yb[(size_t)i], bj, (size_t)handles[j]->M * 4)) ||
                    (j < i && overlaps(Y[i], yb[(size_t)i], Y[j], yb[(size_t)j])))
                    return BSR_ERR_INVALID_ARG;
            }
        }
    }
    std::vector<std::vector<int>> calls;
    plan_order(handles, X, N, n, independent != 0, calls);

    bsr_plan_s *plan = new (std::nothrow) bsr_plan_s;
    if (!plan) return BSR_ERR_ALLOC;
    plan->device = dev;
    std::vector<float *> ws_of((size_t)n, nullptr);
    for (int i = 0; i < n; i++) {
        if (N[i] == 0) continue;
        const Schedule &sc = *handles[i]->sched;
        const size_t bytes = (size_t)sc.n_slots * (size_t)N[i] * sc.ex_R * 4;
        if (!bytes) continue;
        if (cudaMalloc((void **)&ws_of[(size_t)i], bytes) != cudaSuccess) {
            cudaGetLastError();
            delete plan;
            return BSR_ERR_ALLOC;
        }
        plan->ws.push_back(ws_of[(size_t)i]);
    }
    cudaStream_t cs = nullptr;
    if (cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) {
        cudaGetLastError();
        delete plan;
        return BSR_ERR_CUDA;
    }
    bool ok = cudaStreamBeginCapture(cs, cudaStreamCaptureModeRelaxed) == cudaSuccess;
    std::vector<LaunchArgs> as;
    for (size_t c = 0; ok && c < calls.size(); c++) {
        as.clear();
        for (int i : calls[c]) {
            const Handle *h = handles[i];
            as.push_back(LaunchArgs{h->sched.get(), h->data_packed ? h->data_packed : h->data, X[i],
                                    biases ? biases[i] : nullptr, Y[i], ws_of[(size_t)i], h->d_status, N[i], cs,
                                    h->wait_ns, h->stall_chunk});
            plan->order.push_back(i);
            plan->call.push_back((int)c);
        }
        ok = (as.size() == 1 ? launch_spmm(as[0]) : launch_spmm_batch(as.data(), (int)as.size())) == cudaSuccess;
    }
    cudaGraph_t graph = nullptr;
    const bool ended = cudaStreamEndCapture(cs, &graph) == cudaSuccess;
    ok = ok && ended && graph;
    if (ok) {
        size_t nn = 0;
        ok = cudaGraphGetNodes(graph, nullptr, &nn) == cudaSuccess;
        std::vector<cudaGraphNode_t> nodes(nn);
        if (ok && nn) ok = cudaGraphGetNodes(graph, nodes.data(), &nn) == cudaSuccess;
        for (size_t k = 0; ok && k < nn; k++) {
            cudaGraphNodeType t;
            ok = cudaGraphNodeGetType(nodes[k], &t) == cudaSuccess;
            plan->n_kernels += ok && t == cudaGraphNodeTypeKernel;
        }
    }
    plan->graph = graph;
    if (ok) ok = cudaGraphInstantiate(&plan->exec, graph, 0) == cudaSuccess;
    cudaStreamDestroy(cs);
    if (!ok) {
        cudaGetLastError();
        delete plan;
        return BSR_ERR_CUDA;
    }
    *out = plan;
    return BSR_OK;
}

bsr_status_t bsr_plan_launch(bsr_plan_t plan, void *stream) {
    if (!plan) return BSR_ERR_INVALID_ARG;
    DeviceGuard g(plan->device);
    if (!g.ok) return BSR_ERR_CUDA;
    if (cudaGraphLaunch(plan->exec, static_cast<cudaStream_t>(stream)) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    return BSR_OK;
}

bsr_status_t bsr_plan_get_order(bsr_plan_t plan, int *order, int *call, int n, int *n_kernels) {
    if (!plan || n < 0) return BSR_ERR_INVALID_ARG;
    for (int k = 0; k < n; k++) {
        const bool run = k < (int)plan->order.size();
        if (order) order[k] = run ? plan->order[(size_t)k] : -1;
        if (call) call[k] = run ? plan->call[(size_t)k] : -1;
    }
    if (n_kernels) *n_kernels = plan->n_kernels;
    return BSR_OK;
}

void bsr_plan_destroy(bsr_plan_t plan) { delete plan; }

bsr_status_t bsr_check_device_status(bsr_handle_t h) {
    if (!h) return BSR_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    if (!g.ok) return BSR_ERR_CUDA;
    int v = 0;
    if (cudaDeviceSynchronize() != cudaSuccess ||
        cudaMemcpy(&v, h->d_status, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemset(h->d_status, 0, sizeof v) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    if (v == DEV_TIMEOUT) return BSR_ERR_TIMEOUT;
    return BSR_OK;
}

bsr_status_t bsr_get_schedule(bsr_handle_t h, char *buf, size_t len) {
    if (!h || !buf || len == 0) return BSR_ERR_INVALID_ARG;
    const Schedule &sc = *h->sched;
    int64_t split_rows = 0;   // rows split into pieces (the other reduce entries are empty rows)
    for (const Split &sp : sc.splits) split_rows += sp.nslot > 0;
    char stacks[160] = "";   // per tensor-core task size 1, 2, 4, ...: chunks run as stacked MMAs
    for (int gi = 0; gi < kTcTaskSizes; gi++) {
        const size_t at = strlen(stacks);
        snprintf(stacks + at, sizeof stacks - at, gi ? ",%" PRId64 : "%" PRId64,
                 sc.variant == V_TC ? sc.tc.stacks[gi] : (int64_t)0);
    }
    char gks[64] = "";   // task sizes the gathered-K kernel can run
    for (int gi = 0; gi < kGkTaskSizes; gi++) {
        if (sc.gk.off[gi] < 0) continue;
        const size_t at = strlen(gks);
        snprintf(gks + at, sizeof gks - at, at ? ",%d" : "%d", kGkG[gi]);
    }
    if (!gks[0]) snprintf(gks, sizeof gks, "none");
    char xss[64] = "";   // task sizes the SIMT kernel can run (blobs built and within shared memory)
    for (int gi = 0; gi < kXsTaskSizes && sc.variant == V_XSTAGE; gi++) {
        if (sc.xs_blob_off[gi] < 0) continue;
        const size_t at = strlen(xss);
        snprintf(xss + at, sizeof xss - at, at ? ",%d" : "%d", kXsG[gi]);
    }
    if (!xss[0]) snprintf(xss, sizeof xss, "none");
    snprintf(buf, len,
             "variant=%s\ndtype=%s\nR=%d\nC=%d\nexec_R=%d\nexec_C=%d\nM=%" PRId64 "\nK=%" PRId64 "\nMB=%" PRId64
             "\nKB=%" PRId64 "\nnnzb=%" PRId64 "\ntokens_per_cta=%d\nthreads=%d\nsmem_bytes=%zu\n"
             "item_groups=%d\nitems=%zu\nsplit_len=%d\nsplit_rows=%" PRId64 "\nslots=%d\n"
             "empty_rows=%" PRId64 "\nmax_row_blocks=%" PRId64 "\nlaunches_per_call=%d\n"
             "structure_hash=%016" PRIx64 "\ncache_hit=%d\nschedule_reuses=%" PRId64
             "\ncache_hits_total=%" PRId64 "\ncache_misses_total=%" PRId64 "\ntc_stacked_chunks=%s\n"
             "gk_task_sizes=%s\nxstage_task_sizes=%s\n",
             variant_name(sc.variant), sc.dt == BSR_F32 ? "f32" : "bf16", sc.R, sc.C, sc.ex_R, sc.ex_C, sc.M, sc.K,
             sc.MB, sc.KB, sc.nnzb, sc.tn, sc.threads, sc.smem, sc.groups, sc.items.size(),
             sc.split_len, split_rows, sc.n_slots, sc.empty_rows, sc.max_row, launches_per_call(sc),
             sc.hash, (int)h->cache_hit, (int64_t)sc.reuse_count, (int64_t)g_cache_hits,
             (int64_t)g_cache_misses, stacks, gks, xss);
    return BSR_OK;
}

void bsr_destroy(bsr_handle_t h) {
    if (!h) return;
    {
        DeviceGuard g(h->device);
        cudaFree(h->d_status);
        cudaFree(h->ws);
        cudaFree(h->stage_x);
        cudaFree(h->stage_y);
        cudaFree(h->data_packed);
    }
    {
        std::lock_guard<std::mutex> lk(g_cache_mu);
        h->sched.reset();
    }
    delete h;
}

}  // extern "C"
