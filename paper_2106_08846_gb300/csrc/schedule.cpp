// Work list, load balancing and kernel selection: the GPU stand-in for the
// TVM task scheduler of Section 2.2, which tunes each BSR task for the
// hardware and groups tasks by their sparsity structure.
//
// A schedule turns the block rows into work items. Rows much longer than the
// mean are split into pieces whose fp32 partial tiles are summed by a reduce
// pass in a fixed order (so results do not depend on timing). Empty rows stay
// as items so that their outputs receive the bias. Items are ordered longest
// first, the classic LPT rule, so that the long ones start early (except for
// one-row blocks, which keep row order).
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <numeric>
#include <queue>
#include <string>

#include "gk_plan.h"
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

// Splits rows longer than `limit` blocks into ceil(len/limit) near-equal
// pieces; orders the items longest first (LPT). With `drop_empty`, rows
// without blocks get no item: the reduce pass writes their bias (a split
// with no slots), so no CTA streams X for them.
void make_items(Schedule &sc, int64_t limit, bool drop_empty = false) {
    sc.items.clear();
    sc.splits.clear();
    sc.n_slots = 0;
    sc.split_len = (int)std::min<int64_t>(limit, INT32_MAX);
    for (int64_t i = 0; i < sc.MB; i++) {
        int32_t p0 = sc.indptr[i], p1 = sc.indptr[i + 1];
        int64_t len = p1 - p0;
        if (drop_empty && len == 0) {
            sc.splits.push_back({(int32_t)i, 0, 0, 0});
            continue;
        }
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
    // One-row blocks keep rows close together: a task's rows then share the
    // cache lines of Y its output pass writes. Inside each group of twice the
    // consumer warps (a task of two rows per warp), the longest row is paired
    // with the shortest, the second longest with the second shortest, and so
    // on: warp w owns positions 2w and 2w + 1, so its work is about the mean
    // (in tasks of four rows per warp it owns two such pairs).
    if (sc.R == 1) {
        const size_t grp = 2 * kXsConsumerWarpsR1;
        std::vector<Item> g;
        for (size_t at = 0; at < sc.items.size(); at += grp) {
            const size_t n = std::min(grp, sc.items.size() - at);
            g.assign(sc.items.begin() + (int64_t)at, sc.items.begin() + (int64_t)(at + n));
            std::stable_sort(g.begin(), g.end(), [](const Item &a, const Item &b) { return a.p1 - a.p0 > b.p1 - b.p0; });
            for (size_t k = 0; k < n; k++)
                sc.items[at + k] = k % 2 == 0 ? g[k / 2] : g[n - 1 - k / 2];
        }
        return;
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

// One-column blocks: the lanes of a warp read the X columns of NKS (up to 4)
// blocks at once; under the 128-byte swizzle two columns conflict in shared
// memory when they share a residue (column mod 4 for fp32, (column / 2) mod 4
// for bf16). Reorder the blocks [lo, hi) of one item's chunk so that every
// aligned group of four has distinct residues where the counts allow:
// repeatedly take one block from each of the fullest residue classes.
void quad_order(const Schedule &sc, int32_t *perm, int32_t lo, int32_t hi) {
    std::vector<int32_t> cls[4];
    for (int32_t k = lo; k < hi; k++) {
        const int32_t p = perm[k];
        const int64_t col = sc.indices[p];
        const int r = (int)(sc.dt == BSR_F32 ? (col & 3) : ((col >> 1) & 3));
        cls[r].push_back(p);
    }
    size_t at[4] = {0, 0, 0, 0};
    int32_t k = lo;
    while (k < hi) {
        int order[4] = {0, 1, 2, 3};
        std::sort(order, order + 4, [&](int a, int b) {
            const size_t ra = cls[a].size() - at[a], rb = cls[b].size() - at[b];
            return ra != rb ? ra > rb : a < b;
        });
        int taken = 0;
        for (int t = 0; t < 4 && k < hi; t++) {
            const int r = order[t];
            if (at[r] < cls[r].size()) {
                perm[k++] = cls[r][at[r]++];
                taken++;
            }
        }
        // fewer than four classes left: fill the group from the fullest ones
        for (int t = 0; taken < 4 && k < hi; t = (t + 1) % 4) {
            const int r = order[t];
            if (at[r] < cls[r].size()) {
                perm[k++] = cls[r][at[r]++];
                taken++;
            }
        }
    }
}

// For each task size G, the largest block-value and index footprint over
// the tasks formed by G consecutive items of the (LPT-ordered) item list.
// Per-item records fetched by the kernels: one int per block (`value` of its
// block column) padded to 4, then the first block of each chunk of `chunk`
// columns (nchunks + 1 entries) padded to 4.
template <typename F>
void build_records(Schedule &sc, int chunk, F value) {
    const int64_t nch = (sc.K + chunk - 1) / chunk;
    const int bi = xstage_block_ints(sc.R, sc.C);
    sc.xs_rec.clear();
    sc.xs_rec_off.assign(sc.items.size(), 0);
    sc.xs_perm.assign((size_t)sc.nnzb, 0);
    for (size_t i = 0; i < sc.items.size(); i++) {
        const Item &it = sc.items[i];
        const int32_t len = it.p1 - it.p0;
        sc.xs_rec_off[i] = (int32_t)sc.xs_rec.size();
        const size_t base = sc.xs_rec.size();
        sc.xs_rec.resize(base + (size_t)xstage_record_ints(len, nch, bi), 0);
        int32_t b = 0;
        const size_t cbase = base + (size_t)xstage_pad4(bi * len);
        for (int64_t c = 0; c <= nch; c++) {
            const int64_t first_col = c * (chunk / sc.C);
            while (b < len && sc.indices[it.p0 + b] < first_col) b++;
            sc.xs_rec[cbase + c] = b;
        }
        // block order inside each chunk (perm: position -> stored block)
        for (int32_t k = 0; k < len; k++) sc.xs_perm[(size_t)it.p0 + k] = it.p0 + k;
        if (sc.C == 1)
            for (int64_t c = 0; c < nch; c++)
                quad_order(sc, sc.xs_perm.data() + it.p0, sc.xs_rec[cbase + c], sc.xs_rec[cbase + c + 1]);
        for (int32_t k = 0; k < len; k++)   // (a 1x1 block's weight slot is filled by the value packing)
            sc.xs_rec[base + (size_t)bi * k] = value((int64_t)sc.indices[sc.xs_perm[(size_t)it.p0 + k]]);
    }
}

// For each task size G, the largest block-value and record footprint (bytes,
// each item's values padded to 16 bytes) over the tasks formed by G
// consecutive items.
void footprints(const Schedule &sc, size_t per_block, int chunk, const int *Gs, int nG, size_t *wbytes,
                size_t *ibytes) {
    const int64_t nch = (sc.K + chunk - 1) / chunk;
    for (int gi = 0; gi < nG; gi++) {
        const int G = Gs[gi];
        size_t wmax = 0, imax = 0, swmax = 0;
        for (size_t t = 0; t < sc.items.size(); t += G) {
            size_t blocks = 0, rec = 0;
            for (size_t k = t; k < std::min(sc.items.size(), t + G); k++) {
                const int64_t len = sc.items[k].p1 - sc.items[k].p0;
                blocks += (size_t)xstage_pad4(len * (int64_t)per_block / 4) * 4;
                rec += (size_t)xstage_record_ints(len, nch, xstage_block_ints(sc.R, sc.C)) * 4;
            }
            wmax = std::max(wmax, blocks);
            imax = std::max(imax, rec);
        }
        wbytes[gi] = wmax;
        ibytes[gi] = imax;
    }
}

void plan_xstage(Schedule &sc) {
    build_records(sc, kXsChunk, [&](int64_t col) {
        return sc.C == 1 ? (int32_t)xstage_stage_offset(sc.dt, (int)(col % kXsChunk)) : (int32_t)col;
    });
    const int bi = xstage_block_ints(sc.R, sc.C);
    const int per_block = bi == 2 ? 0 : sc.R * sc.C * kXsWDup;   // floats in the value region (1x1: in the records)
    footprints(sc, (size_t)per_block * 4, kXsChunk, kXsG, kXsTaskSizes, sc.xs.task_wbytes, sc.xs.task_ibytes);
    // the task blobs of every task size that fits: layout, then the template
    const int64_t n = (int64_t)sc.items.size();
    const int64_t nch = (sc.K + kXsChunk - 1) / kXsChunk;
    int64_t total = 0;
    for (int gi = 0; gi < kXsTaskSizes; gi++) {
        const int G = kXsG[gi];
        const size_t wb = (sc.xs.task_wbytes[gi] + 15) & ~size_t(15), ib = (sc.xs.task_ibytes[gi] + 15) & ~size_t(15);
        sc.xs_blob_off[gi] = -1;
        if (!xstage_task_size_ok(sc.R, G) ||
            xstage_smem_bytes(sc.dt, sc.R, sc.K, G, wb, ib) > (size_t)kXsMaxSmem)
            continue;
        sc.xs_blob_stride[gi] = (int64_t)G * kXsItab * 4 + (int64_t)ib + (int64_t)wb;
        sc.xs_blob_off[gi] = (total + 255) & ~int64_t(255);
        total = sc.xs_blob_off[gi] + (n + G - 1) / G * sc.xs_blob_stride[gi];
    }
    sc.xs_blob.assign((size_t)(total / 4), 0);
    sc.xs_vdst.assign((size_t)(kXsTaskSizes * n), -1);
    for (int gi = 0; gi < kXsTaskSizes; gi++) {
        if (sc.xs_blob_off[gi] < 0) continue;
        const int G = kXsG[gi];
        const int64_t ib = ((int64_t)sc.xs.task_ibytes[gi] + 15) & ~int64_t(15);
        for (int64_t t = 0; t * G < n; t++) {
            const int64_t blob = (sc.xs_blob_off[gi] + t * sc.xs_blob_stride[gi]) / 4;   // ints
            const int64_t recs = blob + (int64_t)G * kXsItab, vals = recs + ib / 4;
            int64_t woff = 0, roff = 0;
            for (int64_t k = 0; k < G && t * G + k < n; k++) {
                const int64_t i = t * G + k;
                const Item &it = sc.items[(size_t)i];
                const int64_t len = it.p1 - it.p0, rints = xstage_record_ints(len, nch, bi);
                int32_t *h = &sc.xs_blob[(size_t)(blob + k * kXsItab)];
                h[0] = it.row;
                h[1] = it.p0;
                h[2] = it.p1;
                h[3] = it.slot;
                h[5] = (int32_t)len;
                h[7] = (int32_t)woff;
                h[8] = (int32_t)roff;
                std::copy(sc.xs_rec.begin() + sc.xs_rec_off[(size_t)i], sc.xs_rec.begin() + sc.xs_rec_off[(size_t)i] + rints,
                          sc.xs_blob.begin() + (recs + roff));
                if (len) sc.xs_vdst[(size_t)(gi * n + i)] = bi == 2 ? recs + roff + 1 : vals + woff;
                woff += xstage_pad4(len * per_block);
                roff += rints;
            }
        }
    }
}

// Tasks of the tensor-core kernel for every task size G: ceil(items / G)
// tasks of at most G items each, balanced by work (a CTA's MMAs follow its
// blocks): the items, longest first, each go to the least-loaded task that
// still has room (ties: the lower task). Each task's record carries its items,
// its chunk starts and its MMA entries; its block values are packed task by
// task, chunk by chunk. bf16 chunks in which every item of the task has one
// block at the same column offset, all first or all not first, become stacks
// (see tc.h): one MMA of N = g * R per K slice instead of g. An MMA of M = 128
// and K = 16 costs one unit (about 39 SM cycles, the A tile's shared-memory
// read) up to N of about 78 and N / 78 units above (the arithmetic).
void plan_tc(Schedule &sc) {
    const int kc = tc_chunk_cols(sc.dt);
    const int64_t es = (int64_t)dtype_size(sc.dt);
    const int64_t nch = (sc.K + kc - 1) / kc;
    const size_t per_block = tc_block_bytes(sc.R, sc.C, sc.dt);
    const int64_t n_items = (int64_t)sc.items.size();
    const double block_units = sc.dt == BSR_F32 ? 3.0 * sc.C / 8.0 : sc.C / 16.0;
    const bool can_stack = sc.dt == BSR_BF16 && sc.C >= 32;
    int64_t total = 0;   // bytes of packed values over all usable G
    for (int gi = 0; gi < kTcTaskSizes; gi++) {
        const int G = kTcG[gi];
        std::vector<int32_t> &rec = sc.tc.rec[gi];
        std::vector<int32_t> &off = sc.tc.rec_off[gi];
        std::vector<int32_t> &order = sc.tc.worder[gi];
        std::vector<int32_t> &stack = sc.tc.wstack[gi];
        rec.clear();
        off.clear();
        order.clear();
        stack.clear();
        sc.tc.task_cost_max[gi] = 0;
        sc.tc.stacks[gi] = 0;
        size_t wmax = 0, imax = 0, swmax = 0;
        const int64_t n_tasks = (n_items + G - 1) / G;
        std::vector<std::vector<int32_t>> members((size_t)n_tasks);
        {
            using Load = std::pair<int64_t, int64_t>;   // (blocks, task)
            std::priority_queue<Load, std::vector<Load>, std::greater<Load>> open;
            for (int64_t t = 0; t < n_tasks; t++) open.push({0, t});
            for (int64_t k = 0; k < n_items; k++) {
                const Load l = open.top();
                open.pop();
                members[(size_t)l.second].push_back((int32_t)k);
                if ((int)members[(size_t)l.second].size() < G)
                    open.push({l.first + sc.items[(size_t)k].p1 - sc.items[(size_t)k].p0, l.second});
            }
        }
        std::vector<std::vector<int32_t>> per_chunk((size_t)nch), src((size_t)nch);
        for (int64_t t = 0; t < n_tasks; t++) {
            for (auto &v : per_chunk) v.clear();
            for (auto &v : src) v.clear();
            const std::vector<int32_t> &mem = members[(size_t)t];
            const int g_count = (int)mem.size();
            for (int g = 0; g < g_count; g++) {
                const Item &it = sc.items[(size_t)mem[(size_t)g]];
                for (int32_t b = 0; b < it.p1 - it.p0; b++) {
                    const int64_t col = sc.indices[it.p0 + b];
                    const int64_t c = (col * sc.C) / kc;
                    const int32_t a32 = (int32_t)(((col * sc.C) % kc) * es / 32);
                    per_chunk[(size_t)c].push_back(a32 | (g << 2) | ((b == 0) << 7));
                    src[(size_t)c].push_back(it.p0 + b);
                }
            }
            off.push_back((int32_t)rec.size());
            const size_t head = rec.size();
            const size_t items_at = head + 4 + (size_t)tc_pad4(nch + 1);
            rec.resize(items_at + 4 * (size_t)g_count, 0);
            rec[head + 0] = (int32_t)order.size();   // the task's first packed block
            rec[head + 1] = g_count;
            int32_t n = 0;
            for (int64_t c = 0; c < nch; c++) {
                rec[head + 4 + (size_t)c] = n;
                n += (int32_t)per_chunk[(size_t)c].size();
                wmax = std::max(wmax, per_chunk[(size_t)c].size() * per_block);
            }
            rec[head + 4 + (size_t)nch] = n;
            for (int64_t c0 = 0; c0 < nch; c0 += tcp_stage_chunks(sc.dt)) {
                size_t nb = 0;
                for (int64_t c = c0; c < std::min<int64_t>(nch, c0 + tcp_stage_chunks(sc.dt)); c++)
                    nb += per_chunk[(size_t)c].size();
                swmax = std::max(swmax, nb * per_block);
            }
            // stacks, and the task's MMA cost
            double cost = 0.0;
            for (int64_t c = 0; c < nch; c++) {
                std::vector<int32_t> &pc = per_chunk[(size_t)c];
                bool st = can_stack && g_count >= 2 && g_count * sc.R <= 256 && (int)pc.size() == g_count;
                for (int g = 0; st && g < g_count; g++)
                    st = ((pc[(size_t)g] >> 2) & 31) == g && (pc[(size_t)g] & 3) == (pc[0] & 3) &&
                         ((pc[(size_t)g] >> 7) & 1) == ((pc[0] >> 7) & 1);
                if (st) {
                    pc[0] |= 1 << 8;
                    sc.tc.stacks[gi]++;
                    for (int g = 1; g < g_count; g++) pc[(size_t)g] |= 1 << 9;
                    cost += (sc.C / 16.0) * std::max(1.0, g_count * sc.R / 78.0);
                } else {
                    cost += block_units * (double)pc.size();
                }
                for (int g = 0; g < (int)pc.size(); g++) stack.push_back(st ? (g << 16) | g_count : 1);
            }
            sc.tc.task_cost_max[gi] = std::max(sc.tc.task_cost_max[gi], (int64_t)std::ceil(cost));
            for (int g = 0; g < g_count; g++) {
                const Item &it = sc.items[(size_t)mem[(size_t)g]];
                rec[items_at + 4 * (size_t)g + 0] = it.row;
                rec[items_at + 4 * (size_t)g + 1] = it.p0;
                rec[items_at + 4 * (size_t)g + 2] = it.p1;
                rec[items_at + 4 * (size_t)g + 3] = it.slot;
            }
            for (int64_t c = 0; c < nch; c++) {
                rec.insert(rec.end(), per_chunk[(size_t)c].begin(), per_chunk[(size_t)c].end());
                order.insert(order.end(), src[(size_t)c].begin(), src[(size_t)c].end());
            }
            rec.resize(items_at + 4 * (size_t)g_count + (size_t)tc_pad4(n), 0);
            imax = std::max(imax, (rec.size() - head) * 4);
        }
        sc.tc.task_wbytes[gi] = (wmax + 15) & ~size_t(15);
        sc.tc.tcp_wbytes[gi] = (swmax + 15) & ~size_t(15);
        sc.tc.task_ibytes[gi] = imax;
        const bool ok = G * sc.R <= kTcTmemCols &&
                        tc_smem_bytes(sc.R, G, sc.tc.task_wbytes[gi], imax, sc.dt) <= (size_t)kTcMaxSmem &&
                        (int64_t)order.size() < INT32_MAX && (int64_t)rec.size() < INT32_MAX;
        sc.tc.w_off[gi] = ok ? (total + 255) & ~int64_t(255) : -1;
        if (ok) total = sc.tc.w_off[gi] + (int64_t)order.size() * (int64_t)per_block;
        else order.clear();
    }
    sc.tc_w_total = total;
}

// Small or narrow bf16 blocks on the tensor cores: the kept blocks of each
// group of max(R, 16) rows, grouped by 64-column tile, become dense
// max(R, 16) x 64 tiles with zeros for absent blocks -- a gathered-K product
// whose gather is replaced by zero padding. Worth it while the tiles are
// dense enough (below). Fills the tile structure (ptr, ind) and vmap; false
// if the shape or density does not fit.
bool reblock_for_tc(const Schedule &sc, std::vector<int32_t> &ptr, std::vector<int32_t> &ind,
                    std::vector<int32_t> &vmap, int *RT_out) {
    const bool r_ok = sc.R == 1 || sc.R == 2 || sc.R == 4 || sc.R == 8 || sc.R == 16 || sc.R == 32 ||
                      sc.R == 64 || sc.R == 128;
    const bool c_ok = sc.C == 1 || sc.C == 2 || sc.C == 4 || sc.C == 8 || sc.C == 16 || sc.C == 32;
    const int RT = std::max(sc.R, 16);   // tile height: blocks of fewer rows stack 16 / R block rows
    if (sc.dt != BSR_BF16 || !r_ok || !c_ok || sc.M % RT != 0 || sc.K % 8 != 0 || sc.nnzb == 0) return false;
    const int64_t tw = 64 / sc.C;        // block columns per tile
    const int64_t g = RT / sc.R;         // block rows per tile row
    const int64_t MBT = sc.M / RT;
    ptr.assign((size_t)MBT + 1, 0);
    ind.clear();
    vmap.assign((size_t)sc.nnzb, 0);
    std::vector<int32_t> cols;
    for (int64_t it = 0; it < MBT; it++) {
        // the tile row's tiles: every tile column any of its block rows touches
        cols.clear();
        for (int64_t i = it * g; i < (it + 1) * g; i++)
            for (int32_t p = sc.indptr[i]; p < sc.indptr[i + 1]; p++) cols.push_back((int32_t)(sc.indices[p] / tw));
        std::sort(cols.begin(), cols.end());
        cols.erase(std::unique(cols.begin(), cols.end()), cols.end());
        const int64_t first = (int64_t)ind.size();
        ind.insert(ind.end(), cols.begin(), cols.end());
        if ((int64_t)ind.size() * RT * 64 > INT32_MAX) return false;
        for (int64_t i = it * g; i < (it + 1) * g; i++) {
            const int64_t row_off = (i - it * g) * sc.R;
            for (int32_t p = sc.indptr[i]; p < sc.indptr[i + 1]; p++) {
                const int64_t t = sc.indices[p] / tw;
                const int64_t k = first + (std::lower_bound(cols.begin(), cols.end(), (int32_t)t) - cols.begin());
                vmap[(size_t)p] = (int32_t)((k * RT + row_off) * 64 + (sc.indices[p] % tw) * sc.C);
            }
        }
        ptr[(size_t)it + 1] = (int32_t)ind.size();
    }
    *RT_out = RT;
    // Worth it when the kept elements fill enough of the tiles. A tile costs
    // the tensor cores about the same whatever its fill (the MMA issue rate
    // binds), while the SIMT kernel's cost follows the kept elements. Measured
    // (two tensor-core CTAs per SM): on 768 x 768 bf16 weights at 80% sparsity
    // and 1024 tokens (fill about 0.2) the tiles took 17-19 us against the SIMT
    // kernel's 19-42 us for every shape from 1x1 to 32x1; on a 1024 x 1024
    // 32x1 weight at 90% with 16384 tokens (fill 0.10) 111 us against 166 us.
    // So blocks move while they fill at least 1/12 of the tiles.
    const int64_t need = 12;
    return sc.nnzb * sc.R * sc.C * need >= (int64_t)ind.size() * RT * 64;
}

const char *env_str(const char *name) {
    const char *v = getenv(name);
    return v && *v ? v : nullptr;
}

}  // namespace

bsr_status_t build_schedule(Schedule &sc) {
    row_stats(sc);
    sc.threads = 256;
    sc.groups = 1;
    sc.smem = 0;
    if (cudaDeviceGetAttribute(&sc.sm_count, cudaDevAttrMultiProcessorCount, sc.device) != cudaSuccess) {
        cudaGetLastError();
        sc.sm_count = 148;
    }
    const char *force = env_str("BSR_FORCE_VARIANT");
    const bool want_generic = force && std::string(force) == "generic";
    const bool want_xstage = force && std::string(force) == "xstage";
    sc.ex_C = sc.C;
    sc.ex_R = sc.R;
    sc.ex_nnzb = sc.nnzb;
    std::vector<int32_t> tptr, tind;
    int RT = sc.R;
    const bool reblock = !want_generic && !want_xstage && !tc_supports(sc.R, sc.C, sc.dt, sc.K, sc.M * sc.K) &&
                         reblock_for_tc(sc, tptr, tind, sc.vmap, &RT);
    if (!reblock) sc.vmap.clear();
    if (!want_generic && !want_xstage && (reblock || tc_supports(sc.R, sc.C, sc.dt, sc.K, sc.M * sc.K))) {
        // plan on the tile structure (the user's arrays stay the cache key)
        std::vector<int32_t> uptr, uind;
        const int uC = sc.C, uR = sc.R;
        const int64_t unnzb = sc.nnzb, uKB = sc.KB, uMB = sc.MB;
        if (reblock) {
            uptr.swap(sc.indptr);
            uind.swap(sc.indices);
            sc.indptr.swap(tptr);
            sc.indices.swap(tind);
            sc.C = 64;
            sc.R = RT;
            sc.MB = sc.M / RT;
            sc.nnzb = sc.indptr.back();
            sc.KB = (sc.K + 63) / 64;
            sc.ex_C = 64;
            sc.ex_R = RT;
            sc.ex_nnzb = sc.nnzb;
            row_stats(sc);
        }
        sc.variant = V_TC;
        sc.tn = kTcTokens;
        sc.threads = tc_threads(sc.dt == BSR_F32);
        // block values stream per chunk: only balance decides the splitting
        make_items(sc, split_limit(sc), true);
        plan_tc(sc);
        plan_tcp(sc);
        if (reblock) {
            sc.indptr.swap(uptr);
            sc.indices.swap(uind);
            sc.C = uC;
            sc.R = uR;
            sc.MB = uMB;
            sc.nnzb = unnzb;
            sc.KB = uKB;
            row_stats(sc);   // the report's row statistics describe the caller's block rows
        }
    } else if (!want_generic && xstage_supports(sc.R, sc.C, sc.dt, sc.K)) {
        sc.variant = V_XSTAGE;
        sc.tn = kXsTokens;
        sc.threads = (kXsConsumerWarps + 1) * 32;
        const size_t budget = xstage_task_budget(sc.dt, sc.R, sc.K);
        const int64_t nch = (sc.K + kXsChunk - 1) / kXsChunk;
        const int64_t avail = (int64_t)budget - 4 * xstage_pad4(nch + 1) - 16;
        const int64_t lmax =
            std::max<int64_t>(1, avail / (int64_t)((size_t)sc.R * sc.C * 4 * kXsWDup + 4));
        int64_t limit = split_limit(sc);
        limit = limit ? std::min(limit, lmax) : (sc.max_row > lmax ? lmax : 0);
        make_items(sc, limit, sc.R > 1);   // one-row blocks keep their rare empty rows: tasks stay row-contiguous
        plan_xstage(sc);
    }
    if (sc.variant == V_XSTAGE && (int64_t)sc.xs_blob.size() > INT32_MAX) sc.variant = V_GENERIC;   // blob offsets are int32
    // the gathered-K kernel, after the variant's own packed values (the
    // generic kernel's: a copy of the caller's block values)
    if (sc.variant == V_TC)
        plan_gk(sc, sc.tc_w_total);
    else if (sc.variant == V_XSTAGE)
        plan_gk(sc, (int64_t)sc.xs_blob.size() * 4);
    else
        plan_gk(sc, sc.nnzb * sc.R * sc.C * (int64_t)dtype_size(sc.dt));
    if (sc.variant == V_GENERIC) {
        sc.threads = 256;
        sc.xs_rec.clear();
        sc.xs_rec_off.clear();
        sc.xs_perm.clear();
        sc.xs_blob.clear();
        sc.xs_vdst.clear();
        sc.tn = std::max(1, 256 / std::min(sc.R, 256));
        make_items(sc, split_limit(sc));
    }
    sc.group_begin = {0, (int32_t)sc.items.size()};
    if (upload(&sc.d_items, sc.items) != cudaSuccess || upload(&sc.d_splits, sc.splits) != cudaSuccess ||
        upload(&sc.d_group_begin, sc.group_begin) != cudaSuccess ||
        upload(&sc.d_indptr, sc.indptr) != cudaSuccess || upload(&sc.d_indices, sc.indices) != cudaSuccess ||
        upload(&sc.d_xs_perm, sc.xs_perm) != cudaSuccess || upload(&sc.d_xs_vdst, sc.xs_vdst) != cudaSuccess ||
        upload(&sc.d_vmap, sc.vmap) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_ALLOC;
    }
    for (int gi = 0; gi < kGkTaskSizes; gi++)
        if (upload(&sc.gk.d_rec[gi], sc.gk.rec[gi]) != cudaSuccess ||
            upload(&sc.gk.d_rec_off[gi], sc.gk.rec_off[gi]) != cudaSuccess ||
            upload(&sc.gk.d_wsrc[gi], sc.gk.wsrc[gi]) != cudaSuccess ||
            upload(&sc.gk.d_wslot[gi], sc.gk.wslot[gi]) != cudaSuccess ||
            upload(&sc.gk.d_wbase[gi], sc.gk.wbase[gi]) != cudaSuccess ||
            upload(&sc.gk.d_prog[gi], sc.gk.prog[gi]) != cudaSuccess) {
            cudaGetLastError();
            return BSR_ERR_ALLOC;
        }
    for (int gi = 0; gi < kTcTaskSizes; gi++)
        if (upload(&sc.tc.d_rec[gi], sc.tc.rec[gi]) != cudaSuccess ||
            upload(&sc.tc.d_rec_off[gi], sc.tc.rec_off[gi]) != cudaSuccess ||
            upload(&sc.tc.d_worder[gi], sc.tc.worder[gi]) != cudaSuccess ||
            upload(&sc.tc.d_wstack[gi], sc.tc.wstack[gi]) != cudaSuccess ||
            upload(&sc.tc.d_prog[gi], sc.tc.prog[gi]) != cudaSuccess ||
            upload(&sc.tc.d_stab[gi], sc.tc.stab[gi]) != cudaSuccess) {
            cudaGetLastError();
            return BSR_ERR_ALLOC;
        }
    return BSR_OK;
}

bsr_status_t pack_data(Handle &h) {
    h.data_packed = nullptr;
    const Schedule &sc = *h.sched;
    if (sc.variant == V_TC && sc.ex_nnzb == 0 && !sc.gk.ok) return BSR_OK;
    if (sc.variant != V_XSTAGE && sc.variant != V_TC && !sc.gk.ok) return BSR_OK;
    const size_t raw_bytes = (size_t)sc.nnzb * sc.R * sc.C * dtype_size(sc.dt);
    // xstage: the task blobs (item tables and records from the schedule's
    // template, then this handle's block values)
    size_t bytes = sc.variant == V_TC ? (size_t)sc.tc_w_total : sc.variant == V_XSTAGE ? sc.xs_blob.size() * 4 : raw_bytes;
    if (sc.gk.ok) bytes = std::max(bytes, (size_t)sc.gk.total_bytes);
    if (bytes == 0) return BSR_OK;
    if (cudaMalloc(&h.data_packed, bytes) != cudaSuccess) {
        cudaGetLastError();
        h.data_packed = nullptr;
        return BSR_ERR_ALLOC;
    }
    cudaError_t e = cudaSuccess;
    if (sc.variant == V_TC) {
        if (sc.ex_C != sc.C) {
            // re-blocked: zero-filled R x 64 tiles first, then the MMA layout
            void *tiles = nullptr;
            const size_t tbytes = (size_t)sc.ex_nnzb * sc.ex_R * 64 * 2;
            if (cudaMalloc(&tiles, tbytes) != cudaSuccess) {
                cudaGetLastError();
                return BSR_ERR_ALLOC;
            }
            e = cudaMemset(tiles, 0, tbytes);
            if (e == cudaSuccess)
                e = reblock_tc_data((const uint16_t *)h.data, sc.d_vmap, sc.nnzb, sc.R, sc.C, (uint16_t *)tiles, 0);
            for (int gi = 0; gi < kTcTaskSizes && e == cudaSuccess; gi++)
                if (sc.tc.w_off[gi] >= 0)
                    e = pack_tc_data(tiles, sc.dt, sc.tc.d_worder[gi], sc.tc.d_wstack[gi],
                                     (int64_t)sc.tc.worder[gi].size(), sc.ex_R, 64,
                                     (unsigned char *)h.data_packed + sc.tc.w_off[gi], 0);
            if (e == cudaSuccess) e = cudaDeviceSynchronize();
            cudaFree(tiles);
        } else {
            for (int gi = 0; gi < kTcTaskSizes && e == cudaSuccess; gi++)
                if (sc.tc.w_off[gi] >= 0)
                    e = pack_tc_data(h.data, sc.dt, sc.tc.d_worder[gi], sc.tc.d_wstack[gi],
                                     (int64_t)sc.tc.worder[gi].size(), sc.R, sc.C,
                                     (unsigned char *)h.data_packed + sc.tc.w_off[gi], 0);
        }
    } else if (sc.variant != V_XSTAGE) {
        // the generic kernel reads the block values from the start of the packed buffer
        e = cudaMemcpy(h.data_packed, h.data, raw_bytes, cudaMemcpyDeviceToDevice);
    } else {
        e = cudaMemcpy(h.data_packed, sc.xs_blob.data(), sc.xs_blob.size() * 4, cudaMemcpyHostToDevice);
        if (e == cudaSuccess && sc.nnzb > 0)
            e = pack_xstage_data(h.data, sc.dt, sc.d_items, sc.d_xs_perm, sc.d_xs_vdst, (int64_t)sc.items.size(),
                                 sc.R, sc.C, (float *)h.data_packed, 0);
    }
    // the gathered-K kernel's operands: zero padding, then the block values
    int64_t gk_lo = -1;
    for (int gi = 0; gi < kGkTaskSizes; gi++)
        if (sc.gk.off[gi] >= 0 && (gk_lo < 0 || sc.gk.off[gi] < gk_lo)) gk_lo = sc.gk.off[gi];
    if (e == cudaSuccess && gk_lo >= 0)
        e = cudaMemset((unsigned char *)h.data_packed + gk_lo, 0, (size_t)(sc.gk.total_bytes - gk_lo));
    for (int gi = 0; gi < kGkTaskSizes && e == cudaSuccess; gi++)
        if (sc.gk.off[gi] >= 0)
            e = pack_gk_data(h.data, sc.dt, sc.gk.d_wsrc[gi], sc.gk.d_wslot[gi], sc.gk.d_wbase[gi],
                             (int64_t)sc.gk.wsrc[gi].size(), sc.R, sc.C, h.data_packed, 0);
    if (e != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    return BSR_OK;
}

int launches_per_call(const Schedule &sc, int64_t N) {
    if (choose_gk(sc, N) >= 0) return 1;   // no split rows, no reduce pass
    return 1 + (sc.splits.empty() ? 0 : 1);
}

// Task size for this call: the G that minimises a simple cost model,
// waves * (fixed CTA cost + the work of G items), among the G whose shared
// memory fits. One CTA runs per SM. Work is counted in multiply-adds per
// token (blocks x R x C); a CTA's fixed cost (pipeline fill, streaming the
// X tile, staging, epilogue) is worth about kFixed of them, which is about
// two 32x1 rows of a 768-wide weight at 80% block sparsity.
int choose_tasks(const Schedule &sc, int64_t N) {
    static const int forced = [] {
        const char *v = getenv("BSR_XS_G");
        return v ? atoi(v) : 0;
    }();
    auto fits = [&](int G) { return sc.xs_blob_off[g_index(G)] >= 0; };   // blobs exist for G
    for (int gi = 0; gi < kXsTaskSizes; gi++)
        if (forced == kXsG[gi] && fits(forced)) return forced;
    const double kFixed = 10000.0;
    const int64_t tiles = (N + kXsTokens - 1) / kXsTokens;
    const int64_t items = (int64_t)sc.items.size();
    const double item_work = items ? (double)sc.nnzb * sc.R * sc.C / (double)items : 0.0;
    int best = 1;
    double best_cost = -1.0;
    for (int gi = 0; gi < kXsTaskSizes; gi++) {
        const int G = kXsG[gi];
        if (!fits(G)) continue;
        const int64_t tasks = (items + G - 1) / G;
        const int64_t ctas = tiles * tasks;
        const double waves = (double)((ctas + sc.sm_count - 1) / sc.sm_count);
        // a wave's CTAs carry the mean task's items: a light last task (items
        // not a multiple of G) shortens the waves it falls in
        const double cost = waves * (kFixed + (double)items / (double)std::max<int64_t>(tasks, 1) * item_work);
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            best = G;
        }
    }
    return best;
}

// Task size for the tcgen05 kernel: the G that minimises waves x (fixed CTA
// cost + the most loaded task's MMA cost), among the G whose accumulators fit
// tensor memory and whose shared memory fits; a wave is every SM holding as
// many CTAs as fit it at once. A CTA's fixed cost (tensor-memory allocation,
// barriers, work list, first stage round trip, epilogue: several microseconds
// in per-CTA phase stamps) is counted as kOverheadMma MMA units, a
// conservative weight: at 32 the model preferred five waves of two-row tasks
// to three waves of four-row tasks on Zipf rows, measured 9% slower.
int choose_tc_tasks(const Schedule &sc, int64_t N) {
    static const int forced = [] {
        const char *v = getenv("BSR_TC_G");
        return v ? atoi(v) : 0;
    }();
    auto fits = [&](int G) { return sc.tc.w_off[tc_g_index(G)] >= 0; };   // planned and packed for G
    for (int gi = 0; gi < kTcTaskSizes; gi++)
        if (forced == kTcG[gi] && fits(forced)) return forced;
    const double kOverheadMma = 64.0;
    const int64_t tiles = (N + kTcTokens - 1) / kTcTokens;
    int best = 1;
    double best_cost = -1.0;
    for (int gi = 0; gi < kTcTaskSizes; gi++) {
        const int G = kTcG[gi];
        if (!fits(G)) continue;
        const int64_t ctas = tiles * (int64_t)sc.tc.rec_off[gi].size();
        const int64_t slots = (int64_t)sc.sm_count *
                              tc_ctas_per_sm(sc.ex_R, G, sc.tc.task_wbytes[gi], sc.tc.task_ibytes[gi], sc.dt);
        const double waves = (double)((ctas + slots - 1) / slots);
        const double cost = waves * (kOverheadMma + (double)sc.tc.task_cost_max[gi]);
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            best = G;
        }
    }
    return best;
}

int fusion_class(const Schedule &sc, int64_t N, int *G) {
    if (choose_gk(sc, N) >= 0) {   // a grid of its own
        *G = 0;
        return -1;
    }
    if (sc.variant == V_XSTAGE) {
        *G = choose_tasks(sc, N);
        return 2 * xstage_fusion_key(sc, *G);
    }
    if (sc.variant == V_TC) {
        if (choose_tcp(sc, N) >= 0) {   // persistent: a grid of its own
            *G = 0;
            return -1;
        }
        *G = choose_tc_tasks(sc, N);
        return 2 * tc_fusion_key(sc) + 1;
    }
    *G = 0;
    return -1;
}

cudaError_t launch_spmm_batch(const LaunchArgs *as, int n) {
    auto fusion = [](const LaunchArgs &a, int *G) { return fusion_class(*a.sc, a.N, G); };
    std::vector<char> done((size_t)std::max(n, 0), 0);
    std::vector<LaunchArgs> grp;
    std::vector<int> gs;
    for (int i = 0; i < n; i++) {
        if (done[(size_t)i]) continue;
        int G = 0;
        const int key = fusion(as[i], &G);
        if (key < 0) {
            done[(size_t)i] = 1;
            cudaError_t e = launch_spmm(as[i]);
            if (e != cudaSuccess) return e;
            continue;
        }
        // every later product of the same class joins this grid
        const bool tc = as[i].sc->variant == V_TC;
        const int cap = tc ? kTcBatchMax : kXsBatchMax;
        grp.clear();
        gs.clear();
        for (int j = i; j < n && (int)grp.size() < cap; j++) {
            if (done[(size_t)j]) continue;
            int Gj = 0;
            if (fusion(as[j], &Gj) != key) continue;
            grp.push_back(as[j]);
            gs.push_back(Gj);
            done[(size_t)j] = 1;
        }
        const int m = (int)grp.size();
        cudaError_t e = tc ? (m == 1 ? launch_tc(grp[0], gs[0]) : launch_tc_batch(grp.data(), gs.data(), m))
                           : (m == 1 ? launch_xstage(grp[0], gs[0]) : launch_xstage_batch(grp.data(), gs.data(), m));
        if (e != cudaSuccess) return e;
        for (const LaunchArgs &a : grp)
            if (!a.sc->splits.empty() && (e = launch_reduce(a)) != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_spmm(const LaunchArgs &a) {
    const int gG = choose_gk(*a.sc, a.N);
    if (gG >= 0) return launch_gk(a, gG);   // every block row is an item: nothing to reduce
    cudaError_t e;
    const int tG = a.sc->variant == V_TC ? choose_tcp(*a.sc, a.N) : -1;
    if (tG >= 0)
        e = launch_tcp(a, tG);
    else if (a.sc->variant == V_TC)
        e = launch_tc(a, choose_tc_tasks(*a.sc, a.N));
    else if (a.sc->variant == V_XSTAGE)
        e = launch_xstage(a, choose_tasks(*a.sc, a.N));
    else
        e = launch_generic(a);
    if (e != cudaSuccess) return e;
    if (!a.sc->splits.empty()) e = launch_reduce(a);
    return e;
}

}  // namespace bsr
