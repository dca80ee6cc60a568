// Schedule of the gathered-K tensor-core kernel (spmm_gk.cu): tasks, their
// records and the packing order of their block values, for every task size.
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <queue>

#include "gk_plan.h"

namespace bsr {

namespace {

int64_t pad4(int64_t n) { return (n + 3) & ~int64_t(3); }

// Instruction descriptor of the kernel's MMAs: fp32 accumulator, A and B
// K-major, A/B tf32 (format 2) or bf16 (format 1), N = R, M = 128.
uint32_t idesc_words(bool f32, int R) {
    return (1u << 4) | ((f32 ? 2u : 1u) << 7) | ((f32 ? 2u : 1u) << 10) | ((uint32_t)(R >> 3) << 17) |
           ((uint32_t)(kGkTokens >> 4) << 24);
}

// Byte offset of chunk column kk in a gk stage at token row 0, before the
// swizzle: two boxes of 128 token rows x 128 bytes.
int32_t stage_offset(bsr_dtype_t dt, int64_t kk) {
    const int64_t es = dt == BSR_F32 ? 4 : 2, box_cols = 128 / es;
    return (int32_t)((kk / box_cols) * (128 * 128) + (kk % box_cols) * es);
}

}  // namespace

// Every block row is an item (empty rows too: their outputs are the bias).
// For each task size G the items go, most work first, to the least-loaded of
// ceil(rows / G) tasks that still has room; work = K slices of MMAs over all
// chunks (an item's blocks in a chunk, C columns each, padded up to the MMA's
// K). Per task and chunk, each item with blocks there gets an entry: its
// gathered K, its A columns in tensor memory and its B operand in the
// chunk's packed values. A chunk's entries are grouped, in order, into
// batches whose A columns fit one A buffer of tensor memory (gk_slot_cols).
void plan_gk(Schedule &sc, int64_t packed_end) {
    GkPlan &pl = sc.gk;
    pl.ok = false;
    pl.total_bytes = packed_end;
    for (int gi = 0; gi < kGkTaskSizes; gi++) {
        pl.off[gi] = -1;
        pl.rec[gi].clear();
        pl.rec_off[gi].clear();
        pl.wsrc[gi].clear();
        pl.wslot[gi].clear();
        pl.wbase[gi].clear();
        pl.prog[gi].clear();
        pl.pstage[gi] = 0;
    }
    if (packed_end < 0 || !gk_supports(sc.R, sc.C, sc.dt, sc.K) || sc.MB == 0 || sc.nnzb == 0) return;
    const bool f32 = sc.dt == BSR_F32;
    const int64_t KC = gk_chunk_cols(sc.dt), KS = gk_kslice(sc.dt);
    const int64_t nch = (sc.K + KC - 1) / KC;
    const int64_t R = sc.R, C = sc.C, MB = sc.MB;
    const int64_t bpc = KC / C;   // block columns per chunk
    // per item: slices over all chunks
    std::vector<int64_t> work((size_t)MB, 0);
    for (int64_t i = 0; i < MB; i++) {
        int32_t p = sc.indptr[i];
        while (p < sc.indptr[i + 1]) {
            const int64_t c = sc.indices[p] / bpc;
            int64_t m = 0;
            while (p < sc.indptr[i + 1] && sc.indices[p] / bpc == c) m++, p++;
            work[(size_t)i] += (m * C + KS - 1) / KS;
        }
    }
    std::vector<int64_t> order((size_t)MB);
    for (int64_t i = 0; i < MB; i++) order[(size_t)i] = i;
    std::stable_sort(order.begin(), order.end(), [&](int64_t a, int64_t b) { return work[(size_t)a] > work[(size_t)b]; });
    const int64_t mma_per_slice = f32 ? 3 : 1;
    int64_t end = (packed_end + 255) & ~int64_t(255);
    for (int gi = 0; gi < kGkTaskSizes; gi++) {
        const int G = kGkG[gi];
        const int64_t slot = gk_slot_cols(sc.R, sc.C, f32, G);
        if (!slot) continue;
        // blocks of one entry (piece): as many as fill one A buffer
        const int64_t piece = std::max<int64_t>(1, (f32 ? slot / 2 : slot * 2) / C);
        const int64_t n_tasks = (MB + G - 1) / G;
        std::vector<std::vector<int64_t>> members((size_t)n_tasks);
        {
            using Load = std::pair<int64_t, int64_t>;   // (work, task)
            std::priority_queue<Load, std::vector<Load>, std::greater<Load>> open;
            for (int64_t t = 0; t < n_tasks; t++) open.push({0, t});
            for (int64_t i : order) {
                const Load l = open.top();
                open.pop();
                members[(size_t)l.second].push_back(i);
                if ((int)members[(size_t)l.second].size() < G) open.push({l.first + work[(size_t)i], l.second});
            }
        }
        std::vector<int32_t> &rec = pl.rec[gi];
        std::vector<int32_t> &roff = pl.rec_off[gi];
        size_t wmax = 0, imax = 0;
        int64_t cost_max = 0;
        int64_t wtotal = 0;   // bytes of packed values of this task size
        std::vector<int32_t> &wsrc = pl.wsrc[gi], &wslot = pl.wslot[gi];
        std::vector<int64_t> &wbase = pl.wbase[gi];
        std::vector<uint32_t> &prog = pl.prog[gi];
        size_t pmax = 0;
        std::vector<int64_t> pos;
        const uint32_t id = idesc_words(f32, (int)R);
        for (int64_t t = 0; t < n_tasks; t++) {
            const std::vector<int64_t> &mem = members[(size_t)t];
            const int g_count = (int)mem.size();
            pos.assign((size_t)g_count, 0);
            std::vector<int32_t> cb((size_t)nch + 1, 0), cw((size_t)nch + 1, 0), cp((size_t)2 * nch, 0), be, entries,
                clist;
            // issuer of each item: contiguous ranges balanced by work
            std::vector<int> owner((size_t)g_count, 0);
            {
                int64_t tot = 0, acc = 0;
                for (int g = 0; g < g_count; g++) tot += work[(size_t)mem[(size_t)g]];
                for (int g = 0; g < g_count; g++) {
                    const int64_t w = work[(size_t)mem[(size_t)g]];
                    owner[(size_t)g] =
                        tot > 0 ? (int)std::min<int64_t>(kGkIssuers - 1, (2 * acc + w) * kGkIssuers / (2 * tot)) : 0;
                    acc += w;
                }
            }
            std::vector<std::vector<uint32_t>> words;   // per (batch of the chunk, issuer)
            std::vector<int64_t> cl_of_entry;   // column-list position of each entry (relative)
            std::vector<char> seen((size_t)g_count, 0);
            int64_t cost = 0;
            uint32_t wbytes_task = 0;
            for (int64_t c = 0; c < nch; c++) {
                cb[(size_t)c] = (int32_t)be.size();
                cw[(size_t)c] = (int32_t)(wbytes_task / 16);
                int64_t acol = slot;   // forces a new batch at the chunk's first entry
                uint32_t boff = 0;
                words.clear();
                for (int g = 0; g < g_count; g++) {
                    const int64_t i = mem[(size_t)g];
                    const int32_t p0 = sc.indptr[i] + (int32_t)pos[(size_t)g];
                    int64_t m_all = 0;
                    while (p0 + m_all < sc.indptr[i + 1] && sc.indices[p0 + m_all] / bpc == c) m_all++;
                    if (!m_all) continue;
                    pos[(size_t)g] += m_all;
                    for (int64_t q0 = 0; q0 < m_all; q0 += piece) {   // one entry per piece
                        const int64_t m = std::min(piece, m_all - q0);
                        const int32_t pq = p0 + (int32_t)q0;
                        const int64_t kpad = (m * C + KS - 1) / KS * KS;
                        const int64_t need = f32 ? 2 * kpad : kpad / 2;
                        if (acol + need > slot) {   // a new batch (a new A buffer)
                            be.push_back((int32_t)(entries.size() / kGkEntryInts));
                            acol = 0;
                            words.resize(words.size() + kGkIssuers);
                        }
                        {
                            // the entry's MMAs, K slice by K slice: bf16 one,
                            // fp32 high x high + high x low + low x high (low
                            // A parts kpad columns on, low B parts kpad R floats on)
                            std::vector<uint32_t> &wq = words[words.size() - kGkIssuers + (size_t)owner[(size_t)g]];
                            const uint32_t dcol = (uint32_t)(g * R), bslice = (uint32_t)(R * 32 / 16);
                            const bool first = !seen[(size_t)g];
                            for (int64_t q = 0; q < kpad / KS; q++) {
                                const uint32_t bh = boff / 16 + (uint32_t)q * bslice, ah = (uint32_t)(acol + 8 * q);
                                const uint32_t acc = (!first || q > 0) ? 0x80000000u : 0u;
                                wq.insert(wq.end(), {bh, dcol, ah | acc, id});
                                if (f32) {
                                    const uint32_t bl = (uint32_t)((boff + kpad * R * 4) / 16) + (uint32_t)q * bslice;
                                    wq.insert(wq.end(), {bl, dcol, ah | 0x80000000u, id});
                                    wq.insert(wq.end(), {bh, dcol, (uint32_t)(acol + kpad + 8 * q) | 0x80000000u, id});
                                }
                            }
                        }
                        entries.push_back(g);
                        entries.push_back(seen[(size_t)g] ? 0 : 1);
                        entries.push_back((int32_t)acol);
                        entries.push_back((int32_t)(kpad / KS));
                        entries.push_back((int32_t)(boff / 16));
                        entries.push_back((int32_t)m);
                        entries.push_back(0);   // column-list index, set below
                        entries.push_back(0);
                        cl_of_entry.push_back((int64_t)clist.size());
                        seen[(size_t)g] = 1;
                        for (int64_t b = 0; b < m; b++) {
                            const int64_t j = sc.indices[pq + b];
                            clist.push_back(stage_offset(sc.dt, j * C - c * KC));
                            wsrc.push_back(pq + (int32_t)b);
                            wslot.push_back((int32_t)(b * C) | (int32_t)(kpad << 16));
                            wbase.push_back(end + wtotal + wbytes_task + boff);
                        }
                        acol += need;
                        boff += (uint32_t)(kpad * R * (f32 ? 8 : 2));
                        cost += kpad / KS * mma_per_slice;
                    }
                }
                wmax = std::max(wmax, (size_t)boff);
                wbytes_task += boff;
                // the chunk's program: starts per (batch, issuer) and the end, then the words
                if (!words.empty()) {
                    const size_t at = prog.size(), nstart = words.size() + 1;
                    prog.resize(at + (size_t)pad4((int64_t)nstart), 0u);
                    uint32_t n = 0;
                    for (size_t k = 0; k < words.size(); k++) {
                        prog[at + k] = n;
                        n += (uint32_t)(words[k].size() / 4);
                    }
                    prog[at + words.size()] = n;
                    for (const auto &w : words) prog.insert(prog.end(), w.begin(), w.end());
                    cp[(size_t)(2 * c)] = (int32_t)(at / 4);
                    cp[(size_t)(2 * c + 1)] = (int32_t)((prog.size() - at) * 4);
                    pmax = std::max(pmax, (prog.size() - at) * 4);
                }
            }
            const int n_batches = (int)be.size();
            cb[(size_t)nch] = n_batches;
            cw[(size_t)nch] = (int32_t)(wbytes_task / 16);
            be.push_back((int32_t)(entries.size() / kGkEntryInts));
            const int64_t n_ent = (int64_t)cl_of_entry.size();
            // [ header | chunk batches | chunk W offsets | chunk programs | batch entries | items | entries
            //   | column list ]
            const int64_t head = (int64_t)rec.size();
            roff.push_back((int32_t)head);
            const int64_t cb_at = 4, cw_at = cb_at + pad4(nch + 1), cp_at = cw_at + pad4(nch + 1);
            const int64_t be_at = cp_at + pad4(2 * nch);
            const int64_t items_at = be_at + pad4(n_batches + 1), ent_at = items_at + 4 * g_count;
            const int64_t cl_at = ent_at + kGkEntryInts * n_ent;
            const int64_t total_ints = pad4(cl_at + (int64_t)clist.size());
            rec.resize((size_t)(head + total_ints), 0);
            int32_t *r = rec.data() + head;
            r[0] = g_count;
            r[1] = n_batches;
            r[2] = (int32_t)(wtotal / 16);
            r[3] = (int32_t)(total_ints * 4);
            std::copy(cb.begin(), cb.end(), r + cb_at);
            std::copy(cw.begin(), cw.end(), r + cw_at);
            std::copy(cp.begin(), cp.end(), r + cp_at);
            std::copy(be.begin(), be.end(), r + be_at);
            for (int g = 0; g < g_count; g++) {
                const int64_t i = mem[(size_t)g];
                r[items_at + 4 * g] = (int32_t)i;
                r[items_at + 4 * g + 1] = sc.indptr[i + 1] - sc.indptr[i];
            }
            for (int64_t e = 0; e < n_ent; e++) entries[(size_t)(kGkEntryInts * e + 6)] = (int32_t)(cl_at + cl_of_entry[(size_t)e]);
            std::copy(entries.begin(), entries.end(), r + ent_at);
            std::copy(clist.begin(), clist.end(), r + cl_at);
            imax = std::max(imax, (size_t)total_ints * 4);
            cost_max = std::max(cost_max, cost);
            wtotal += wbytes_task;
        }
        pl.n_tasks[gi] = (int)n_tasks;
        pl.wstage[gi] = (uint32_t)((wmax + 15) & ~size_t(15));
        pl.pstage[gi] = (uint32_t)((pmax + 15) & ~size_t(15));
        pl.ibytes[gi] = (uint32_t)((imax + 15) & ~size_t(15));
        pl.acols[gi] = (uint32_t)slot;
        pl.cost_max[gi] = cost_max;
        const bool fits = gk_smem_bytes(sc.dt, pl.wstage[gi] + pl.pstage[gi], pl.ibytes[gi], G, sc.R) <=
                              (size_t)kGkMaxSmem &&
                          (int64_t)rec.size() < INT32_MAX && wtotal / 16 < INT32_MAX && prog.size() / 4 < INT32_MAX;
        if (!fits) {
            rec.clear();
            roff.clear();
            wsrc.clear();
            wslot.clear();
            wbase.clear();
            prog.clear();
            continue;
        }
        pl.off[gi] = end;
        end = (end + wtotal + 255) & ~int64_t(255);
        pl.ok = true;
    }
    pl.total_bytes = end;
}

// The gk task size for a call of N tokens, or -1 (the schedule's own
// kernel). Every task re-reads X from L2 once, so the largest task size
// that still gives every SM a unit (a task on a 128-token tile) wins; below
// that, the one with the most units. By default the kernel takes the calls
// of schedules whose own kernel is the generic one (blocks the specialised
// kernels do not run, such as fp32 blocks of 64 or more rows), of 512 or more
// tokens: its MMAs have N = R outputs, and one thread issues an MMA in about
// 60 ns whatever N is, so for 16- and 32-row blocks the SIMT and tile
// kernels measured faster. BSR_GK=0 turns it off, BSR_GK=1 uses it whenever
// it fits; BSR_GK_G forces a task size.
int choose_gk(const Schedule &sc, int64_t N) {
    static const int mode = [] {
        const char *v = getenv("BSR_GK");
        return v ? atoi(v) : -1;
    }();
    static const int forced = [] {
        const char *v = getenv("BSR_GK_G");
        return v ? atoi(v) : 0;
    }();
    if (mode == 0 || !sc.gk.ok || N <= 0) return -1;
    if (mode != 1 && (N < 512 || sc.variant != V_GENERIC)) return -1;
    for (int gi = 0; gi < kGkTaskSizes; gi++)
        if (forced == kGkG[gi] && sc.gk.off[gi] >= 0) return forced;
    const int64_t tiles = (N + kGkTokens - 1) / kGkTokens;
    int most = -1;          // the task size with the most units
    int64_t most_units = 0;
    for (int gi = kGkTaskSizes - 1; gi >= 0; gi--) {   // largest first
        if (sc.gk.off[gi] < 0) continue;
        const int64_t units = tiles * sc.gk.n_tasks[gi];
        if (units >= sc.sm_count) return kGkG[gi];
        if (units > most_units) {
            most = kGkG[gi];
            most_units = units;
        }
    }
    return most;
}

}  // namespace bsr
