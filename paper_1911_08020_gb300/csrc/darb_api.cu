// darb_api.cu -- the C ABI of libdarb (include/darb.h): argument checking,
// handle lifetime, the binned device layout, and kernel launches.
#include "darb.h"
#include "darb_internal.h"
#include "launch.cuh"
#include "tma.cuh"
#include "trace.h"

#include <algorithm>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <new>
#include <numeric>
#include <unordered_set>
#include <vector>

using darb::Format;
using darb::Group;
using darb::kChunk;
using darb::kSlots;

struct darb_handle_s {
    int64_t rows = 0, cols = 0;
    darb_dtype_t wtype = DARB_F32;
    int64_t nnzb = 0;
    int32_t nbins = 0;
    // host copy of the layout
    std::vector<Group> groups;
    std::vector<int32_t> rowmap, rowloc, row_m;
    std::vector<darb::EncTile> enc_tiles;   // every encoder tile, resolved
    int32_t max_tile = 0;                   // elements of the largest encoder tile (nb * m)
    std::vector<darb::EncTile> row_tiles;   // tiles of the bf16 row encoder (empty where it does not apply)
    std::vector<darb::WorkItem> items;   // CTA work tables of every (level, split), concatenated
    int32_t item_first[darb::kWorkLevels][darb::kWorkSplits] = {};
    int32_t nitems[darb::kWorkLevels][darb::kWorkSplits] = {};
    int32_t item_work[darb::kWorkLevels][darb::kWorkSplits] = {};
    std::vector<int64_t> set_prefix[darb::kWorkLevels];   // work of the row sets of items[l][0], prefix sums
    std::vector<darb::SetGeo> xsets;                      // row sets of xres, both tables concatenated
    int32_t xset_first[darb::kXresTables] = {}, nxsets[darb::kXresTables] = {};
    std::vector<int64_t> xset_prefix[darb::kXresTables];
    darb::SetGeo *d_xsets = nullptr;
    int64_t val_elems = 0, off_words = 0;
    // device memory: one allocation holding the layout, values and offsets
    void *dmem = nullptr;
    size_t dbytes = 0;
    Group *d_groups = nullptr;
    darb::EncTile *d_tiles = nullptr, *d_row_tiles = nullptr;
    darb::WorkItem *d_items = nullptr;
    int32_t *d_rowmap = nullptr, *d_rowloc = nullptr, *d_row_m = nullptr, *d_status = nullptr;
    void *d_vals = nullptr;
    uint32_t *d_offs = nullptr;
    // PDL prefetch of the handle's data is safe only once no re-encode of it can
    // still be running: reencode_event marks the last one; in_graph disables it
    cudaEvent_t reencode_event = nullptr;
    bool reencode_pending = false;
    bool reencoded_in_graph = false;
    // RNN step scratch (grown on demand)
    float *d_gates = nullptr;
    size_t gates_cap = 0;     // floats
    int32_t *d_counters = nullptr;
    size_t counters_cap = 0;  // ints
};

namespace {

std::mutex g_mu;
std::unordered_set<const darb_handle_s *> g_live;

bool live(const darb_handle_s *h) {
    std::lock_guard<std::mutex> lk(g_mu);
    return h != nullptr && g_live.count(h) != 0;
}

// Test hook: DARB_FAIL_ALLOC=1 makes every device allocation of the library fail.
bool alloc_fault_injected() {
    const char *v = std::getenv("DARB_FAIL_ALLOC");
    return v != nullptr && v[0] == '1';
}

darb_status_t dev_alloc(void **p, size_t bytes) {
    *p = nullptr;
    if (alloc_fault_injected()) return DARB_ERR_OOM;
    const cudaError_t e = cudaMalloc(p, bytes);
    if (e == cudaErrorMemoryAllocation) {
        cudaGetLastError();
        return DARB_ERR_OOM;
    }
    if (e != cudaSuccess) {
        cudaGetLastError();
        return DARB_ERR_CUDA;
    }
    return DARB_OK;
}

inline darb_status_t cuda_status(cudaError_t e) { return e == cudaSuccess ? DARB_OK : DARB_ERR_CUDA; }

constexpr int64_t kMaxDim = int64_t(1) << 30;
constexpr int64_t kMaxBatch = int64_t(1) << 19;

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

void build_work_tables(darb_handle_s *h);

// Bin rows by block size (stable: ascending m, then ascending row) and cut
// each bin into 32-row groups.
void build_layout(darb_handle_s *h, const int32_t *m) {
    const int64_t rows = h->rows, cols = h->cols;
    std::vector<int32_t> order(static_cast<size_t>(rows));
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(), [m](int32_t a, int32_t b) { return m[a] < m[b]; });
    h->row_m.assign(m, m + rows);
    h->rowloc.assign(static_cast<size_t>(rows), -1);
    h->groups.clear();
    h->rowmap.clear();
    h->nbins = 0;
    h->nnzb = 0;
    int64_t val = 0, off = 0;
    size_t i = 0;
    while (i < order.size()) {
        const int32_t mb = m[order[i]];
        size_t e = i;
        while (e < order.size() && m[order[e]] == mb) ++e;
        ++h->nbins;
        for (size_t s = i; s < e; s += kSlots) {
            Group g{};
            g.m = mb;
            g.n = static_cast<int32_t>(ceil_div(cols, mb));
            g.nrows = static_cast<int32_t>(std::min<size_t>(kSlots, e - s));
            g.nib = mb <= 16 ? 1 : 0;
            const int64_t nch = ceil_div(g.n, kChunk);
            g.val_off = val;
            g.off_off = off;
            val += nch * kSlots * kChunk;
            off += nch * kSlots * (g.nib ? 1 : 2);
            const int32_t gi = static_cast<int32_t>(h->groups.size());
            for (int k = 0; k < kSlots; ++k) {
                if (k < g.nrows) {
                    const int32_t r = order[s + k];
                    h->rowmap.push_back(r);
                    h->rowloc[r] = gi * kSlots + k;
                } else {
                    h->rowmap.push_back(-1);
                }
            }
            h->nnzb += static_cast<int64_t>(g.n) * g.nrows;
            h->groups.push_back(g);
        }
        i = e;
    }
    h->val_elems = val;
    h->off_words = off;
    build_work_tables(h);
    // tiles of tb(m) blocks, every row in order; tb a multiple of the chunk
    auto tiles_of = [h, rows, cols](std::vector<darb::EncTile> &out, int (*tb_of)(int)) {
        out.clear();
        for (int64_t r = 0; r < rows; ++r) {
            const int32_t loc = h->rowloc[static_cast<size_t>(r)];
            const Group &g = h->groups[static_cast<size_t>(loc / kSlots)];
            const int64_t slot = loc % kSlots;
            const int tb = tb_of(g.m);
            for (int64_t jt = 0; jt < g.n; jt += tb) {
                darb::EncTile t{};
                const int64_t nb = std::min<int64_t>(tb, g.n - jt);
                const int64_t rec = (jt / kChunk) * kSlots + slot;   // jt is a multiple of the chunk
                t.row = static_cast<int32_t>(r);
                t.c0 = static_cast<int32_t>(jt * g.m);
                t.span = static_cast<int32_t>(std::min<int64_t>(cols, (jt + nb) * g.m) - jt * g.m);
                t.m = static_cast<int16_t>(g.m);
                t.nb = static_cast<int16_t>(nb);
                t.val_base = g.val_off + rec * kChunk;
                t.off_base = g.off_off + rec * (g.nib ? 1 : 2);
                out.push_back(t);
            }
        }
    };
    tiles_of(h->enc_tiles, darb::enc_tile_blocks);
    h->max_tile = 0;
    for (const darb::EncTile &t : h->enc_tiles)
        h->max_tile = std::max<int32_t>(h->max_tile, static_cast<int32_t>(t.nb) * t.m);
    bool pow2 = h->wtype == DARB_BF16;
    for (const Group &g : h->groups)
        if (g.m < 8 || g.m > 256 || (g.m & (g.m - 1)) != 0) pow2 = false;
    h->row_tiles.clear();
    if (pow2) tiles_of(h->row_tiles, [](int m) { return darb::kRowPassElems / m; });
}

// The CTA work tables of batch_kernel (darb::WorkItem).  For row sets of up to
// 2^l consecutive groups of one bin and clusters of C = 2^c CTAs, every set is
// split over k = min(C, its chunks) CTAs, each multiplying a contiguous 1/k of
// the chunks.  (Splitting the sets of heavy bins over more CTAs than those of
// light bins, to give every CTA the same work, measured slower: a light set on
// few CTAs becomes a long run of short rounds whose copies the two-stage ring
// cannot hide.)  Sets are packed into clusters by descending k (powers of two,
// so no set straddles two clusters) and the last cluster is filled with idle
// ranks.
void build_work_tables(darb_handle_s *h) {
    h->items.clear();
    for (int l = 0; l < darb::kWorkLevels; ++l) {
        const int cap = 1 << l;
        std::vector<int2> sets;   // (first group, groups)
        size_t gbeg = 0;
        while (gbeg < h->groups.size()) {
            size_t gend = gbeg;
            while (gend < h->groups.size() && h->groups[gend].m == h->groups[gbeg].m) ++gend;
            for (size_t s = gbeg; s < gend; s += cap)
                sets.push_back(make_int2(static_cast<int>(s), static_cast<int>(std::min<size_t>(cap, gend - s))));
            gbeg = gend;
        }
        auto nch_of = [h](const int2 &s) {
            return static_cast<int64_t>(ceil_div(h->groups[static_cast<size_t>(s.x)].n, kChunk));
        };
        for (int c = 0; c < darb::kWorkSplits; ++c) {
            const int C = 1 << c;
            std::vector<std::pair<int, int2>> ks;
            for (const int2 &s : sets) {
                int k = 1;
                while (2 * k <= C && 2 * k <= nch_of(s)) k *= 2;
                ks.push_back({k, s});
            }
            std::stable_sort(ks.begin(), ks.end(), [](const auto &a, const auto &b) { return a.first > b.first; });
            h->item_first[l][c] = static_cast<int32_t>(h->items.size());
            int64_t most = 0;
            for (const auto &e : ks) {
                const int k = e.first;
                const int64_t nch = nch_of(e.second);
                for (int q = 0; q < k; ++q) {
                    darb::WorkItem it{};
                    it.g0 = e.second.x;
                    it.ng = static_cast<int16_t>(e.second.y);
                    it.qsub = static_cast<int8_t>(q);
                    it.ksub = static_cast<int8_t>(k);
                    it.c0 = static_cast<int32_t>(nch * q / k);
                    it.c1 = static_cast<int32_t>(nch * (q + 1) / k);
                    most = std::max<int64_t>(most, int64_t(it.ng) * (it.c1 - it.c0));
                    h->items.push_back(it);
                }
            }
            while ((h->items.size() - h->item_first[l][c]) % C != 0) {
                darb::WorkItem idle{};
                idle.ksub = 1;
                h->items.push_back(idle);
            }
            h->nitems[l][c] = static_cast<int32_t>(h->items.size()) - h->item_first[l][c];
            h->item_work[l][c] = static_cast<int32_t>(std::min<int64_t>(most, INT32_MAX));
        }
        // the sets of items[l][0] (one CTA each, in set order) and their work
        h->set_prefix[l].assign(1, 0);
        for (const int2 &s : sets) h->set_prefix[l].push_back(h->set_prefix[l].back() + s.y * nch_of(s));
    }
    // Row sets of xres: each bin's groups in runs of G = the largest power of
    // two <= kXresMaxGroups with G * nch(bin) <= base * nch(heaviest bin), so that every set
    // is about `base` groups of the heaviest bin's work; bins in layout order
    // (heaviest first).
    h->xsets.clear();
    const int64_t nch_max = h->groups.empty() ? 1 : ceil_div(h->groups.front().n, kChunk);
    for (int i = 0; i < darb::kXresTables; ++i) {
        const int64_t base = int64_t(2) << i;
        h->xset_first[i] = static_cast<int32_t>(h->xsets.size());
        h->xset_prefix[i].assign(1, 0);
        size_t gbeg = 0;
        while (gbeg < h->groups.size()) {
            size_t gend = gbeg;
            while (gend < h->groups.size() && h->groups[gend].m == h->groups[gbeg].m) ++gend;
            const Group &g = h->groups[gbeg];
            const int64_t nch = ceil_div(g.n, kChunk);
            int G = 1;
            while (2 * G <= darb::kXresMaxGroups && 2 * G * nch <= base * nch_max) G *= 2;
            for (size_t s = gbeg; s < gend; s += static_cast<size_t>(G)) {
                darb::SetGeo sg{};
                const size_t ng = std::min<size_t>(static_cast<size_t>(G), gend - s);
                sg.g0 = static_cast<int32_t>(s);
                sg.ng = static_cast<int32_t>(ng);
                sg.m = g.m;
                sg.n = g.n;
                sg.nib = g.nib;
                sg.nrows_last = h->groups[s + ng - 1].nrows;
                sg.val_off = h->groups[s].val_off;
                sg.off_off = h->groups[s].off_off;
                h->xsets.push_back(sg);
                h->xset_prefix[i].push_back(h->xset_prefix[i].back() + int64_t(ng) * nch);
            }
            gbeg = gend;
        }
        h->nxsets[i] = static_cast<int32_t>(h->xsets.size()) - h->xset_first[i];
    }
}

darb_status_t alloc_device(darb_handle_s *h) {
    const size_t esz = h->wtype == DARB_BF16 ? 2 : 4;
    size_t o = 0;
    const size_t o_groups = o; o = align_up(o + h->groups.size() * sizeof(Group), 256);
    const size_t o_tiles = o;  o = align_up(o + h->enc_tiles.size() * sizeof(darb::EncTile), 256);
    const size_t o_rtiles = o; o = align_up(o + h->row_tiles.size() * sizeof(darb::EncTile), 256);
    const size_t o_items = o;  o = align_up(o + h->items.size() * sizeof(darb::WorkItem), 256);
    const size_t o_sgeo = o;   o = align_up(o + h->xsets.size() * sizeof(darb::SetGeo), 256);
    const size_t o_rowmap = o; o = align_up(o + h->rowmap.size() * 4, 256);
    const size_t o_rowloc = o; o = align_up(o + h->rowloc.size() * 4, 256);
    const size_t o_rowm = o;   o = align_up(o + h->row_m.size() * 4, 256);
    const size_t o_err = o;    o = align_up(o + 4, 256);
    const size_t o_vals = o;   o = align_up(o + static_cast<size_t>(h->val_elems) * esz, 256);
    const size_t o_offs = o;   o = align_up(o + static_cast<size_t>(h->off_words) * 4, 256);
    void *p = nullptr;
    const darb_status_t st = dev_alloc(&p, o);
    if (st != DARB_OK) return st;
    char *b = static_cast<char *>(p);
    h->dmem = p;
    h->dbytes = o;
    h->d_groups = reinterpret_cast<Group *>(b + o_groups);
    h->d_tiles = reinterpret_cast<darb::EncTile *>(b + o_tiles);
    h->d_row_tiles = reinterpret_cast<darb::EncTile *>(b + o_rtiles);
    h->d_items = reinterpret_cast<darb::WorkItem *>(b + o_items);
    h->d_xsets = reinterpret_cast<darb::SetGeo *>(b + o_sgeo);
    h->d_rowmap = reinterpret_cast<int32_t *>(b + o_rowmap);
    h->d_rowloc = reinterpret_cast<int32_t *>(b + o_rowloc);
    h->d_row_m = reinterpret_cast<int32_t *>(b + o_rowm);
    h->d_status = reinterpret_cast<int32_t *>(b + o_err);
    h->d_vals = b + o_vals;
    h->d_offs = reinterpret_cast<uint32_t *>(b + o_offs);
    return DARB_OK;
}

darb_status_t upload_layout(darb_handle_s *h, cudaStream_t stream) {
    cudaError_t e = cudaMemsetAsync(h->dmem, 0, h->dbytes, stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->d_groups, h->groups.data(), h->groups.size() * sizeof(Group),
                            cudaMemcpyHostToDevice, stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->d_tiles, h->enc_tiles.data(), h->enc_tiles.size() * sizeof(darb::EncTile),
                            cudaMemcpyHostToDevice, stream);
    if (e == cudaSuccess && !h->row_tiles.empty())
        e = cudaMemcpyAsync(h->d_row_tiles, h->row_tiles.data(), h->row_tiles.size() * sizeof(darb::EncTile),
                            cudaMemcpyHostToDevice, stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->d_items, h->items.data(), h->items.size() * sizeof(darb::WorkItem),
                            cudaMemcpyHostToDevice, stream);
    if (e == cudaSuccess && !h->xsets.empty())
        e = cudaMemcpyAsync(h->d_xsets, h->xsets.data(), h->xsets.size() * sizeof(darb::SetGeo),
                            cudaMemcpyHostToDevice, stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->d_rowmap, h->rowmap.data(), h->rowmap.size() * 4,
                            cudaMemcpyHostToDevice, stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->d_rowloc, h->rowloc.data(), h->rowloc.size() * 4,
                            cudaMemcpyHostToDevice, stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->d_row_m, h->row_m.data(), h->row_m.size() * 4,
                            cudaMemcpyHostToDevice, stream);
    return cuda_status(e);
}

void free_handle(darb_handle_s *h) {
    if (h == nullptr) return;
    if (h->dmem) cudaFree(h->dmem);
    if (h->d_gates) cudaFree(h->d_gates);
    if (h->d_counters) cudaFree(h->d_counters);
    if (h->reencode_event) cudaEventDestroy(h->reencode_event);
    delete h;
}

void register_handle(darb_handle_s *h) {
    std::lock_guard<std::mutex> lk(g_mu);
    g_live.insert(h);
}

Format format_of(const darb_handle_s *h) {
    Format f{};
    f.groups = h->d_groups;
    f.rowmap = h->d_rowmap;
    f.rowloc = h->d_rowloc;
    f.row_m = h->d_row_m;
    f.vals = h->d_vals;
    f.offs = h->d_offs;
    f.status = h->d_status;
    for (int l = 0; l < darb::kWorkLevels; ++l)
        for (int c = 0; c < darb::kWorkSplits; ++c) {
            f.items[l][c] = h->d_items + h->item_first[l][c];
            f.nitems[l][c] = h->nitems[l][c];
            f.item_work[l][c] = h->item_work[l][c];
        }
    f.nch_max = h->groups.empty() ? 1 : static_cast<int32_t>(ceil_div(h->groups.front().n, kChunk));
    for (int l = 0; l < darb::kWorkLevels; ++l) f.set_prefix[l] = h->set_prefix[l].data();
    for (int i = 0; i < darb::kXresTables; ++i) {
        f.xsets[i] = h->d_xsets + h->xset_first[i];
        f.nxsets[i] = h->nxsets[i];
        f.xset_prefix[i] = h->xset_prefix[i].data();
        f.xsets_host[i] = h->xsets.data() + h->xset_first[i];
    }
    f.ngroups = static_cast<int32_t>(h->groups.size());
    f.bf16 = h->wtype == DARB_BF16 ? 1 : 0;
    f.m_max = h->groups.empty() ? 1 : h->groups.back().m;   // groups are sorted by block size
    f.m_min = h->groups.empty() ? 1 : h->groups.front().m;
    f.rows = h->rows;
    f.cols = h->cols;
    return f;
}

darb::EncodeTarget target_of(darb_handle_s *h) {
    darb::EncodeTarget t{};
    t.tiles = h->d_tiles;
    t.ntiles = static_cast<int32_t>(h->enc_tiles.size());
    t.max_tile = h->max_tile;
    t.row_tiles = h->d_row_tiles;
    t.n_row_tiles = static_cast<int32_t>(h->row_tiles.size());
    t.vals = h->d_vals;
    t.offs = h->d_offs;
    t.bf16 = h->wtype == DARB_BF16 ? 1 : 0;
    t.rows = h->rows;
    t.cols = h->cols;
    return t;
}

bool valid_dtype(darb_dtype_t t) { return t == DARB_F32 || t == DARB_BF16; }

darb_status_t check_shape_and_m(int64_t rows, int64_t cols, const int32_t *m) {
    if (rows <= 0 || cols <= 0 || rows > kMaxDim || cols > kMaxDim || m == nullptr)
        return DARB_ERR_INVALID_ARG;
    for (int64_t r = 0; r < rows; ++r)
        if (m[r] < 1 || m[r] > DARB_MAX_BLOCK) return DARB_ERR_INVALID_ARG;
    return DARB_OK;
}

darb_status_t ensure_scratch(darb_handle_s *h, size_t gate_floats, size_t counter_ints) {
    if (gate_floats > h->gates_cap) {
        if (h->d_gates) {
            cudaDeviceSynchronize();
            cudaFree(h->d_gates);
            h->d_gates = nullptr;
            h->gates_cap = 0;
        }
        void *p = nullptr;
        const darb_status_t st = dev_alloc(&p, gate_floats * sizeof(float));
        if (st != DARB_OK) return st;
        h->d_gates = static_cast<float *>(p);
        h->gates_cap = gate_floats;
    }
    if (counter_ints > h->counters_cap) {
        if (h->d_counters) {
            cudaDeviceSynchronize();
            cudaFree(h->d_counters);
            h->d_counters = nullptr;
            h->counters_cap = 0;
        }
        void *p = nullptr;
        const darb_status_t st = dev_alloc(&p, counter_ints * sizeof(int32_t));
        if (st != DARB_OK) return st;
        if (cudaMemset(p, 0, counter_ints * sizeof(int32_t)) != cudaSuccess ||
            cudaDeviceSynchronize() != cudaSuccess) {
            cudaFree(p);
            return DARB_ERR_CUDA;
        }
        h->d_counters = static_cast<int32_t *>(p);
        h->counters_cap = counter_ints;
    }
    return DARB_OK;
}

// May a kernel read the handle's values before the previous kernel on `stream`
// has finished?  Yes unless a re-encode of this handle might still be running.
bool early_ok(darb_handle_s *h, cudaStream_t stream) {
    if (h->reencoded_in_graph) return false;
    if (!h->reencode_pending) return true;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(stream, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) {
        cudaGetLastError();
        return false;
    }
    const cudaError_t q = cudaEventQuery(h->reencode_event);
    if (q == cudaSuccess) {
        h->reencode_pending = false;
        return true;
    }
    cudaGetLastError();
    return false;
}

size_t gate_floats_for(const darb_handle_s *h, int64_t B, bool gru) {
    return static_cast<size_t>(h->rows) * static_cast<size_t>(B) * (gru ? 2 : 1);
}

size_t counter_ints_for(int64_t H, int64_t B) {
    const int bt = darb::rnn_batch_tile(B);
    return static_cast<size_t>(H) * static_cast<size_t>(ceil_div(B, bt));
}

bool overlaps(const void *a, size_t abytes, const void *b, size_t bbytes) {
    if (a == nullptr || b == nullptr) return false;
    const char *pa = static_cast<const char *>(a), *pb = static_cast<const char *>(b);
    return pa < pb + bbytes && pb < pa + abytes;
}

}  // namespace

extern "C" {

const char *darb_status_string(darb_status_t s) {
    switch (s) {
        case DARB_OK: return "DARB_OK";
        case DARB_ERR_INVALID_ARG: return "DARB_ERR_INVALID_ARG";
        case DARB_ERR_NONFINITE: return "DARB_ERR_NONFINITE";
        case DARB_ERR_OOM: return "DARB_ERR_OOM";
        case DARB_ERR_CUDA: return "DARB_ERR_CUDA";
        case DARB_ERR_TIMEOUT: return "DARB_ERR_TIMEOUT";
        case DARB_ERR_UNSUPPORTED: return "DARB_ERR_UNSUPPORTED";
    }
    return "DARB_ERR_UNKNOWN";
}

darb_status_t darb_assign_block_sizes(const int64_t *row_nnz, int64_t rows, int64_t cols,
                                      int32_t m_min, int32_t m_max, int32_t *m_out) {
    DARB_TRACE("darb_assign_block_sizes");
    if (row_nnz == nullptr || m_out == nullptr || rows <= 0 || cols <= 0 || m_min < 1 ||
        m_max < m_min || m_max > DARB_MAX_BLOCK)
        return DARB_ERR_INVALID_ARG;
    // total retained weights; a row is "dense" when nnz_r/cols >= total/(rows*cols)
    __int128 total = 0;
    for (int64_t r = 0; r < rows; ++r) {
        if (row_nnz[r] < 0 || row_nnz[r] > cols) return DARB_ERR_INVALID_ARG;
        total += row_nnz[r];
    }
    for (int64_t r = 0; r < rows; ++r) {
        const int64_t nnz = row_nnz[r];
        int64_t mm;
        if (nnz == 0) {
            mm = m_max;
        } else {
            // q = cols / nnz >= 1; dense rows take 2^floor(log2 q), sparse 2^ceil(log2 q)
            const bool dense = static_cast<__int128>(nnz) * rows >= total;
            int e = 0;
            if (dense) {
                while ((nnz << (e + 1)) <= cols) ++e;
            } else {
                while ((nnz << e) < cols) ++e;
            }
            mm = int64_t(1) << e;
        }
        m_out[r] = static_cast<int32_t>(std::min<int64_t>(std::max<int64_t>(mm, m_min), m_max));
    }
    return DARB_OK;
}

darb_status_t darb_encode(const void *W, darb_dtype_t wtype, int64_t rows, int64_t cols,
                          int64_t ldw, const int32_t *m, darb_handle_t *out, cudaStream_t stream) {
    DARB_TRACE("darb_encode");
    if (out == nullptr) return DARB_ERR_INVALID_ARG;
    *out = nullptr;
    if (W == nullptr || !valid_dtype(wtype) || ldw < cols) return DARB_ERR_INVALID_ARG;
    const size_t esz = wtype == DARB_BF16 ? 2 : 4;
    if (reinterpret_cast<uintptr_t>(W) % esz != 0) return DARB_ERR_INVALID_ARG;
    darb_status_t st = check_shape_and_m(rows, cols, m);
    if (st != DARB_OK) return st;
    darb_handle_s *h = new (std::nothrow) darb_handle_s();
    if (h == nullptr) return DARB_ERR_OOM;
    h->rows = rows;
    h->cols = cols;
    h->wtype = wtype;
    try {
        build_layout(h, m);
    } catch (const std::bad_alloc &) {
        delete h;
        return DARB_ERR_OOM;
    }
    st = alloc_device(h);
    if (st == DARB_OK) st = upload_layout(h, stream);
    if (st == DARB_OK) st = cuda_status(darb::launch_encode(target_of(h), W, ldw, h->d_status, stream));
    int32_t err = 0;
    if (st == DARB_OK)
        st = cuda_status(cudaMemcpyAsync(&err, h->d_status, 4, cudaMemcpyDeviceToHost, stream));
    if (st == DARB_OK) st = cuda_status(cudaStreamSynchronize(stream));
    if (st == DARB_OK && err != 0) st = DARB_ERR_NONFINITE;
    if (st != DARB_OK) {
        if (h->dmem) cudaStreamSynchronize(stream);
        free_handle(h);
        return st;
    }
    register_handle(h);
    *out = h;
    return DARB_OK;
}

darb_status_t darb_reencode(darb_handle_t h, const void *W, int64_t ldw, cudaStream_t stream) {
    DARB_TRACE("darb_reencode");
    if (!live(h) || W == nullptr || ldw < h->cols) return DARB_ERR_INVALID_ARG;
    const size_t esz = h->wtype == DARB_BF16 ? 2 : 4;
    if (reinterpret_cast<uintptr_t>(W) % esz != 0) return DARB_ERR_INVALID_ARG;
    darb_status_t st = cuda_status(darb::launch_encode(target_of(h), W, ldw, h->d_status, stream));
    if (st != DARB_OK) return st;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(stream, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) {
        cudaGetLastError();
        h->reencoded_in_graph = true;
        return DARB_OK;
    }
    if (h->reencode_event == nullptr &&
        cudaEventCreateWithFlags(&h->reencode_event, cudaEventDisableTiming) != cudaSuccess)
        return DARB_ERR_CUDA;
    if (cudaEventRecord(h->reencode_event, stream) != cudaSuccess) return DARB_ERR_CUDA;
    h->reencode_pending = true;
    return DARB_OK;
}

// A host <-> device copy of `rows` rows of `width` bytes, one cudaMemcpyAsync
// when both sides are contiguous, else one pitched copy.
static cudaError_t copy_rows(void *dst, size_t dpitch, const void *src, size_t spitch, size_t width, int64_t rows,
                             cudaMemcpyKind kind, cudaStream_t stream) {
    if (dpitch == width && spitch == width)
        return cudaMemcpyAsync(dst, src, width * static_cast<size_t>(rows), kind, stream);
    return cudaMemcpy2DAsync(dst, dpitch, src, spitch, width, static_cast<size_t>(rows), kind, stream);
}

darb_status_t darb_reencode_host(darb_handle_t h, const void *W, int64_t ldw, void *W_dev, cudaStream_t stream) {
    DARB_TRACE("darb_reencode_host");
    if (!live(h) || W == nullptr || W_dev == nullptr || ldw < h->cols) return DARB_ERR_INVALID_ARG;
    const size_t esz = h->wtype == DARB_BF16 ? 2 : 4;
    if (reinterpret_cast<uintptr_t>(W) % esz != 0 || reinterpret_cast<uintptr_t>(W_dev) % esz != 0)
        return DARB_ERR_INVALID_ARG;
    const size_t pitch = static_cast<size_t>(ldw) * esz;
    if (copy_rows(W_dev, pitch, W, pitch, static_cast<size_t>(h->cols) * esz, h->rows, cudaMemcpyHostToDevice,
                  stream) != cudaSuccess)
        return DARB_ERR_CUDA;
    return darb_reencode(h, W_dev, ldw, stream);
}

darb_status_t darb_sync_status(darb_handle_t h, cudaStream_t stream) {
    DARB_TRACE("darb_sync_status");
    if (!live(h)) return DARB_ERR_INVALID_ARG;
    int32_t bits = 0;
    cudaError_t e = cudaMemcpyAsync(&bits, h->d_status, 4, cudaMemcpyDeviceToHost, stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(h->d_status, 0, 4, stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return DARB_ERR_CUDA;
    if (bits & darb::kStatusTimeout) return DARB_ERR_TIMEOUT;
    return (bits & darb::kStatusNaN) ? DARB_ERR_NONFINITE : DARB_OK;
}

darb_status_t darb_spmm(darb_handle_t h, const float *X, int64_t ldx, int64_t batch, float *Y,
                        int64_t ldy, cudaStream_t stream) {
    DARB_TRACE("darb_spmm");
    return darb_spmm_ex(h, X, ldx, batch, Y, ldy, DARB_PATH_AUTO, stream);
}

darb_status_t darb_spmm_ex(darb_handle_t h, const float *X, int64_t ldx, int64_t batch, float *Y,
                           int64_t ldy, darb_path_t path, cudaStream_t stream) {
    DARB_TRACE("darb_spmm_ex");
    if (path != DARB_PATH_AUTO && path != DARB_PATH_CUDA_CORES && path != DARB_PATH_TENSOR_CORES)
        return DARB_ERR_INVALID_ARG;
    if (!live(h) || X == nullptr || Y == nullptr || batch <= 0 || ldx < batch || ldy < batch)
        return DARB_ERR_INVALID_ARG;
    if (reinterpret_cast<uintptr_t>(X) % 4 != 0 || reinterpret_cast<uintptr_t>(Y) % 4 != 0)
        return DARB_ERR_INVALID_ARG;
    if (batch > kMaxBatch) return DARB_ERR_UNSUPPORTED;
    if (overlaps(X, static_cast<size_t>((h->cols - 1) * ldx + batch) * 4, Y,
                 static_cast<size_t>((h->rows - 1) * ldy + batch) * 4))
        return DARB_ERR_INVALID_ARG;
    const cudaError_t e = darb::launch_spmm(format_of(h), X, ldx, batch, Y, ldy, early_ok(h, stream), path, stream);
    if (e == cudaErrorNotSupported) {
        cudaGetLastError();
        return DARB_ERR_UNSUPPORTED;
    }
    if (e == cudaErrorMemoryAllocation) {
        cudaGetLastError();
        return DARB_ERR_OOM;
    }
    return cuda_status(e);
}

darb_status_t darb_spmm_host(darb_handle_t h, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy,
                             float *X_dev, float *Y_dev, cudaStream_t stream) {
    DARB_TRACE("darb_spmm_host");
    if (!live(h) || X == nullptr || Y == nullptr || X_dev == nullptr || Y_dev == nullptr || batch <= 0 ||
        ldx < batch || ldy < batch)
        return DARB_ERR_INVALID_ARG;
    if (reinterpret_cast<uintptr_t>(X) % 4 != 0 || reinterpret_cast<uintptr_t>(Y) % 4 != 0 ||
        reinterpret_cast<uintptr_t>(X_dev) % 4 != 0 || reinterpret_cast<uintptr_t>(Y_dev) % 4 != 0)
        return DARB_ERR_INVALID_ARG;
    if (batch > kMaxBatch) return DARB_ERR_UNSUPPORTED;
    const size_t row = static_cast<size_t>(batch) * 4;
    // every check before the first copy: a rejected call does no device work
    if (overlaps(X_dev, row * static_cast<size_t>(h->cols), Y_dev, row * static_cast<size_t>(h->rows)))
        return DARB_ERR_INVALID_ARG;
    if (copy_rows(X_dev, row, X, static_cast<size_t>(ldx) * 4, row, h->cols, cudaMemcpyHostToDevice, stream) !=
        cudaSuccess)
        return DARB_ERR_CUDA;
    const darb_status_t st = darb_spmm(h, X_dev, batch, batch, Y_dev, batch, stream);
    if (st != DARB_OK) return st;
    if (copy_rows(Y, static_cast<size_t>(ldy) * 4, Y_dev, row, row, h->rows, cudaMemcpyDeviceToHost, stream) !=
        cudaSuccess)
        return DARB_ERR_CUDA;
    return DARB_OK;
}

darb_status_t darb_assign_from_weights(const void *W, darb_dtype_t wtype, int64_t rows, int64_t cols, int64_t ldw,
                                       int64_t keep, int32_t m_min, int32_t m_max, int64_t *row_nnz_out,
                                       int32_t *m_out, cudaStream_t stream) {
    DARB_TRACE("darb_assign_from_weights");
    if (W == nullptr || m_out == nullptr || !valid_dtype(wtype)) return DARB_ERR_INVALID_ARG;
    if (rows <= 0 || cols <= 0 || rows > kMaxDim || cols > kMaxDim || ldw < cols) return DARB_ERR_INVALID_ARG;
    if (m_min < 1 || m_max < m_min || m_max > DARB_MAX_BLOCK) return DARB_ERR_INVALID_ARG;
    const size_t esz = wtype == DARB_BF16 ? 2 : 4;
    if (reinterpret_cast<uintptr_t>(W) % esz != 0) return DARB_ERR_INVALID_ARG;
    if (keep < 1 || keep > rows * cols) return DARB_ERR_INVALID_ARG;
    if (rows * cols >= (int64_t(1) << 32)) return DARB_ERR_UNSUPPORTED;
    std::vector<int64_t> nnz;
    try {
        nnz.resize(static_cast<size_t>(rows));
    } catch (const std::bad_alloc &) {
        return DARB_ERR_OOM;
    }
    // scratch: selection state and histograms (4608 B), the NaN flag, the row counts
    const size_t o_flag = 4608, o_rows = 4864;
    // the call synchronises, so one scratch buffer per device serves every call
    // (kept between calls, grown when a matrix has more rows; calls serialise on it)
    static std::mutex scratch_mu;
    static std::map<int, std::pair<void *, size_t>> scratch;
    std::lock_guard<std::mutex> lk(scratch_mu);
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {   // no device: the allocation below reports it
        cudaGetLastError();
        dev = -1;
    }
    auto &slot = scratch[dev];
    const size_t need = o_rows + static_cast<size_t>(rows) * 8;
    if (slot.second < need) {
        if (slot.first) {
            cudaDeviceSynchronize();
            cudaFree(slot.first);
            slot = {nullptr, 0};
        }
        void *p = nullptr;
        const darb_status_t st = dev_alloc(&p, need);
        if (st != DARB_OK) return st;
        slot = {p, need};
    }
    void *work = slot.first;
    char *b = static_cast<char *>(work);
    int32_t nan_flag = 0;
    cudaError_t e = darb::launch_topk_row_nnz(W, wtype == DARB_BF16, rows, cols, ldw, keep,
                                              reinterpret_cast<int64_t *>(b + o_rows), work,
                                              reinterpret_cast<int32_t *>(b + o_flag), stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(nnz.data(), b + o_rows, static_cast<size_t>(rows) * 8, cudaMemcpyDeviceToHost, stream);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&nan_flag, b + o_flag, 4, cudaMemcpyDeviceToHost, stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return DARB_ERR_CUDA;
    if (nan_flag) return DARB_ERR_NONFINITE;
    if (row_nnz_out) std::copy(nnz.begin(), nnz.end(), row_nnz_out);
    return darb_assign_block_sizes(nnz.data(), rows, cols, m_min, m_max, m_out);
}

darb_status_t darb_spmm_path(darb_handle_t h, int64_t batch, darb_path_t *path, int32_t *kernels) {
    DARB_TRACE("darb_spmm_path");
    if (!live(h) || batch <= 0 || path == nullptr || kernels == nullptr) return DARB_ERR_INVALID_ARG;
    // darb_spmm always takes the CUDA-core gather: one kernel per call
    *path = DARB_PATH_CUDA_CORES;
    *kernels = 1;
    return DARB_OK;
}

darb_status_t darb_rnn_reserve(darb_handle_t h, int64_t max_batch) {
    DARB_TRACE("darb_rnn_reserve");
    if (!live(h) || max_batch <= 0 || max_batch > kMaxBatch) return DARB_ERR_INVALID_ARG;
    // GRU needs the larger gate buffer; the smallest tile gives the most counters
    const int64_t units = h->rows;   // upper bound on H for either cell
    size_t counters = 0;
    for (int64_t b = 1; b <= std::min<int64_t>(max_batch, 8); ++b)
        counters = std::max(counters, counter_ints_for(units, b));
    counters = std::max(counters, counter_ints_for(units, max_batch));
    return ensure_scratch(h, gate_floats_for(h, max_batch, true), counters);
}

static darb_status_t check_step(darb_handle_t h, int64_t I, int64_t H, int64_t B, int gates,
                                const float *x, const float *h_prev) {
    if (!live(h)) return DARB_ERR_INVALID_ARG;
    if (I < 0 || H <= 0 || B <= 0 || h->rows != gates * H || h->cols != I + H)
        return DARB_ERR_INVALID_ARG;
    if ((I > 0 && x == nullptr) || h_prev == nullptr) return DARB_ERR_INVALID_ARG;
    if (B > kMaxBatch) return DARB_ERR_UNSUPPORTED;
    return DARB_OK;
}

darb_status_t darb_lstm_step(darb_handle_t h, int64_t I, int64_t H, int64_t B, const float *x,
                             const float *h_prev, const float *c_prev, const float *bias,
                             float *h_out, float *c_out, cudaStream_t stream) {
    DARB_TRACE("darb_lstm_step");
    darb_status_t st = check_step(h, I, H, B, 4, x, h_prev);
    if (st != DARB_OK) return st;
    if (c_prev == nullptr || h_out == nullptr || c_out == nullptr) return DARB_ERR_INVALID_ARG;
    const size_t hb = static_cast<size_t>(H * B) * 4;
    const void *ins[4] = {x, h_prev, c_prev, bias};
    const size_t inb[4] = {static_cast<size_t>(I * B) * 4, hb, hb, static_cast<size_t>(4 * H) * 4};
    for (int i = 0; i < 4; ++i)
        if (overlaps(h_out, hb, ins[i], inb[i]) || overlaps(c_out, hb, ins[i], inb[i]))
            return DARB_ERR_INVALID_ARG;
    if (overlaps(h_out, hb, c_out, hb)) return DARB_ERR_INVALID_ARG;
    st = ensure_scratch(h, gate_floats_for(h, B, false), counter_ints_for(H, B));
    if (st != DARB_OK) return st;
    darb::RnnScratch sc{h->d_gates, h->d_counters};
    return cuda_status(darb::launch_lstm_step(format_of(h), I, H, B, x, h_prev, c_prev, bias,
                                              h_out, c_out, sc, stream, early_ok(h, stream)));
}

darb_status_t darb_gru_step(darb_handle_t h, int64_t I, int64_t H, int64_t B, const float *x,
                            const float *h_prev, const float *b_ih, const float *b_hh,
                            float *h_out, cudaStream_t stream) {
    DARB_TRACE("darb_gru_step");
    darb_status_t st = check_step(h, I, H, B, 3, x, h_prev);
    if (st != DARB_OK) return st;
    if (h_out == nullptr) return DARB_ERR_INVALID_ARG;
    const size_t hb = static_cast<size_t>(H * B) * 4;
    const void *ins[4] = {x, h_prev, b_ih, b_hh};
    const size_t inb[4] = {static_cast<size_t>(I * B) * 4, hb, static_cast<size_t>(3 * H) * 4,
                           static_cast<size_t>(3 * H) * 4};
    for (int i = 0; i < 4; ++i)
        if (overlaps(h_out, hb, ins[i], inb[i])) return DARB_ERR_INVALID_ARG;
    st = ensure_scratch(h, gate_floats_for(h, B, true), counter_ints_for(H, B));
    if (st != DARB_OK) return st;
    darb::RnnScratch sc{h->d_gates, h->d_counters};
    return cuda_status(darb::launch_gru_step(format_of(h), I, H, B, x, h_prev, b_ih, b_hh, h_out,
                                             sc, stream, early_ok(h, stream)));
}

// Arrival counts of the sequence kernels' barrier stay below 2^32.
constexpr int64_t kMaxSequenceSteps = int64_t(1) << 22;

static darb_status_t sequence_status(cudaError_t e) {
    if (e == cudaErrorNotSupported) return DARB_ERR_UNSUPPORTED;
    if (e == cudaErrorMemoryAllocation) return DARB_ERR_OOM;
    return cuda_status(e);
}

darb_status_t darb_lstm_sequence(darb_handle_t h, int64_t T, int64_t I, int64_t H, int64_t B, const float *x_seq,
                                 const float *h0, const float *c0, const float *bias, float *h_seq, float *c_seq,
                                 float *c_last, cudaStream_t stream) {
    DARB_TRACE("darb_lstm_sequence");
    // x_seq may be NULL when there are no steps
    darb_status_t st = check_step(h, I, H, B, 4, T > 0 ? x_seq : h0, h0);
    if (st != DARB_OK) return st;
    if (T < 0 || c0 == nullptr || (T > 0 && h_seq == nullptr)) return DARB_ERR_INVALID_ARG;
    if (T > kMaxSequenceSteps) return DARB_ERR_UNSUPPORTED;
    const size_t hb = static_cast<size_t>(H * B) * 4, sb = hb * static_cast<size_t>(T);
    const void *ins[4] = {x_seq, h0, c0, bias};
    const size_t inb[4] = {static_cast<size_t>(I * B) * 4 * static_cast<size_t>(T), hb, hb,
                           static_cast<size_t>(4 * H) * 4};
    void *outs[3] = {h_seq, c_seq, c_last};
    const size_t outb[3] = {sb, sb, hb};
    for (int o = 0; o < 3; ++o) {
        for (int i = 0; i < 4; ++i)
            if (overlaps(outs[o], outb[o], ins[i], inb[i])) return DARB_ERR_INVALID_ARG;
        for (int p = o + 1; p < 3; ++p)
            if (overlaps(outs[o], outb[o], outs[p], outb[p])) return DARB_ERR_INVALID_ARG;
    }
    if (T == 0)
        return c_last ? cuda_status(cudaMemcpyAsync(c_last, c0, hb, cudaMemcpyDeviceToDevice, stream)) : DARB_OK;
    return sequence_status(darb::launch_lstm_sequence(format_of(h), h->row_m.data(), T, I, H, B, x_seq, h0, c0,
                                                      bias, h_seq, c_seq, c_last, stream));
}

darb_status_t darb_gru_sequence(darb_handle_t h, int64_t T, int64_t I, int64_t H, int64_t B, const float *x_seq,
                                const float *h0, const float *b_ih, const float *b_hh, float *h_seq,
                                cudaStream_t stream) {
    DARB_TRACE("darb_gru_sequence");
    darb_status_t st = check_step(h, I, H, B, 3, T > 0 ? x_seq : h0, h0);
    if (st != DARB_OK) return st;
    if (T < 0 || (T > 0 && h_seq == nullptr)) return DARB_ERR_INVALID_ARG;
    if (T > kMaxSequenceSteps) return DARB_ERR_UNSUPPORTED;
    const size_t hb = static_cast<size_t>(H * B) * 4, sb = hb * static_cast<size_t>(T);
    const void *ins[4] = {x_seq, h0, b_ih, b_hh};
    const size_t inb[4] = {static_cast<size_t>(I * B) * 4 * static_cast<size_t>(T), hb,
                           static_cast<size_t>(3 * H) * 4, static_cast<size_t>(3 * H) * 4};
    for (int i = 0; i < 4; ++i)
        if (overlaps(h_seq, sb, ins[i], inb[i])) return DARB_ERR_INVALID_ARG;
    if (T == 0) return DARB_OK;
    return sequence_status(darb::launch_gru_sequence(format_of(h), h->row_m.data(), T, I, H, B, x_seq, h0, b_ih,
                                                     b_hh, h_seq, stream));
}

darb_status_t darb_info(darb_handle_t h, darb_info_t *info) {
    DARB_TRACE("darb_info");
    if (!live(h) || info == nullptr) return DARB_ERR_INVALID_ARG;
    darb_info_t r{};
    r.rows = h->rows;
    r.cols = h->cols;
    r.nnzb = h->nnzb;
    r.wtype = h->wtype;
    r.nbins = h->nbins;
    r.ngroups = static_cast<int32_t>(h->groups.size());
    r.value_bytes = h->nnzb * (h->wtype == DARB_BF16 ? 2 : 4);
    int64_t off_bits = 0, idx_bits = 0;
    for (int64_t i = 0; i < h->rows; ++i) {
        const int32_t mm = h->row_m[i];
        const int64_t n = ceil_div(h->cols, mm);
        off_bits += n * (mm <= 16 ? 4 : 8);
        int b = 0;
        while ((int64_t(1) << b) < mm) ++b;
        idx_bits += n * b;
    }
    r.offset_bytes = (off_bits + 7) / 8;
    r.meta_bytes = h->rows * 6;
    r.index_bits_min = idx_bits;
    r.device_bytes = static_cast<int64_t>(h->dbytes + h->gates_cap * 4 + h->counters_cap * 4);
    *info = r;
    return DARB_OK;
}

darb_status_t darb_export(darb_handle_t h, void *val, uint8_t *off, int64_t *blk_ptr, int32_t *m) {
    DARB_TRACE("darb_export");
    if (!live(h)) return DARB_ERR_INVALID_ARG;
    const size_t esz = h->wtype == DARB_BF16 ? 2 : 4;
    std::vector<uint8_t> hv;
    std::vector<uint32_t> ho;
    try {
        hv.resize(static_cast<size_t>(h->val_elems) * esz);
        ho.resize(static_cast<size_t>(h->off_words));
    } catch (const std::bad_alloc &) {
        return DARB_ERR_OOM;
    }
    if (cudaDeviceSynchronize() != cudaSuccess) return DARB_ERR_CUDA;
    if (cudaMemcpy(hv.data(), h->d_vals, hv.size(), cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemcpy(ho.data(), h->d_offs, ho.size() * 4, cudaMemcpyDeviceToHost) != cudaSuccess)
        return DARB_ERR_CUDA;
    std::vector<int64_t> bp(static_cast<size_t>(h->rows) + 1, 0);
    for (int64_t r = 0; r < h->rows; ++r) bp[r + 1] = bp[r] + ceil_div(h->cols, h->row_m[r]);
    for (int64_t r = 0; r < h->rows; ++r) {
        const int32_t loc = h->rowloc[r];
        const Group &g = h->groups[loc / kSlots];
        const int slot = loc % kSlots;
        for (int64_t j = 0; j < g.n; ++j) {
            const int64_t c = j / kChunk, e = j % kChunk;
            const int64_t vi = g.val_off + (c * kSlots + slot) * kChunk + e;
            const int64_t p = bp[r] + j;
            if (val) std::memcpy(static_cast<char *>(val) + p * esz, hv.data() + vi * esz, esz);
            if (off) {
                uint32_t o;
                if (g.nib) {
                    o = (ho[g.off_off + c * kSlots + slot] >> (4 * e)) & 15u;
                } else {
                    const uint32_t w = ho[g.off_off + 2 * (c * kSlots + slot) + (e >= 4 ? 1 : 0)];
                    o = (w >> (8 * (e & 3))) & 255u;
                }
                off[p] = static_cast<uint8_t>(o);
            }
        }
    }
    if (blk_ptr) std::memcpy(blk_ptr, bp.data(), bp.size() * sizeof(int64_t));
    if (m) std::memcpy(m, h->row_m.data(), h->row_m.size() * sizeof(int32_t));
    return DARB_OK;
}

darb_status_t darb_import(const void *val, const uint8_t *off, const int32_t *m,
                          darb_dtype_t wtype, int64_t rows, int64_t cols, darb_handle_t *out,
                          cudaStream_t stream) {
    DARB_TRACE("darb_import");
    if (out == nullptr) return DARB_ERR_INVALID_ARG;
    *out = nullptr;
    if (val == nullptr || off == nullptr || !valid_dtype(wtype)) return DARB_ERR_INVALID_ARG;
    darb_status_t st = check_shape_and_m(rows, cols, m);
    if (st != DARB_OK) return st;
    darb_handle_s *h = new (std::nothrow) darb_handle_s();
    if (h == nullptr) return DARB_ERR_OOM;
    h->rows = rows;
    h->cols = cols;
    h->wtype = wtype;
    const size_t esz = wtype == DARB_BF16 ? 2 : 4;
    std::vector<uint8_t> hv;
    std::vector<uint32_t> ho;
    try {
        build_layout(h, m);
        hv.assign(static_cast<size_t>(h->val_elems) * esz, 0);
        ho.assign(static_cast<size_t>(h->off_words), 0);
    } catch (const std::bad_alloc &) {
        delete h;
        return DARB_ERR_OOM;
    }
    int64_t p = 0;
    for (int64_t r = 0; r < rows; ++r) {
        const int32_t loc = h->rowloc[r];
        const Group &g = h->groups[loc / kSlots];
        const int slot = loc % kSlots;
        for (int64_t j = 0; j < g.n; ++j, ++p) {
            if (off[p] >= g.m || j * g.m + off[p] >= cols) {
                delete h;
                return DARB_ERR_INVALID_ARG;
            }
            const int64_t c = j / kChunk, e = j % kChunk;
            const int64_t vi = g.val_off + (c * kSlots + slot) * kChunk + e;
            std::memcpy(hv.data() + vi * esz, static_cast<const char *>(val) + p * esz, esz);
            if (g.nib) {
                ho[g.off_off + c * kSlots + slot] |= static_cast<uint32_t>(off[p]) << (4 * e);
            } else {
                ho[g.off_off + 2 * (c * kSlots + slot) + (e >= 4 ? 1 : 0)] |=
                    static_cast<uint32_t>(off[p]) << (8 * (e & 3));
            }
        }
    }
    st = alloc_device(h);
    if (st == DARB_OK) st = upload_layout(h, stream);
    if (st == DARB_OK)
        st = cuda_status(cudaMemcpyAsync(h->d_vals, hv.data(), hv.size(), cudaMemcpyHostToDevice, stream));
    if (st == DARB_OK)
        st = cuda_status(cudaMemcpyAsync(h->d_offs, ho.data(), ho.size() * 4, cudaMemcpyHostToDevice, stream));
    if (st == DARB_OK) st = cuda_status(cudaStreamSynchronize(stream));
    if (st != DARB_OK) {
        if (h->dmem) cudaStreamSynchronize(stream);
        free_handle(h);
        return st;
    }
    register_handle(h);
    *out = h;
    return DARB_OK;
}

darb_status_t darb_set_pdl(int enabled) {
    DARB_TRACE("darb_set_pdl");
    darb::pdl_setting().store(enabled ? 1 : 0, std::memory_order_relaxed);
    return DARB_OK;
}

darb_status_t darb_destroy(darb_handle_t h) {
    DARB_TRACE("darb_destroy");
    if (h == nullptr) return DARB_OK;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        if (g_live.erase(h) == 0) return DARB_ERR_INVALID_ARG;
    }
    free_handle(h);
    return DARB_OK;
}

}  // extern "C"

namespace darb {

darb_status_t lstm_step_view(darb_handle_t h, int64_t I, int64_t H, int64_t B, const float *x,
                             const float *h_prev, const float *c_prev, const float *bias,
                             const float *h_out, const float *c_out, Format *f) {
    darb_status_t st = check_step(h, I, H, B, 4, x, h_prev);
    if (st != DARB_OK) return st;
    if (c_prev == nullptr || h_out == nullptr || c_out == nullptr || f == nullptr) return DARB_ERR_INVALID_ARG;
    const size_t hb = static_cast<size_t>(H * B) * 4;
    const void *ins[4] = {x, h_prev, c_prev, bias};
    const size_t inb[4] = {static_cast<size_t>(I * B) * 4, hb, hb, static_cast<size_t>(4 * H) * 4};
    for (int i = 0; i < 4; ++i)
        if (overlaps(h_out, hb, ins[i], inb[i]) || overlaps(c_out, hb, ins[i], inb[i]))
            return DARB_ERR_INVALID_ARG;
    if (overlaps(h_out, hb, c_out, hb)) return DARB_ERR_INVALID_ARG;
    *f = format_of(h);
    return DARB_OK;
}

}  // namespace darb
