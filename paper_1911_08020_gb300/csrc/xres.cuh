// xres.cuh -- Y = W_darb X for batch > 4 with each CTA's slice of the activation
// tile resident in shared memory (Sec. 3.2, Fig. 6(b): block j of a row selects
// activation row j*m + off).
//
// Why: the product multiplies every kept weight by one activation row of the
// batch tile, and the rows a block can select are only its own m.  Split the
// columns of W into C slices of S columns; a block belongs to the slice its
// first column falls in, so a CTA that holds rows [q*S, (q+1)*S + m_max - 1)
// of the tile can multiply every block of its slice, of every row, without
// staging anything else (rows [q*S, (q+1)*S) when S is a multiple of every
// block size: no block then reaches past its slice).  C is the split whose
// clusters occupy the most SMs: clusters of 8 fill 120 of the 152, of 6 138,
// of 4 144.  A cluster of C CTAs (one per slice) therefore loads the tile
// once and then streams only the kept values and packed offsets (2.5 bytes
// per kept weight for bf16) through a ring of bulk copies.  The C partial
// sums of a row meet in distributed shared memory.
//
// Layout of the work:
//  * persistent clusters (as many as the GPU holds at once), one CTA per SM;
//  * a unit = (batch tile of T columns, row set): a run of up to 4 groups of
//    one block-size bin, sized so that every set has about the work of a
//    fixed number of groups of the heaviest bin (the SetGeo tables of the
//    handle); units in tile-major order; each cluster takes a contiguous run
//    of units of about equal work, so it loads the tile of a run once or twice;
//  * 16 consumer warps: 4 lanes per row, each lane 8 of the tile's 32
//    columns (two 16-byte loads per kept weight, so that one offset, one value
//    and one address serve 8 FMAs; the two rows of a quarter-warp read
//    opposite halves of their activation rows, which keeps the loads free of
//    bank conflicts); a pass covers 128 rows, the largest set, and a thread
//    owns one row of it;
//  * one producer warp: bulk copies of the values and offsets of each round
//    (a run of chunks of the set's groups) into a ring of 3 to 6 stages (as
//    many as fit beside the slice) with full / empty mbarriers, and
//    tensor-map copies of the tile slice (rows past the matrix or columns
//    past the batch arrive as zeros), box by box, each box on its own
//    barrier: a round waits only for the boxes holding the rows its blocks
//    can select, so the consumers start on the first rows while the rest
//    land; a run's first slice is requested before its first set record is
//    read;
//  * three reducer warps: when every CTA of the cluster has stored its partial
//    sums of a set (each consumer warp, once its rows are stored, arrives on
//    every CTA's "ready" barrier), they add, for this CTA's share of the
//    set's R rows ([q R / C, (q + 1) R / C)), the C partial sums in rank
//    order (deterministic), write Y, and each reducer
//    warp arrives on every CTA's "freed" barrier; the consumers meanwhile
//    multiply the next set, and store its partial sums only once every CTA's
//    reducers have read the previous ones.  No CTA-wide barrier separates
//    the sets.  (Every warp arrives once per set on each barrier, and issues
//    its arrivals for set t + 1 on one barrier only after every CTA has got
//    past set t on the other -- microseconds after every arrival for set t
//    was issued.)
//
// Waits poll try_wait, which parks the warp in hardware until the phase
// completes, without sleeping in between (a lane that slept past the phase
// would hold up its warp).  Every wait is bounded; one that gives up records
// DARB_ERR_TIMEOUT, the
// warp skips the remaining work, the producer lets its own copies land
// (bounded) and all warps meet at the final cluster barrier, so no CTA leaves
// while another may still read its shared memory or arrive on its barriers.
#pragma once

#include "kernels_common.cuh"
#include "launch.cuh"
#include "tma.cuh"

#include <cooperative_groups.h>
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <type_traits>
#include <vector>

namespace darb {
namespace xres {

namespace cg = cooperative_groups;

// 16 bytes of the staged activation slice at a 32-bit shared address.  Not
// volatile: the address depends on offsets read after the stage's wait, and
// the slice itself changes only across the waits on its boxes.
__device__ __forceinline__ float4 lds_f4(uint32_t addr) {
    float4 v;
    asm("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr));
    return v;
}

constexpr int kCWarps = 16;                    // consumer warps
constexpr int kCThreads = kCWarps * 32;
constexpr int kRWarps = 3;                     // reducer warps (20 warps in all: 96 registers a thread)
constexpr int kRThreads = kRWarps * 32;
constexpr int kProducerWarp = kCWarps;
constexpr int kThreads = kCThreads + 32 + kRThreads;
constexpr int kMaxStages = 6;                  // rounds of values and offsets in the ring, at most
constexpr int kMinStages = 3;                  // and at least, unless nothing else fits
constexpr int kRecCap = 8;                     // (group, chunk) records per round
constexpr int kMaxGroups = kXresMaxGroups;     // groups of a row set, at most
constexpr int kMaxClusters = 160;
constexpr int kUnitCost = 10;                  // fixed cost of a unit, in group-chunks
constexpr int kSwitchCost = 40;                // a run's move to another batch tile, in group-chunks
constexpr size_t kSmemCap = 227 * 1024;        // dynamic shared memory, at most (the kernel has no static part)

template <bool BF16>
__host__ __device__ constexpr uint32_t rec_val_bytes() { return kSlots * kChunk * (BF16 ? 2 : 4); }
constexpr uint32_t kRecOffBytes = kSlots * 8;  // room for 8-byte offset records
template <bool BF16>
__host__ __device__ constexpr uint32_t ring_val_bytes() { return kRecCap * rec_val_bytes<BF16>(); }
template <bool BF16>
__host__ __device__ constexpr uint32_t stage_bytes() { return ring_val_bytes<BF16>() + kRecCap * kRecOffBytes; }

struct Plan {
    int C;            // CTAs per cluster = column slices (1 .. 8)
    int S;            // a slice's blocks start in columns [q*S, (q+1)*S)
    int nst;          // stages of the ring (fewer than kMinStages only when nothing else fits)
    int box_rows;     // activation rows per tensor-map box
    int nboxes;       // boxes per slice
    int table;        // row-set table (SetGeo) of the handle
    int nsets;        // row sets of that table
    uint32_t x_bytes; // bytes of the staged slice (nboxes * box_rows * T * 4)
    uint32_t ring_off, part_off;   // offsets in dynamic shared memory
    int2 range[kMaxClusters];      // units [x, y) of each cluster
};

// Barriers at the start of dynamic shared memory.
constexpr int kMaxBoxes = 8;       // tensor-map boxes of a slice, at most (1816 rows of 128 bytes fill 227 KB)
constexpr uint32_t kBarBytes = 256; // the barriers, in front of the slice
struct Bars {
    uint64_t full[kMaxStages], empty[kMaxStages];
    uint64_t xbox[kMaxBoxes];   // box i of the slice has landed
    uint64_t xfree;             // the consumers are done with the slice
    uint64_t ready, freed;
};
static_assert(sizeof(Bars) <= kBarBytes, "the barriers fit in front of the slice");

// A row set as the kernel keeps it in registers (constant indexing only).
struct Set {
    int g0, ng, m, n, nib, nrows_last;
    long long val_off, off_off;
};

template <bool BF16, int T>
__global__ void __launch_bounds__(kThreads, 1)
xres_kernel(Format f, const float *__restrict__ X, int64_t batch, float *__restrict__ Y, int64_t ldy,
            const __grid_constant__ CUtensorMap xmap, const __grid_constant__ Plan p) {
    static_assert(T == 32, "the consumer layouts assume 32-column tiles (128-byte activation rows)");
    constexpr int kEsz = BF16 ? 2 : 4;
    extern __shared__ __align__(128) unsigned char sm[];
    Bars &bar = *reinterpret_cast<Bars *>(sm);
    float *s_x = reinterpret_cast<float *>(sm + kBarBytes);
    unsigned char *s_ring = sm + p.ring_off;
    float *s_part = reinterpret_cast<float *>(sm + p.part_off);   // [kMaxGroups * 32 rows][T]

    pdl_launch_dependents();
    cg::cluster_group cluster = cg::this_cluster();
    const int C = p.C, NS = p.nst;
    const int q = static_cast<int>(cluster.block_rank());
    const int cl = static_cast<int>(blockIdx.x) / C;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int u_begin = p.range[cl].x, u_end = p.range[cl].y;
    const SetGeo *sets = f.xsets[p.table];
    const int kq0 = q * p.S;                // first activation row of the slice

    if (tid == 0) {
        for (int st = 0; st < NS; ++st) {
            mbar_init(&bar.full[st], 1);
            mbar_init(&bar.empty[st], kCWarps);
        }
        for (int i = 0; i < p.nboxes; ++i) mbar_init(&bar.xbox[i], 1);
        mbar_init(&bar.xfree, kCWarps);
        mbar_init(&bar.ready, kCWarps * C);   // every consumer warp of every CTA, once a set
        mbar_init(&bar.freed, kRWarps * C);   // every reducer warp of every CTA, once a set
        fence_mbar_init();
    }
    // every CTA's barriers exist before any CTA arrives on them remotely
    cluster.sync();
    pdl_wait_previous();   // X may come from the previous kernel, and Y may still be read by it

    // A unit's row set, loaded one unit ahead so that its latency hides behind
    // the current unit's work.
    // (volatile loads: issued where they are written, a whole unit before use,
    // instead of being moved down to it)
    auto load_set = [&](int sidx) {
        const int4 *src = reinterpret_cast<const int4 *>(sets + sidx);
        int4 a, b, c;
        asm volatile("ld.global.nc.v4.s32 {%0, %1, %2, %3}, [%4];" : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w) : "l"(src));
        asm volatile("ld.global.nc.v4.s32 {%0, %1, %2, %3}, [%4];" : "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w) : "l"(src + 1));
        asm volatile("ld.global.nc.v4.s32 {%0, %1, %2, %3}, [%4];" : "=r"(c.x), "=r"(c.y), "=r"(c.z), "=r"(c.w) : "l"(src + 2));
        Set s;
        s.g0 = a.x; s.ng = a.y; s.m = a.z; s.n = a.w;
        s.nib = b.x; s.nrows_last = b.y;
        s.val_off = static_cast<long long>((static_cast<unsigned long long>(static_cast<unsigned>(b.w)) << 32) |
                                           static_cast<unsigned>(b.z));
        s.off_off = static_cast<long long>((static_cast<unsigned long long>(static_cast<unsigned>(c.y)) << 32) |
                                           static_cast<unsigned>(c.x));
        return s;
    };
    // This CTA's share of a unit: blocks [j0, j1), chunks [c0, c0 + nch), in rounds of cpr chunks.
    struct Unit {
        int tile, j0, j1, c0, nch, cpr, rounds;
    };
    // Unit u = tile * nsets + sidx; the running position (no division per unit).
    struct Cursor {
        int tile, sidx;
    };
    auto cursor_at = [&](int u) {
        Cursor c;
        c.tile = u / p.nsets;
        c.sidx = u - c.tile * p.nsets;
        return c;
    };
    auto advance = [&](Cursor &c) {
        if (++c.sidx == p.nsets) {
            c.sidx = 0;
            ++c.tile;
        }
    };
    // The first blocks of this slice in a row of block size m, ceil(q*S / m) and
    // ceil((q+1)*S / m), recomputed only when m changes (the sets of a bin are
    // consecutive, so a CTA divides a few times per launch).
    int geo_m = -1, geo_ja = 0, geo_jb = 0;
    auto unit_geo = [&](int tile, const Set &s) {
        Unit g;
        g.tile = tile;
        if (s.m != geo_m) {
            const unsigned lo = static_cast<unsigned>(q) * static_cast<unsigned>(p.S), hi = lo + static_cast<unsigned>(p.S);
            const unsigned mu = static_cast<unsigned>(s.m);
            geo_m = s.m;
            geo_ja = static_cast<int>((lo + mu - 1) / mu);
            geo_jb = static_cast<int>((hi + mu - 1) / mu);
        }
        g.j0 = geo_ja < s.n ? geo_ja : s.n;
        g.j1 = geo_jb < s.n ? geo_jb : s.n;
        g.c0 = g.j0 / kChunk;
        g.nch = g.j1 > g.j0 ? (g.j1 + kChunk - 1) / kChunk - g.c0 : 0;
        g.cpr = max(1, kRecCap / max(1, s.ng));
        g.rounds = (g.nch + g.cpr - 1) / g.cpr;
        return g;
    };

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------ producer
        bool ok = true;
        int rc = 0;           // rounds issued
        int pst = 0;          // the stage of round rc (rc % NS)
        uint32_t pph = 0u;    // and the parity of its use ((rc / NS) & 1)
        int xloads = 0;       // slices loaded
        int cur_tile = -1;
        // the boxes of tile `tile`'s slice, each completing its own barrier.  A
        // box no round needed (past the matrix) may not have been waited for:
        // every box of the previous slice has landed before a box is reused,
        // so that the phases of a box's barrier never overlap
        // (false, nothing issued, if one of them did not land in time)
        auto load_slice = [&](int tile) {
            bool drained = true;
            if (lane == 0 && xloads > 0)
                for (int i = 0; i < p.nboxes; ++i) drained = mbar_wait(&bar.xbox[i], (xloads - 1) & 1) && drained;
            if (__shfl_sync(0xFFFFFFFFu, drained ? 1 : 0, 0) == 0) return false;
            if (lane == 0) {
                fence_proxy_async_smem();
                for (int i = 0; i < p.nboxes; ++i) {
                    mbar_arrive_expect_tx(&bar.xbox[i], uint32_t(p.box_rows) * T * 4);
                    tensor2d_g2s(s_x + size_t(i) * p.box_rows * T, &xmap, tile * T, kq0 + i * p.box_rows,
                                 &bar.xbox[i]);
                }
            }
            ++xloads;
            cur_tile = tile;
            return true;
        };
        Cursor cu = cursor_at(u_begin), cn = cu;
        advance(cn);
        if (u_begin < u_end) ok = load_slice(cu.tile);   // the run's first tile is known: no wait for its set
        Set s_next = u_begin < u_end ? load_set(cu.sidx) : Set{};
        for (int u = u_begin; u < u_end && ok; ++u, cu = cn, advance(cn)) {
            const Set s = s_next;
            if (u + 1 < u_end) s_next = load_set(cn.sidx);
            const Unit g = unit_geo(cu.tile, s);
            if (g.tile != cur_tile) {
                // the consumers are done with the previous slice
                if (xloads > 0) ok = mbar_wait(&bar.xfree, (xloads - 1) & 1, false);
                ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
                if (!ok) break;
                ok = load_slice(g.tile);
                if (!ok) break;
            }
            const int rw = s.nib ? 1 : 2;
            const int64_t gnch = (s.n + kChunk - 1) / kChunk;   // chunks of a group
            for (int r = 0; r < g.rounds; ++r, ++rc) {
                const int st = pst;
                if (rc >= NS) ok = mbar_wait(&bar.empty[st], pph ^ 1u, false);
                ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
                if (!ok) break;
                if (lane == 0) {
                    const int cr0 = g.c0 + r * g.cpr, nchr = min(g.cpr, g.nch - r * g.cpr);
                    const uint32_t bv = uint32_t(nchr) * kSlots * kChunk * kEsz;
                    const uint32_t bo = uint32_t(nchr) * kSlots * rw * 4;
                    unsigned char *sv = s_ring + size_t(st) * stage_bytes<BF16>();
                    unsigned char *so = sv + ring_val_bytes<BF16>();
                    fence_proxy_async_smem();
                    mbar_arrive_expect_tx(&bar.full[st], uint32_t(s.ng) * (bv + bo));
                    for (int gi = 0; gi < s.ng; ++gi) {
                        const int64_t vo = s.val_off + (gi * gnch + cr0) * (kSlots * kChunk);
                        const int64_t oo = s.off_off + (gi * gnch + cr0) * (kSlots * rw);
                        bulk_g2s(sv + size_t(gi) * bv, static_cast<const unsigned char *>(f.vals) + vo * kEsz, bv,
                                 &bar.full[st]);
                        bulk_g2s(so + size_t(gi) * bo, f.offs + oo, bo, &bar.full[st]);
                    }
                }
                if (++pst == NS) {
                    pst = 0;
                    pph ^= 1u;
                }
            }
        }
        if (!ok && lane == 0) atomicOr(f.status, kStatusTimeout);
        // the copies this CTA started have landed before it can leave
        if (lane == 0) {
            for (int k = 1; k <= NS && k <= rc; ++k) {
                const int last = rc - k;
                mbar_wait(&bar.full[last % NS], (last / NS) & 1);
            }
            if (xloads > 0)
                for (int i = 0; i < p.nboxes; ++i) mbar_wait(&bar.xbox[i], (xloads - 1) & 1);
        }
    } else if (warp > kProducerWarp) {
        // ------------------------------------------------------------ reducers
        const int rt = tid - (kCThreads + 32);   // 0 .. kRThreads-1
        bool ok = true;
        Cursor cu = cursor_at(u_begin), cn = cu;
        advance(cn);
        Set s_next = u_begin < u_end ? load_set(cu.sidx) : Set{};
        for (int u = u_begin, t = 0; u < u_end; ++u, ++t, cu = cn, advance(cn)) {
            const Set s = s_next;
            if (u + 1 < u_end) s_next = load_set(cn.sidx);
            if (ok) ok = mbar_wait_acq_cluster(&bar.ready, t & 1);
            if (ok) {
                const int64_t tile = cu.tile;
                // this CTA's rows of the set: [q R / C, (q + 1) R / C)
                const int R = s.ng * kSlots, r0 = q * R / C, r1 = (q + 1) * R / C;
                for (int i = rt; i < (r1 - r0) * (T / 4); i += kRThreads) {
                    const int row = r0 + i / (T / 4), c4 = i % (T / 4);
                    const int gg = row / kSlots, sl = row % kSlots;
                    if (gg == s.ng - 1 && sl >= s.nrows_last) continue;
                    const int idx = row * (T / 4) + c4;
                    // ranks in a fixed order (deterministic), four loads in flight at a time
                    float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                    for (int h = 0; h < 8; h += 4) {
                        float4 pv[4];
#pragma unroll
                        for (int r = 0; r < 4; ++r)
                            if (h + r < C)
                                pv[r] = reinterpret_cast<const float4 *>(cluster.map_shared_rank(s_part, h + r))[idx];
#pragma unroll
                        for (int r = 0; r < 4; ++r)
                            if (h + r < C) {
                                if (h + r == 0) {
                                    sum = pv[r];
                                } else {
                                    sum.x += pv[r].x;
                                    sum.y += pv[r].y;
                                    sum.z += pv[r].z;
                                    sum.w += pv[r].w;
                                }
                            }
                    }
                    float *yr = Y + int64_t(f.rowmap[(s.g0 + gg) * kSlots + sl]) * ldy;
                    const int64_t b0 = tile * T + c4 * 4;
                    if (b0 < batch) yr[b0] = sum.x;
                    if (b0 + 1 < batch) yr[b0 + 1] = sum.y;
                    if (b0 + 2 < batch) yr[b0 + 2] = sum.z;
                    if (b0 + 3 < batch) yr[b0 + 3] = sum.w;
                }
            }
            // this warp is done reading the partial sums of every CTA: tell them all
            __syncwarp();
            if (lane < C) mbar_arrive_remote(&bar.freed, static_cast<uint32_t>((q + lane) % C));   // one lane per CTA
        }
        if (!ok && lane == 0) atomicOr(f.status, kStatusTimeout);
    } else {
        // ------------------------------------------------------------ consumers
        // Two layouts of the consumer threads, chosen per set:
        //  * LPR = 4 lanes a row (sets of more than 64 rows): a lane owns 8 of
        //    the tile's 32 columns, quads qd + 4h and then qd + 4(1 - h) (h =
        //    parity of its row), so that one offset, one value and one address
        //    serve two 16-byte loads, and the two rows of a quarter-warp read
        //    opposite halves of their activation rows -- 8 distinct bank groups;
        //  * LPR = 8 lanes a row (sets of up to 64 rows, which would leave half
        //    of a 128-row pass idle): a lane owns one quad, a quarter-warp reads
        //    one whole activation row.
        bool ok = true;
        int rc = 0, xloads = 0, cur_tile = -1;
        int nready = 0;       // boxes of the current slice known to have landed
        int cst = 0;          // the stage of round rc (rc % NS)
        uint32_t cph = 0u;    // and the parity of its use ((rc / NS) & 1)
        Cursor cu = cursor_at(u_begin), cn = cu;
        advance(cn);
        Set s_next = u_begin < u_end ? load_set(cu.sidx) : Set{};
        const uint32_t x0 = smem_addr(s_x);   // slice row k at x0 + 128 k (rows of 32 floats)
        // one unit with LPR lanes a row, NP row passes and 4-bit (NIB) or 8-bit
        // offsets: multiply, then store the partial sums once every CTA's
        // reducers have read the previous set's (t: sets stored)
        auto unit = [&](auto lprc, auto npc, auto nibc, const Set &s, const Unit &g, int t) {
            constexpr int LPR = decltype(lprc)::value;
            constexpr int NP = decltype(npc)::value;
            constexpr bool NIB = decltype(nibc)::value;
            constexpr bool kTwo = LPR == 4;          // two quads a lane
            constexpr int kRpw = 32 / LPR;           // rows per warp and pass
            constexpr int kPassRows = kCWarps * kRpw;
            const int qd = lane % LPR;
            const int cA = kTwo ? qd + 4 * ((lane >> 2) & 1) : qd;   // the lane's (first) column quad
            const int cB = cA ^ 4;                                   // its second (LPR = 4)
            const int rs = warp * kRpw + lane / LPR;                 // row of the set in pass 0
            const uint32_t xl = x0 + uint32_t(cA) * 16u;
            float4 accA[NP], accB[NP];
#pragma unroll
            for (int pp = 0; pp < NP; ++pp) accA[pp] = accB[pp] = make_float4(0.f, 0.f, 0.f, 0.f);
            // a row past the set (the last pass of a set with fewer groups) repeats a
            // row of its last group; its sums are stored but never read
            int gip[NP], slotp[NP];
#pragma unroll
            for (int pp = 0; pp < NP; ++pp) {
                const int row = rs + pp * kPassRows;
                gip[pp] = min(row / kSlots, s.ng - 1);
                slotp[pp] = row % kSlots;
            }
            const uint32_t mrow = uint32_t(s.m) << 7;   // bytes between the first rows of consecutive blocks
            for (int r = 0; r < g.rounds; ++r, ++rc) {
                const int st = cst;
                if (ok) ok = mbar_wait(&bar.full[st], cph, false);
                const int cr0 = g.c0 + r * g.cpr, nchr = min(g.cpr, g.nch - r * g.cpr);
                // the boxes holding the slice rows this round's blocks can select
                // (rows below (cr0 + nchr) * 8 * m - kq0), in order
                const int hi = (cr0 + nchr) * kChunk * s.m - kq0;
                while (ok && nready < p.nboxes && nready * p.box_rows < hi) {
                    ok = mbar_wait(&bar.xbox[nready], (xloads - 1) & 1, false);
                    ++nready;
                }
                ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
                if (ok) {
                    const unsigned char *sv = s_ring + size_t(st) * stage_bytes<BF16>();
                    const uint32_t *so = reinterpret_cast<const uint32_t *>(sv + ring_val_bytes<BF16>());
                    for (int lc = 0; lc < nchr; ++lc) {
                        const int jc = (cr0 + lc) * kChunk;
                        const int e_lo = max(0, g.j0 - jc), e_hi = min(kChunk, g.j1 - jc);
                        // address of the slice row selected by block jc + e:
                        // xl + (((jc + e) * m + off - kq0) << 7) (below the slice for a first
                        // chunk whose leading blocks belong to the previous slice; those
                        // blocks are never read)
                        const uint32_t xb = xl + (uint32_t(jc * s.m - kq0) << 7);
#pragma unroll
                        for (int pp = 0; pp < NP; ++pp) {
                            const int rec = (gip[pp] * nchr + lc) * kSlots + slotp[pp];
                            uint32_t vw[BF16 ? 4 : 8];
                            {
                                const uint4 *pv = reinterpret_cast<const uint4 *>(sv) + rec * (BF16 ? 1 : 2);
                                const uint4 w0 = pv[0];
                                vw[0] = w0.x; vw[1] = w0.y; vw[2] = w0.z; vw[3] = w0.w;
                                if constexpr (!BF16) {
                                    const uint4 w1 = pv[1];
                                    vw[4] = w1.x; vw[5] = w1.y; vw[6] = w1.z; vw[7] = w1.w;
                                }
                            }
                            const uint2 ow = NIB ? make_uint2(so[rec], 0u) : reinterpret_cast<const uint2 *>(so)[rec];
                            // block e: its kept value times the lane's quads of its selected activation row
                            auto block = [&](int e) {
                                uint32_t off;
                                if constexpr (NIB) off = (ow.x >> (4 * e)) & 15u;
                                else off = ((e < 4 ? ow.x : ow.y) >> (8 * (e & 3))) & 255u;
                                float v;
                                if constexpr (BF16)
                                    v = __uint_as_float((e & 1) ? (vw[e >> 1] & 0xFFFF0000u) : (vw[e >> 1] << 16));
                                else
                                    v = __uint_as_float(vw[e]);
                                const uint32_t ad = xb + uint32_t(e) * mrow + (off << 7);
                                fma4(accA[pp], v, lds_f4(ad));
                                if constexpr (kTwo) fma4(accB[pp], v, lds_f4(ad ^ 64u));   // the other half of the row
                            };
                            if (e_lo == 0 && e_hi == kChunk) {
                                // a whole chunk: one straight run, every load can be issued early
#pragma unroll
                                for (int e = 0; e < kChunk; ++e) block(e);
                            } else {
#pragma unroll
                                for (int e = 0; e < kChunk; ++e)
                                    if (e >= e_lo && e < e_hi) block(e);
                            }
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&bar.empty[st]);
                if (++cst == NS) {
                    cst = 0;
                    cph ^= 1u;
                }
            }
            if (t >= 1 && ok) ok = mbar_wait_acq_cluster(&bar.freed, (t - 1) & 1);
#pragma unroll
            for (int pp = 0; pp < NP; ++pp) {
                float4 *pr = reinterpret_cast<float4 *>(s_part) + (rs + pp * kPassRows) * (T / 4);
                pr[cA] = accA[pp];
                if constexpr (kTwo) pr[cB] = accB[pp];
            }
        };
        int t = 0;   // sets stored
        for (int u = u_begin; u < u_end; ++u, ++t, cu = cn, advance(cn)) {
            const Set s = s_next;
            if (u + 1 < u_end) s_next = load_set(cn.sidx);
            const Unit g = unit_geo(cu.tile, s);
            if (g.tile != cur_tile) {
                if (xloads > 0) {   // done with the previous slice
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&bar.xfree);
                }
                ++xloads;           // its boxes are waited for by the rounds that read them
                nready = 0;
                cur_tile = g.tile;
            }
            using L4 = std::integral_constant<int, 4>;
            using L8 = std::integral_constant<int, 8>;
            using N1 = std::integral_constant<int, 1>;
            using Nib = std::true_type;
            using Byte = std::false_type;
            static_assert(kCWarps * 8 >= kMaxGroups * kSlots, "one 128-row pass covers the largest set");
            const int rows = s.ng * kSlots;
            if (rows <= kCWarps * 4) {   // one pass of 8 lanes a row
                if (s.nib) unit(L8{}, N1{}, Nib{}, s, g, t);
                else unit(L8{}, N1{}, Byte{}, s, g, t);
            } else {                     // one pass of 4 lanes a row
                if (s.nib) unit(L4{}, N1{}, Nib{}, s, g, t);
                else unit(L4{}, N1{}, Byte{}, s, g, t);
            }
            // this warp's partial sums are stored: tell every CTA's reducers
            __syncwarp();
            if (lane < C) mbar_arrive_remote(&bar.ready, static_cast<uint32_t>((q + lane) % C));   // one lane per CTA
        }
        // every CTA's reducers have read this CTA's last partial sums
        if (t >= 1 && ok) ok = mbar_wait_acq_cluster(&bar.freed, (t - 1) & 1);
        if (xloads > 0) {
            __syncwarp();
            if (lane == 0) mbar_arrive(&bar.xfree);
        }
        if (!ok && lane == 0) atomicOr(f.status, kStatusTimeout);
    }
    cluster.sync();   // no CTA leaves while another may still read its shared memory
}


// Clusters of C CTAs of this kernel resident at once with `smem` bytes each.
template <bool BF16, int T>
inline int max_clusters(int C, uint32_t smem) {
    const auto fn = xres_kernel<BF16, T>;
    return static_cast<int>(per_device(reinterpret_cast<const void *>(fn), (long long)C << 32 | smem, [&]() -> long long {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(C) * 64);
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = static_cast<unsigned>(C);
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) {
            cudaGetLastError();
            n = 0;
        }
        return n;
    }));
}

// The product on this kernel, or cudaErrorNotSupported when the call does not
// fit it (the slice of the tile does not fit in shared memory even split 8
// ways with a two-stage ring, or X cannot be described by a tensor map).
template <bool BF16, int T>
cudaError_t launch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy, bool early,
                   cudaStream_t stream) {
    (void)early;
    const int64_t tiles = (batch + T - 1) / T;
    if (f.nxsets[0] <= 0 || f.nxsets[1] <= 0 || f.xset_prefix[0] == nullptr || f.xset_prefix[1] == nullptr ||
        tiles * f.nxsets[0] > (int64_t(1) << 30))
        return cudaErrorNotSupported;
    if (reinterpret_cast<uintptr_t>(X) % 16 != 0 || (ldx * 4) % 16 != 0) return cudaErrorNotSupported;
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (enc == nullptr) return cudaErrorNotSupported;
    const cudaError_t attr = allow_smem(xres_kernel<BF16, T>, kSmemCap);
    if (attr != cudaSuccess) return attr;
    // least common multiple of the block sizes (0 when it grows past any slice)
    int64_t lcm = 1;
    for (int i = 0; i < f.nxsets[0] && lcm != 0; ++i) {
        const int64_t m = f.xsets_host[0][i].m;
        int64_t a = lcm, b = m;
        while (b != 0) {
            const int64_t r = a % b;
            a = b;
            b = r;
        }
        lcm = lcm / a * m;
        if (lcm > f.cols) lcm = 0;
    }
    // Per split C = 1 .. 8: slices of S columns.  A slice's blocks start in
    // [q S, (q + 1) S) and select rows up to m_max - 1 past it (rows past the
    // matrix arrive as zeros), unless S is a multiple of every block size: then
    // no block crosses into the next slice and the slice is S rows, which is
    // used whenever it is no longer.  Beside the slice: the deepest ring that
    // fits (up to kMaxStages) and the partial sums of the largest set.  Of the
    // splits with kMinStages or more, the one whose clusters occupy the most
    // SMs, then the deeper ring, then the smaller split; a shallower ring only
    // when no split has that.
    Plan p{};
    uint32_t smem = 0;
    int64_t best_sms = 0;
    int best_nst = 0;
    bool best_deep = false;
    for (int C = 1; C <= 8; ++C) {
        int64_t S = (f.cols + C - 1) / C;
        int64_t rows = S + f.m_max - 1;
        if (lcm > 0) {
            const int64_t Sa = (S + lcm - 1) / lcm * lcm;
            if (Sa <= rows) S = rows = Sa;
        }
        const int nboxes = static_cast<int>((rows + 255) / 256);
        const int box_rows = static_cast<int>((rows + nboxes - 1) / nboxes);
        const uint64_t x_bytes = uint64_t(nboxes) * box_rows * T * 4;
        if (nboxes > kMaxBoxes) continue;
        const uint64_t ring_off = kBarBytes + x_bytes;
        const uint64_t part_bytes = uint64_t(kMaxGroups) * kSlots * T * 4;
        if (ring_off + 2 * stage_bytes<BF16>() + part_bytes > kSmemCap) continue;
        const int nst = static_cast<int>(
            std::min<uint64_t>(kMaxStages, (kSmemCap - ring_off - part_bytes) / stage_bytes<BF16>()));
        const uint64_t part_off = ring_off + uint64_t(nst) * stage_bytes<BF16>();
        const uint32_t total = static_cast<uint32_t>(part_off + part_bytes);
        const int64_t sms = std::min<int64_t>(max_clusters<BF16, T>(C, total), kMaxClusters) * C;
        const bool deep = nst >= kMinStages;
        const bool better = deep != best_deep ? deep : (sms != best_sms ? sms > best_sms : nst > best_nst);
        if (sms <= 0 || !better) continue;
        best_sms = sms;
        best_nst = nst;
        best_deep = deep;
        p.C = C;
        p.S = static_cast<int>(S);
        p.nst = nst;
        p.box_rows = box_rows;
        p.nboxes = nboxes;
        p.x_bytes = static_cast<uint32_t>(x_bytes);
        p.ring_off = static_cast<uint32_t>(ring_off);
        p.part_off = static_cast<uint32_t>(part_off);
        smem = total;
    }
    if (best_sms <= 0) return cudaErrorNotSupported;
    const int64_t occ = std::min<int64_t>(max_clusters<BF16, T>(p.C, smem), kMaxClusters);
    // Row sets of about 4 heaviest groups (table 1: 128 rows, the consumers'
    // efficient layout) when they still give every cluster 2 units or more;
    // else sets of about 2 (table 0), whose finer units balance better.  (At
    // 3 units a cluster FC6 batch 64 took table 0 on clusters of 6: 20.3
    // against 18.8 us; at 1, FC7 batch 64 took table 1: 13.8 against 12.8.)
    const int table = tiles * f.nxsets[1] >= 2 * occ ? 1 : 0;
    const int nsets = f.nxsets[table];
    const int64_t units = tiles * nsets;
    p.table = table;
    p.nsets = nsets;
    const int ncl = static_cast<int>(std::min<int64_t>(occ, units));
    if (ncl <= 0) return cudaErrorNotSupported;
    // Contiguous runs of units, at most ncl of them, whose longest is as short
    // as it can be.  The ranks of a cluster go through a unit together, so a
    // unit costs what its busiest rank streams -- its set's groups times the
    // most chunks any slice's blocks touch -- plus a fixed cost per unit (the
    // hand-off of its partial sums and the start of its rounds); a run that
    // crosses into the next batch tile also pays for the drain of its
    // consumers and the load of the new slice.  kUnitCost and kSwitchCost
    // were swept on FC6/FC7 at batch 64 and 256 (10 and 40 group-chunks of
    // multiplying).  The bound on a run is found by bisection, each candidate
    // tried by a greedy pass that closes a run where the next unit would pass
    // it.
    thread_local std::vector<int64_t> cost;   // host; reused across calls
    const SetGeo *hs = f.xsets_host[table];
    cost.assign(static_cast<size_t>(nsets) + 1, 0);
    for (int s = 0; s < nsets; ++s) {
        int64_t most = 0;
        for (int qq = 0; qq < p.C; ++qq) {
            const int64_t lo = int64_t(qq) * p.S, hi = lo + p.S;
            const int64_t j0 = std::min<int64_t>(hs[s].n, (lo + hs[s].m - 1) / hs[s].m);
            const int64_t j1 = std::min<int64_t>(hs[s].n, (hi + hs[s].m - 1) / hs[s].m);
            if (j1 > j0) most = std::max<int64_t>(most, (j1 + kChunk - 1) / kChunk - j0 / kChunk);
        }
        cost[static_cast<size_t>(s) + 1] = cost[static_cast<size_t>(s)] + hs[s].ng * most + kUnitCost;
    }
    const int64_t *pre = cost.data();
    // One greedy pass for a bound: a run takes its first unit whatever that
    // costs, then the following units while they fit, a unit that opens a
    // tile inside the run carrying kSwitchCost.  Whole tiles are taken at
    // once and the fitting prefix of a tile is found in the prefix sums, so a
    // pass costs about one step per tile and per run, not one per unit.
    const int64_t wt = pre[nsets];   // the units of one tile
    auto greedy = [&](int64_t bound, bool write) {
        int c = 0;
        for (int64_t u = 0; u < units; ++c) {
            const int64_t u0 = u;
            int64_t sidx = u % nsets;
            int64_t acc = pre[sidx + 1] - pre[sidx];
            ++u;
            ++sidx;
            while (u < units) {
                if (sidx == nsets) {   // the next unit opens a tile
                    if (acc + kSwitchCost + wt <= bound) {
                        acc += kSwitchCost + wt;
                        u += nsets;
                        continue;
                    }
                    const int64_t k = std::upper_bound(pre, pre + nsets + 1, bound - acc - kSwitchCost) - pre - 1;
                    if (k > 0) u += k;
                    break;
                }
                // the largest e with pre[e] - pre[sidx] <= bound - acc (e >= sidx: acc <= bound)
                const int64_t e = std::upper_bound(pre + sidx, pre + nsets + 1, bound - acc + pre[sidx]) - pre - 1;
                u += e - sidx;
                if (e < nsets) break;
                acc += wt - pre[sidx];
                sidx = nsets;
            }
            if (write) p.range[c] = make_int2(static_cast<int>(u0), static_cast<int>(u));
        }
        return c;
    };
    int64_t lo = 0;
    for (int sidx = 0; sidx < nsets; ++sidx) lo = std::max<int64_t>(lo, pre[sidx + 1] - pre[sidx]);
    int64_t hi = tiles * (wt + kSwitchCost);   // one run of everything fits
    while (lo < hi) {   // the smallest bound whose runs fit ncl clusters
        const int64_t mid = lo + (hi - lo) / 2;
        if (greedy(mid, false) <= ncl) hi = mid;
        else lo = mid + 1;
    }
    const int nrun = greedy(lo, true);
    CUtensorMap xmap;
    std::memset(&xmap, 0, sizeof xmap);
    const cuuint64_t dims[2] = {cuuint64_t(batch), cuuint64_t(f.cols)};
    const cuuint64_t strides[1] = {cuuint64_t(ldx) * 4};
    const cuuint32_t box[2] = {cuuint32_t(T), cuuint32_t(p.box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    if (enc(&xmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(X), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return cudaErrorNotSupported;
    return launch_ex(xres_kernel<BF16, T>, dim3(static_cast<unsigned>(nrun * p.C)), dim3(kThreads), smem, stream,
                     static_cast<unsigned>(p.C), true, f, X, batch, Y, ldy, xmap, p);
}

}  // namespace xres
}  // namespace darb
