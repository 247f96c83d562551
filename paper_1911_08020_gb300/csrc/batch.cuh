// batch.cuh -- the batch-per-lane product kernel (batch > 4), as a template
// over its output: plain Y, or the gate sums of a fused LSTM / GRU step.
//
// Work unit (a WorkItem of the handle's tables): a row set (up to 8
// consecutive 32-row groups of one block-size bin, so up to 256 rows), the
// share of its blocks one cluster rank multiplies -- sets of small block size
// have more blocks per row and are split over more ranks, so every CTA gets
// about the same work -- and one batch tile of LPR*CPL columns.  The rank's blocks are walked in rounds
// through a two-stage ring in shared memory.  A producer warp starts, per
// round, the bulk (TMA) copies of the round's kept values and packed offsets
// (one contiguous run per group) and the 2-D tensor-map copies of the
// activation rows those blocks can select, X[j*m .. j*m+m) for the batch tile
// (rows and columns out of range arrive as zeros).  Eight consumer warps wait
// on the stage's "full" barrier, compute, and release it on its "empty"
// barrier; no CTA-wide barrier separates rounds.  In the consumers LPR lanes
// share a row and each lane owns CPL columns, interleaved so that a
// quarter-warp reads 128 contiguous bytes of an activation row: the gathers
// are free of bank conflicts and each kept value is reused across the tile's
// columns from registers.  A thread works on the same chunk of all its rows at
// once, so the gathers of different rows overlap.  Accumulators live in
// registers across rounds; at the end the ranks of a set add their partial
// sums through distributed shared memory in a fixed order (deterministic),
// each rank finishing a slice of the set's rows.
//
// Why row sets: an activation row staged in shared memory is selected by about
// rows/m of the set's rows, so staging traffic per FMA is 4*m/rows bytes;
// 128-256 rows keep it well under the on-chip bandwidth for the block sizes the
// paper uses.
//
// RNN modes read the stacked input [x_t; h_{t-1}] in place through two tensor
// maps; the rows from x and the rows from h land in two regions of the stage.
#pragma once

#include "kernels_common.cuh"
#include "launch.cuh"
#include "rnn_epilogue.cuh"
#include "tma.cuh"

#include <cooperative_groups.h>
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>

namespace darb {
namespace batch {

namespace cg = cooperative_groups;

constexpr int kXcapB = 8192;      // activation floats per round
constexpr int kXslack = 1024;     // room for the last tensor box of a region to run past it
constexpr int kXstage = kXcapB + kXslack;
constexpr int kRecCap = 16;       // (group, chunk) records staged per round
constexpr int kStages = 2;        // rounds in flight per CTA
constexpr int kConsumers = 8;     // consumer warps; one more warp produces
constexpr int kThreads = (kConsumers + 1) * 32;

// Lanes per row LPR, columns per lane CPL: the batch tile is LPR*CPL columns.
// Wide tiles keep fewer rows per set so that the accumulators fit in registers.
template <int LPR, int CPL>
__host__ __device__ constexpr int max_set_groups() { return CPL == 8 ? 4 : 8; }

template <int LPR, int CPL>
__host__ __device__ constexpr int box_rows() { return kXslack / (LPR * CPL); }

template <bool BF16>
__host__ __device__ constexpr size_t stage_val_bytes() { return size_t(kRecCap) * kSlots * kChunk * (BF16 ? 2 : 4); }

constexpr size_t kStageOffBytes = size_t(kRecCap) * kSlots * 2 * 4;

template <bool BF16>
__host__ __device__ constexpr size_t smem_bytes() {
    return 128 + kStages * (size_t(kXstage) * 4 + stage_val_bytes<BF16>() + kStageOffBytes);
}

// Largest block size a tile of kBt columns can stage for one block (plus, for
// the stacked RNN input, one box of slack for the second region).
template <int LPR, int CPL>
__host__ __device__ constexpr int max_block(bool stacked) {
    return kXcapB / (LPR * CPL) - (stacked ? box_rows<LPR, CPL>() : 0);
}

// Where the activation rows of a round sit in its stage: rows [kx0, kxa) of the
// x part at tile row 0, rows [kxb, kx1) of the h part at tile row hbase.
struct Round {
    int jr0, jr1, cr0, nchr;   // blocks [jr0, jr1), chunks [cr0, cr0 + nchr)
    int kx0, kxa, kxb, kx1;    // activation rows
    int hbase;                 // first tile row of the h part
};

// One chunk (8 blocks) of one row slot: decode the offsets and add the 8 kept
// values times their selected activation rows into acc (SPLIT: rows >= split
// into acc2).  NIB (4-bit offsets), WHOLE (all 8 blocks inside the round) and
// STACKED (two regions) are compile-time so that the innermost loop is just
// offset extraction, one address, the loads and the FMAs.
template <bool BF16, bool NIB, bool WHOLE, bool STACKED, bool SPLIT, int KQ, int LPR>
__device__ __forceinline__ void chunk(const unsigned char *s_vals, const uint32_t *s_offs, int rec,
                                      const float4 *sx4, int qd, const Round &g, int jc, int m, int row_f4,
                                      int e_lo, int e_hi, int split, float4 (&acc)[KQ], float4 (&acc2)[KQ]) {
    float v[kChunk];
    if constexpr (BF16) {
        const uint4 w4 = *reinterpret_cast<const uint4 *>(s_vals + size_t(rec) * 16);
        const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            v[2 * e] = __uint_as_float(w[e] << 16);
            v[2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
        }
    } else {
        const float4 *pv = reinterpret_cast<const float4 *>(s_vals + size_t(rec) * 32);
        const float4 x0 = pv[0], x1 = pv[1];
        v[0] = x0.x; v[1] = x0.y; v[2] = x0.z; v[3] = x0.w;
        v[4] = x1.x; v[5] = x1.y; v[6] = x1.z; v[7] = x1.w;
    }
    uint2 ow;
    if constexpr (NIB) ow = make_uint2(s_offs[rec], 0u);
    else ow = reinterpret_cast<const uint2 *>(s_offs)[rec];
    const int mstride = m * row_f4;
    const float4 *xb = sx4 + (jc * m - g.kx0) * row_f4 + qd;
#pragma unroll
    for (int e = 0; e < kChunk; ++e) {
        if (WHOLE || (e >= e_lo && e < e_hi)) {
            int off;
            if constexpr (NIB) off = int((ow.x >> (4 * e)) & 15u);
            else off = int(((e < 4 ? ow.x : ow.y) >> (8 * (e & 3))) & 255u);
            const float4 *xr;
            int kg = 0;
            if constexpr (STACKED) {
                kg = (jc + e) * m + off;
                const int tr = kg < g.kxa ? kg - g.kx0 : g.hbase + kg - g.kxb;
                xr = sx4 + tr * row_f4 + qd;
            } else {
                xr = xb + e * mstride + off * row_f4;
            }
            if (!SPLIT || kg < split) {
#pragma unroll
                for (int u = 0; u < KQ; ++u) {
                    const float4 xv = xr[u * LPR];
                    fma4(acc[u], v[e], xv);
                }
            } else {
#pragma unroll
                for (int u = 0; u < KQ; ++u) {
                    const float4 xv = xr[u * LPR];
                    fma4(acc2[u], v[e], xv);
                }
            }
        }
    }
}

// One chunk (8 blocks) of NP row slots of this thread at once (no GRU split):
// rec[p] is the staged record of row slot p.  Blocks outer, rows inner, so the
// activation loads of the NP rows of one block are in flight together and
// every accumulator gets one FMA per block.
template <bool BF16, bool NIB, bool WHOLE, bool STACKED, int NP, int KQ, int LPR>
__device__ __forceinline__ void chunk_rows(const unsigned char *s_vals, const uint32_t *s_offs, const int *rec,
                                           const float4 *sx4, int qd, const Round &g, int jc, int m, int row_f4,
                                           int e_lo, int e_hi, float4 (*acc)[KQ]) {
    constexpr int kW = BF16 ? 4 : 8;
    uint32_t vw[NP][kW];
    uint2 ow[NP];
#pragma unroll
    for (int p = 0; p < NP; ++p) {
        const uint4 *pv = reinterpret_cast<const uint4 *>(s_vals + size_t(rec[p]) * (BF16 ? 16 : 32));
        const uint4 w0 = pv[0];
        vw[p][0] = w0.x; vw[p][1] = w0.y; vw[p][2] = w0.z; vw[p][3] = w0.w;
        if constexpr (!BF16) {
            const uint4 w1 = pv[1];
            vw[p][4] = w1.x; vw[p][5] = w1.y; vw[p][6] = w1.z; vw[p][7] = w1.w;
        }
        if constexpr (NIB) ow[p] = make_uint2(s_offs[rec[p]], 0u);
        else ow[p] = reinterpret_cast<const uint2 *>(s_offs)[rec[p]];
    }
    const int mstride = m * row_f4;
    const float4 *xb = sx4 + (jc * m - g.kx0) * row_f4 + qd;
#pragma unroll
    for (int e = 0; e < kChunk; ++e) {
        if (WHOLE || (e >= e_lo && e < e_hi)) {
#pragma unroll
            for (int p = 0; p < NP; ++p) {
                int off;
                if constexpr (NIB) off = int((ow[p].x >> (4 * e)) & 15u);
                else off = int(((e < 4 ? ow[p].x : ow[p].y) >> (8 * (e & 3))) & 255u);
                float v;
                if constexpr (BF16) v = __uint_as_float((e & 1) ? (vw[p][e >> 1] & 0xFFFF0000u) : (vw[p][e >> 1] << 16));
                else v = __uint_as_float(vw[p][e]);
                const float4 *xr;
                if constexpr (STACKED) {
                    const int kg = (jc + e) * m + off;
                    const int tr = kg < g.kxa ? kg - g.kx0 : g.hbase + kg - g.kxb;
                    xr = sx4 + tr * row_f4 + qd;
                } else {
                    xr = xb + e * mstride + off * row_f4;
                }
#pragma unroll
                for (int u = 0; u < KQ; ++u) {
                    const float4 xv = xr[u * LPR];
                    fma4(acc[p][u], v, xv);
                }
            }
        }
    }
}

template <bool BF16, int LPR, int CPL, int MODE>
__global__ void __launch_bounds__(kThreads, 2)
batch_kernel(Format f, const WorkItem *__restrict__ items, const float *__restrict__ X, int64_t ldx, int64_t batch,
       float *__restrict__ Y, int64_t ldy, const __grid_constant__ CUtensorMap xmap,
       const __grid_constant__ CUtensorMap hmap, RnnArgs ra, int use_tma, int early) {
    constexpr bool kStacked = MODE != kModeY;
    constexpr bool kSplit = MODE == kModeGru;
    constexpr int kParts = kSplit ? 2 : 1;
    constexpr int kBt = LPR * CPL;        // batch tile
    constexpr int kQ = CPL / 4;           // float4 per lane
    constexpr int kRpw = 32 / LPR;        // rows per consumer warp at a time
    constexpr int kRptMax = max_set_groups<LPR, CPL>() * kSlots / (kConsumers * kRpw);
    constexpr int kBoxRows = box_rows<LPR, CPL>();
    constexpr int kEsz = BF16 ? 2 : 4;
    // rows a thread multiplies together in the inner loop
    constexpr int kNpg = (BF16 || kQ == 1) ? (kRptMax < 4 ? kRptMax : 4) : (kRptMax < 2 ? kRptMax : 2);
    static_assert(kRptMax % kNpg == 0, "row passes come in whole sub-groups");
    extern __shared__ __align__(128) unsigned char sm[];
    // layout: full[kStages] empty[kStages] | X stages | values stages | offsets stages
    uint64_t *full = reinterpret_cast<uint64_t *>(sm);
    uint64_t *empty = full + kStages;
    float *s_x0 = reinterpret_cast<float *>(sm + 128);
    unsigned char *s_v0 = sm + 128 + size_t(kStages) * kXstage * 4;
    unsigned char *s_o0 = s_v0 + kStages * stage_val_bytes<BF16>();

    pdl_launch_dependents();
    cg::cluster_group cluster = cg::this_cluster();
    const int ksc = static_cast<int>(cluster.num_blocks());
    const int q = static_cast<int>(cluster.block_rank());
    const WorkItem item = items[blockIdx.x];
    const int ng = item.ng;   // 0: an idle rank, it only joins the cluster barriers
    const int gfirst = item.g0;
    const Group g0 = f.groups[gfirst];
    const int m = g0.m, n = g0.n, rw = g0.nib ? 1 : 2;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t b0 = int64_t(blockIdx.y) * kBt;
    const int split = kStacked ? ra.I : int(f.cols);   // first activation row of the h part
    const int J0 = item.c0 * kChunk, J1 = min(n, item.c1 * kChunk);
    // blocks per round: bounded by the activation tile and by the staged records
    const int rows_cap = kXcapB / kBt - (kStacked ? kBoxRows : 0);
    const int rb = ng > 0 ? max(1, min(rows_cap / m, (kRecCap / ng - 1) * kChunk)) : 1;
    const int rounds = ng > 0 ? (J1 - J0 + rb - 1) / rb : 0;

    if (tid == 0) {
        for (int st = 0; st < kStages; ++st) {
            mbar_init(&full[st], 1);
            mbar_init(&empty[st], kConsumers);
        }
        fence_mbar_init();
    }
    __syncthreads();

    auto round_geo = [&](int r) {
        Round g;
        g.jr0 = J0 + r * rb;
        g.jr1 = min(J1, g.jr0 + rb);
        g.cr0 = g.jr0 / kChunk;
        g.nchr = (g.jr1 + kChunk - 1) / kChunk - g.cr0;
        g.kx0 = g.jr0 * m;
        const int64_t kxe = int64_t(g.jr1) * m;
        g.kx1 = static_cast<int>(kxe < f.cols ? kxe : f.cols);
        g.kxa = min(g.kx1, split);
        g.kxb = max(g.kx0, split);
        const int rows_a = max(0, g.kxa - g.kx0);
        g.hbase = (rows_a + kBoxRows - 1) / kBoxRows * kBoxRows;
        return g;
    };
    // Round r's copies into stage st (producer lane 0).  The handle part (kept
    // values and offsets, one contiguous run per group) may go before the PDL
    // wait; the activation part only after it.  Exactly one arrival per round
    // closes full[st] together with the transferred bytes.
    auto issue = [&](int r, int st, bool handle, bool xpart) {
        const Round g = round_geo(r);
        const uint32_t bv = uint32_t(g.nchr) * kSlots * kChunk * kEsz;
        const uint32_t bo = uint32_t(g.nchr) * kSlots * rw * 4;
        const int nboxa = (max(0, g.kxa - g.kx0) + kBoxRows - 1) / kBoxRows;
        const int nboxb = (max(0, g.kx1 - g.kxb) + kBoxRows - 1) / kBoxRows;
        const uint32_t hbytes = handle ? uint32_t(ng) * (bv + bo) : 0u;
        const uint32_t xbytes = (xpart && use_tma) ? uint32_t(nboxa + nboxb) * kBoxRows * kBt * 4 : 0u;
        if (xpart) mbar_arrive_expect_tx(&full[st], hbytes + xbytes);
        else mbar_expect_tx(&full[st], hbytes);
        if (handle)
            for (int gi = 0; gi < ng; ++gi) {
                const Group gg = f.groups[gfirst + gi];
                bulk_g2s(s_v0 + st * stage_val_bytes<BF16>() + size_t(gi) * bv,
                         static_cast<const unsigned char *>(f.vals) +
                             (size_t(gg.val_off) + size_t(g.cr0) * kSlots * kChunk) * kEsz,
                         bv, &full[st]);
                bulk_g2s(s_o0 + st * kStageOffBytes + size_t(gi) * bo,
                         f.offs + gg.off_off + size_t(g.cr0) * kSlots * rw, bo, &full[st]);
            }
        if (xpart && use_tma) {
            float *s_x = s_x0 + size_t(st) * kXstage;
            for (int i = 0; i < nboxa; ++i)
                tensor2d_g2s(s_x + size_t(i) * kBoxRows * kBt, &xmap, int(b0), g.kx0 + i * kBoxRows, &full[st]);
            for (int i = 0; i < nboxb; ++i)
                tensor2d_g2s(s_x + size_t(g.hbase + i * kBoxRows) * kBt, &hmap, int(b0),
                             g.kxb - split + i * kBoxRows, &full[st]);
        }
    };
    // activation tile without tensor maps: the producer warp loads it itself
    auto load_x_plain = [&](int r, int st) {
        const Round g = round_geo(r);
        float *s_x = s_x0 + size_t(st) * kXstage;
        const int na = max(0, g.kxa - g.kx0) * kBt, nbh = max(0, g.kx1 - g.kxb) * kBt;
        for (int base = 0; base < na + nbh; base += 8 * 32) {
            float tmp[8];
            int dst[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int idx = base + u * 32 + lane;
                float v = 0.0f;
                dst[u] = -1;
                if (idx < na + nbh) {
                    const int part = idx < na ? 0 : 1;
                    const int li = part == 0 ? idx : idx - na;
                    const int kk = li / kBt, t = li % kBt;
                    const int64_t b = b0 + t;
                    dst[u] = (part == 0 ? kk : g.hbase + kk) * kBt + t;
                    if (b < batch) {
                        if constexpr (kStacked)
                            v = part == 0 ? __ldg(ra.x + int64_t(g.kx0 + kk) * ra.B + b)
                                          : __ldg(ra.h + int64_t(g.kxb - split + kk) * ra.B + b);
                        else
                            v = __ldg(X + int64_t(g.kx0 + kk) * ldx + b);
                    }
                }
                tmp[u] = v;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u)
                if (dst[u] >= 0) s_x[dst[u]] = tmp[u];
        }
        __threadfence_block();
        __syncwarp();
    };

    bool ok = true;
    int issued = 0;   // rounds whose copies were started (producer warp), for the drain below
    if (warp == kConsumers) {
        // ---------------- producer warp
        const int pre = min(rounds, kStages);
        if (early) issued = pre;
        if (early && lane == 0)
            for (int r = 0; r < pre; ++r) issue(r, r, true, false);
        pdl_wait_previous();
        for (int r = 0; r < rounds && ok; ++r) {
            const int st = r % kStages;
            if (r >= kStages) {
                // the consumers have released this stage's previous round
                ok = mbar_wait(&empty[st], ((r / kStages) - 1) & 1);
                ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
                if (!ok) break;
                if (lane == 0) fence_proxy_async_smem();
            }
            if (!use_tma) load_x_plain(r, st);
            if (lane == 0) issue(r, st, !(early && r < kStages), true);
            issued = max(issued, r + 1);
        }
        if (!ok && lane == 0) atomicOr(f.status, kStatusTimeout);
    } else {
        pdl_wait_previous();
    }

    // ---------------- consumer warps: thread = (row slot, column quads)
    const int qd = lane % LPR, rr = lane / LPR;
    float4 acc[kRptMax][kQ], acc2[kRptMax][kQ];
#pragma unroll
    for (int p = 0; p < kRptMax; ++p)
#pragma unroll
        for (int u = 0; u < kQ; ++u) acc[p][u] = acc2[p][u] = make_float4(0.f, 0.f, 0.f, 0.f);
    const int rpt = (ng * kSlots + kConsumers * kRpw - 1) / (kConsumers * kRpw);
    uint32_t valid_mask = 0u;
    // every row pass in use and no GRU split: all rows of a chunk at once
    const bool all_rows = !kSplit && rpt == kRptMax;
    if (warp < kConsumers) {
#pragma unroll
        for (int p = 0; p < kRptMax; ++p) {
            const int s = warp * kRpw + rr + p * kConsumers * kRpw;
            const int gi = s / kSlots;
            if (p < rpt && gi < ng && (s % kSlots) < f.groups[gfirst + gi].nrows) valid_mask |= 1u << p;
        }
        for (int r = 0; r < rounds && ok; ++r) {
            const int st = r % kStages;
            ok = mbar_wait(&full[st], (r / kStages) & 1);
            ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
            if (!ok) break;
            const Round g = round_geo(r);
            const float4 *sx4 = reinterpret_cast<const float4 *>(s_x0 + size_t(st) * kXstage);
            const unsigned char *s_vals = s_v0 + st * stage_val_bytes<BF16>();
            const uint32_t *s_offs = reinterpret_cast<const uint32_t *>(s_o0 + st * kStageOffBytes);
            for (int lc = 0; lc < g.nchr; ++lc) {
                const int jc = (g.cr0 + lc) * kChunk;
                // blocks of this chunk inside the round (all 8 except at the round's ends)
                const int e_lo = max(0, g.jr0 - jc), e_hi = min(kChunk, g.jr1 - jc);
                const bool whole = e_lo == 0 && e_hi == kChunk;
                if constexpr (!kSplit) {
                    if (all_rows) {
                        // a row past the set (the last pass of an odd set) repeats a
                        // row of its last group; its sums are never written
                        int rec[kRptMax];
#pragma unroll
                        for (int p = 0; p < kRptMax; ++p) {
                            const int s = warp * kRpw + rr + p * kConsumers * kRpw;
                            const int gi = min(s / kSlots, ng - 1);
                            rec[p] = (gi * g.nchr + lc) * kSlots + (s % kSlots);
                        }
                        // rows in sub-groups of kNpg, so that the values, offsets and
                        // loads in flight of a sub-group fit in registers
#pragma unroll
                        for (int p0 = 0; p0 < kRptMax; p0 += kNpg) {
#define DARB_ROWS(NIBV, WHOLEV)                                                                                 \
    chunk_rows<BF16, NIBV, WHOLEV, kStacked, kNpg, kQ, LPR>(s_vals, s_offs, rec + p0, sx4, qd, g, jc, m, kBt / 4, \
                                                           e_lo, e_hi, acc + p0)
                            if (rw == 1) {
                                if (whole) DARB_ROWS(true, true);
                                else DARB_ROWS(true, false);
                            } else {
                                if (whole) DARB_ROWS(false, true);
                                else DARB_ROWS(false, false);
                            }
#undef DARB_ROWS
                        }
                        continue;
                    }
                }
#pragma unroll
                for (int p = 0; p < kRptMax; ++p) {
                    if (valid_mask & (1u << p)) {
                        const int s = warp * kRpw + rr + p * kConsumers * kRpw;
                        const int rec = ((s / kSlots) * g.nchr + lc) * kSlots + (s % kSlots);
#define DARB_CHUNK(NIBV, WHOLEV)                                                                        \
    chunk<BF16, NIBV, WHOLEV, kStacked, kSplit, kQ, LPR>(s_vals, s_offs, rec, sx4, qd, g, jc, m, kBt / 4, \
                                                        e_lo, e_hi, split, acc[p], acc2[p])
                        if (rw == 1) {
                            if (whole) DARB_CHUNK(true, true);
                            else DARB_CHUNK(true, false);
                        } else {
                            if (whole) DARB_CHUNK(false, true);
                            else DARB_CHUNK(false, false);
                        }
#undef DARB_CHUNK
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[st]);
        }
        if (!ok && lane == 0) atomicOr(f.status, kStatusTimeout);
    }
    if (!__syncthreads_and(ok) && warp == kConsumers && lane == 0) {
        // a wait gave up: copies may still be landing in the stages.  Give the
        // last round issued into each stage a second bounded wait before the
        // stages are reused below (the sums of this call are not valid).
        for (int st = 0; st < kStages; ++st) {
            const int last = issued - 1 - ((issued - 1 - st) % kStages + kStages) % kStages;
            if (last >= 0 && last < issued) mbar_wait(&full[st], (last / kStages) & 1);
        }
    }
    __syncthreads();   // every round consumed: the stages are free for the partial sums
    // partial sums of every row slot of the set, slot-major: part[s][part][0..kBt)
    float *part = s_x0;
    float4 *part4 = reinterpret_cast<float4 *>(part);
    if (warp < kConsumers) {
#pragma unroll
        for (int p = 0; p < kRptMax; ++p) {
            const int s = warp * kRpw + rr + p * kConsumers * kRpw;
            if (p < rpt && s < ng * kSlots) {
#pragma unroll
                for (int u = 0; u < kQ; ++u) {
                    part4[(s * kParts) * (kBt / 4) + u * LPR + qd] = acc[p][u];
                    if constexpr (kSplit) part4[(s * kParts + 1) * (kBt / 4) + u * LPR + qd] = acc2[p][u];
                }
            }
        }
    }
    __syncthreads();
    if (ksc > 1) cluster.sync();
    // this rank (index qsub of the ksub ranks sharing the set, cluster ranks
    // qbase ..) finishes rows [s0, s1) of the set for the whole tile
    const int ksub = item.ksub, qsub = item.qsub, qbase = q - qsub;
    const int R = ng * kSlots;
    const int per = (R + ksub - 1) / ksub;
    const int s0 = min(R, qsub * per), s1 = min(R, s0 + per);
    for (int idx = tid; idx < (s1 - s0) * kBt * kParts; idx += kThreads) {
        const int s = s0 + idx / (kBt * kParts), pt = (idx / kBt) % kParts, t = idx % kBt;
        const int gi = s / kSlots, slot = s % kSlots;
        // every rank's partial sum requested before any is added (one round trip
        // through distributed shared memory, not one per rank), with the row's
        // map entry and its group's row count alongside
        const int pidx = (s * kParts + pt) * kBt + t;
        float pv[8];
#pragma unroll
        for (int r = 0; r < 8; ++r)
            if (r < ksub) pv[r] = (ksc > 1 ? cluster.map_shared_rank(part, qbase + r) : part)[pidx];
        const int row = f.rowmap[(gfirst + gi) * kSlots + slot];
        if (b0 + t >= batch || slot >= f.groups[gfirst + gi].nrows) continue;
        float sum = 0.0f;   // ranks in a fixed order: deterministic
#pragma unroll
        for (int r = 0; r < 8; ++r)
            if (r < ksub) sum += pv[r];
        if constexpr (MODE == kModeY) Y[int64_t(row) * ldy + b0 + t] = sum;
        else (pt == 0 ? ra.gx : ra.gh)[int64_t(row) * ra.B + b0 + t] = sum;
    }
    if constexpr (MODE != kModeY) {
        // the rows this rank finished, for the unit counts (in the free value stages)
        int *s_rows = reinterpret_cast<int *>(s_v0);
        int *s_units = s_rows + R;
        int *s_nunits = s_units + R;
        if (tid == 0) s_nunits[1] = 0;
        __syncthreads();
        for (int s = s0 + tid; s < s1; s += kThreads) {
            const int gi = s / kSlots, slot = s % kSlots;
            if (slot < f.groups[gfirst + gi].nrows)
                s_rows[atomicAdd(&s_nunits[1], 1)] = f.rowmap[(gfirst + gi) * kSlots + slot];
        }
        __syncthreads();
        const int nloc = s_nunits[1];
        const int nc = static_cast<int>(batch - b0 < kBt ? batch - b0 : kBt);
        rnn_finish<MODE>(ra, s_rows, nloc, blockIdx.y, gridDim.y, b0, nc, s_units, s_nunits);
    }
    if (ksc > 1) cluster.sync();
}

// Tensor map over a rows x `batch` fp32 matrix (row pitch ld floats) with a
// boxr x bt box; false if it cannot be described (alignment).
inline bool make_map(CUtensorMap *map, const float *A, int64_t ld, int64_t batch, int64_t rows, int bt,
                     int boxr) {
    if (A == nullptr || rows <= 0 || reinterpret_cast<uintptr_t>(A) % 16 != 0 || (ld * 4) % 16 != 0) return false;
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (enc == nullptr) return false;
    const cuuint64_t dims[2] = {cuuint64_t(batch), cuuint64_t(rows)};
    const cuuint64_t strides[1] = {cuuint64_t(ld) * 4};
    const cuuint32_t box[2] = {cuuint32_t(bt), cuuint32_t(boxr)};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(A), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Grid shape of a plain product: row-set level l (sets of up to 2^l groups)
// and cluster size C = 2^c (the work table items[l][c]).
// A CTA's work is at most item_work group-chunks, plus a fixed cost (prologue,
// reduction) of about 0.2 x nch_max group-chunks, and the launch takes
// ceil(CTAs / resident CTAs) waves, so the cost is
// waves * (item_work / nch_max + 0.2); on a tie the shape with fewer waves
// wins, then the larger sets (each staged activation row serves more rows).
template <int LPR, int CPL>
inline void grid_shape(const Format &f, int64_t tiles, int per_sm, int *level, int *split) {
    const int64_t slots = int64_t(per_sm > 0 ? per_sm : 1) * sm_count();
    double best = 1e300;
    int64_t best_waves = 0;
    *level = 0;
    *split = 0;
    for (int l = kWorkLevels - 1; l >= 0; --l) {
        if ((1 << l) > max_set_groups<LPR, CPL>()) continue;
        for (int c = kWorkSplits - 1; c >= 0; --c) {
            if (f.nitems[l][c] <= 0) continue;
            const int64_t ctas = int64_t(f.nitems[l][c]) * tiles;
            const int64_t waves = (ctas + slots - 1) / slots;
            const double cost = double(waves) * (double(f.item_work[l][c]) / double(f.nch_max) + 0.2);
            if (cost < best * (1 - 1e-9) || (cost <= best * (1 + 1e-9) && waves < best_waves)) {
                best = cost;
                best_waves = waves;
                *level = l;
                *split = c;
            }
        }
    }
}

// Grid shape of the fused RNN steps: each CTA also runs the cell epilogue
// (arrival counters, the cell of the units it completes), so fewer, larger
// CTAs win there: the largest row sets that still give two CTAs per SM with a
// split of 8, then the smallest split that reaches three CTAs per SM.
template <int LPR, int CPL>
inline void grid_shape_rnn(const Format &f, int64_t tiles, int *level, int *split) {
    const int64_t want_min = 2 * int64_t(sm_count()), target = 3 * int64_t(sm_count());
    const int cmax = kWorkSplits - 1;
    *level = 0;
    for (int l = kWorkLevels - 1; l >= 0; --l) {
        if ((1 << l) > max_set_groups<LPR, CPL>()) continue;
        *level = l;
        if (int64_t(f.nitems[l][cmax]) * tiles >= want_min) break;
    }
    *split = 0;
    while (*split < cmax && int64_t(f.nitems[*level][*split]) * tiles < target) ++*split;
}

// CTAs of one batch_kernel instantiation resident per SM (shared memory is the limit).
template <bool BF16, int LPR, int CPL, int MODE>
inline int resident_per_sm() {
    const auto fn = batch_kernel<BF16, LPR, CPL, MODE>;
    return static_cast<int>(per_device(reinterpret_cast<const void *>(fn), 0, [fn] {
        int v = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, fn, kThreads, smem_bytes<BF16>()) != cudaSuccess) {
            cudaGetLastError();
            v = 0;
        }
        return static_cast<long long>(v > 0 ? v : 1);
    }));
}

template <bool BF16, int LPR, int CPL, int MODE>
cudaError_t launch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy,
                   const RnnArgs &ra, bool early, cudaStream_t stream) {
    constexpr int kBt = LPR * CPL;
    constexpr size_t smem = smem_bytes<BF16>();
    const cudaError_t attr = allow_smem(batch_kernel<BF16, LPR, CPL, MODE>, smem);
    if (attr != cudaSuccess) return attr;
    CUtensorMap xmap, hmap;
    std::memset(&xmap, 0, sizeof xmap);
    std::memset(&hmap, 0, sizeof hmap);
    int use_tma;
    if constexpr (MODE == kModeY) {
        use_tma = make_map(&xmap, X, ldx, batch, f.cols, kBt, box_rows<LPR, CPL>()) ? 1 : 0;
    } else {
        const bool ok_x = ra.I == 0 || make_map(&xmap, ra.x, ra.B, ra.B, ra.I, kBt, box_rows<LPR, CPL>());
        const bool ok_h = make_map(&hmap, ra.h, ra.B, ra.B, ra.H, kBt, box_rows<LPR, CPL>());
        use_tma = ok_x && ok_h ? 1 : 0;
    }
    const int64_t tiles = (batch + kBt - 1) / kBt;
    int level, split;
    if constexpr (MODE == kModeY) grid_shape<LPR, CPL>(f, tiles, resident_per_sm<BF16, LPR, CPL, MODE>(), &level, &split);
    else grid_shape_rnn<LPR, CPL>(f, tiles, &level, &split);
    const dim3 grid(static_cast<unsigned>(f.nitems[level][split]), static_cast<unsigned>(tiles));
    return launch_ex(batch_kernel<BF16, LPR, CPL, MODE>, grid, dim3(kThreads), smem, stream, 1u << split, true, f,
                     f.items[level][split], X, ldx, batch, Y, ldy, xmap, hmap, ra, use_tma, early ? 1 : 0);
}

// Tile width by batch, within what one block of the largest m can stage.
template <bool BF16, int MODE>
cudaError_t launch_any(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy,
                       const RnnArgs &ra, bool early, cudaStream_t stream) {
    const bool stacked = MODE != kModeY;
    if (batch <= 16 || f.m_max > max_block<8, 4>(stacked))
        return launch<BF16, 4, 4, MODE>(f, X, ldx, batch, Y, ldy, ra, early, stream);
    // GRU keeps two accumulator sets: 8 columns per lane would not leave room
    // for a second CTA per SM
    if (batch <= 32 || MODE == kModeGru || f.m_max > max_block<8, 8>(stacked))
        return launch<BF16, 8, 4, MODE>(f, X, ldx, batch, Y, ldy, ra, early, stream);
    return launch<BF16, 8, 8, MODE>(f, X, ldx, batch, Y, ldy, ra, early, stream);
}

}  // namespace batch
}  // namespace darb
