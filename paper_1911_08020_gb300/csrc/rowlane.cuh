// rowlane.cuh -- the row-per-lane product kernel (batch <= 4), as a template
// over its output: plain Y, or the gate sums of a fused LSTM / GRU step.
//
// A cluster of KSC CTAs works on one 32-row group (one block size m); CTA q of
// the cluster takes the q-th contiguous range of the group's chunks.  Per
// round of at most kCpr chunks, one thread starts two bulk (TMA) copies -- the
// chunks' kept values and packed offsets, contiguous in HBM -- into shared
// memory, while all threads stage the activation rows those chunks can
// select, [j*m, j*m+m) for every block j (one more bulk copy when X is one
// contiguous run).  Warps then split the round's chunks, lane i computing
// slot i from shared memory: at a given block the 32 lanes select activations
// from one window of X, so the gathers are (nearly) free of bank conflicts.
// Partial sums meet in shared memory (8 warps, fixed order) and then across
// the cluster through distributed shared memory (fixed rank order); each rank
// finishes a slice of the group's rows.
//
// The handle's values and offsets never change after encoding, so when the
// caller allows it (`early`) the first round's copies are issued before
// griddepcontrol.wait and overlap the previous kernel on the stream; X and the
// outputs are touched only after that wait.
#pragma once

#include "kernels_common.cuh"
#include "launch.cuh"
#include "rnn_epilogue.cuh"
#include "tma.cuh"

#include <cooperative_groups.h>

namespace darb {
namespace rowlane {

namespace cg = cooperative_groups;

constexpr int kCpr = 32;        // chunks per round, at most
constexpr int kXcap = 8192;     // activation floats staged per round, at most

template <bool BF16, int BT, int MODE>
__host__ __device__ constexpr size_t smem_bytes() {
    constexpr int kParts = MODE == kModeGru ? 2 : 1;
    return 128 + size_t(kCpr) * kSlots * kChunk * (BF16 ? 2 : 4) + size_t(kCpr) * kSlots * 2 * 4 +
           size_t(kXcap) * 4 + size_t(kWarps) * kSlots * BT * kParts * 4 + size_t(kSlots) * BT * kParts * 4 +
           2 * kSlots * 4 + 16;
}

// Chunks [lc_begin, lc_end) of this round for lane's slot.  SPLIT sends the
// products whose activation row is >= split into acc2 (the GRU h part).
template <bool BF16, bool NIB, int BT, bool SPLIT>
__device__ __forceinline__ void chunks(const Group &g, int rc0, int lc_begin, int lc_end, int lane, int k0,
                                       int split, const unsigned char *s_vals, const uint32_t *s_offs,
                                       const float *s_x, float (&acc)[BT], float (&acc2)[BT]) {
    const int m = g.m, n = g.n;
    for (int lc = lc_begin; lc < lc_end; ++lc) {
        float v[kChunk];
        const int rec = lc * kSlots + lane;
        if constexpr (BF16) {
            const uint4 q = *reinterpret_cast<const uint4 *>(s_vals + size_t(rec) * 16);
            const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                v[2 * e] = __uint_as_float(w[e] << 16);
                v[2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
            }
        } else {
            const float4 *p = reinterpret_cast<const float4 *>(s_vals + size_t(rec) * 32);
            const float4 a = p[0], b = p[1];
            v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
            v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
        }
        uint2 ow;
        if constexpr (NIB) ow = make_uint2(s_offs[rec], 0u);
        else ow = reinterpret_cast<const uint2 *>(s_offs)[rec];
        const int c = rc0 + lc;
        const bool full = (c + 1) * kChunk <= n;
#pragma unroll
        for (int e = 0; e < kChunk; ++e) {
            const int j = c * kChunk + e;
            if (full || j < n) {
                const int kg = j * m + unpack_offset<NIB>(ow, e);
                const int k = kg - k0;
                if (!SPLIT || kg < split) {
#pragma unroll
                    for (int t = 0; t < BT; ++t) acc[t] = fmaf(v[e], s_x[k * BT + t], acc[t]);
                } else {
#pragma unroll
                    for (int t = 0; t < BT; ++t) acc2[t] = fmaf(v[e], s_x[k * BT + t], acc2[t]);
                }
            }
        }
    }
}

template <bool BF16, int BT, int MODE>
__global__ void __launch_bounds__(kWarps * 32)
rowlane_kernel(Format f, const float *__restrict__ X, int64_t ldx, int64_t batch, float *__restrict__ Y, int64_t ldy,
       RnnArgs ra, int early, int x_contig) {
    constexpr int kEsz = BF16 ? 2 : 4;
    constexpr int kParts = MODE == kModeGru ? 2 : 1;
    constexpr int kPb = BT * kParts;   // partial sums per slot
    extern __shared__ __align__(128) unsigned char sm[];
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm);
    unsigned char *s_vals = sm + 128;
    uint32_t *s_offs = reinterpret_cast<uint32_t *>(s_vals + size_t(kCpr) * kSlots * kChunk * kEsz);
    float *s_x = reinterpret_cast<float *>(s_offs + size_t(kCpr) * kSlots * 2);
    float *s_red = s_x + kXcap;
    float *s_part = s_red + kWarps * kSlots * kPb;
    int *s_rows = reinterpret_cast<int *>(s_part + kSlots * kPb);
    int *s_units = s_rows + kSlots;
    int *s_nunits = s_units + kSlots;

    pdl_launch_dependents();
    cg::cluster_group cluster = cg::this_cluster();
    const int ksc = static_cast<int>(cluster.num_blocks());
    const int q = static_cast<int>(cluster.block_rank());
    const int gi = blockIdx.x / ksc;
    const Group g = f.groups[gi];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int m = g.m;
    const int nch = (g.n + kChunk - 1) / kChunk;
    const int cpc = (nch + ksc - 1) / ksc;
    const int c0 = min(nch, q * cpc), c1 = min(nch, c0 + cpc);
    const int cpr = max(1, min(kCpr, kXcap / (kChunk * m * BT)));
    const int rw = g.nib ? 1 : 2;   // offset record words
    const unsigned char *vals_g = static_cast<const unsigned char *>(f.vals) + size_t(g.val_off) * kEsz;
    const uint32_t *offs_g = f.offs + g.off_off;
    const int nb = batch < BT ? static_cast<int>(batch) : BT;
    const int split = MODE == kModeY ? int(f.cols) : ra.I;   // first row of the h part

    if (tid == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    __syncthreads();
    // Round r's copies all complete one phase of `bar`: the handle's values and
    // offsets (issued before the PDL wait when `early`), plus the activation
    // slice when it is one contiguous, 16-byte aligned run of X.
    auto issue_handle = [&](int rc0, int rc1) {
        const uint32_t bv = uint32_t(rc1 - rc0) * kSlots * kChunk * kEsz;
        const uint32_t bo = uint32_t(rc1 - rc0) * kSlots * rw * 4;
        mbar_expect_tx(bar, bv + bo);
        bulk_g2s(s_vals, vals_g + size_t(rc0) * kSlots * kChunk * kEsz, bv, bar);
        bulk_g2s(s_offs, offs_g + size_t(rc0) * kSlots * rw, bo, bar);
    };
    const int rounds = (c1 - c0 + cpr - 1) / cpr;
    if (early && rounds > 0 && tid == 0) issue_handle(c0, min(c1, c0 + cpr));
    pdl_wait_previous();

    float acc[BT], acc2[BT];
#pragma unroll
    for (int t = 0; t < BT; ++t) acc[t] = acc2[t] = 0.0f;
    bool ok = true;
    int r_fail = 0;
    for (int r = 0; r < rounds && ok; ++r) {
        r_fail = r;
        const int rc0 = c0 + r * cpr, rc1 = min(c1, rc0 + cpr);
        const int k0 = rc0 * kChunk * m;
        const int64_t kend = int64_t(rc1) * kChunk * m;
        const int k1 = static_cast<int>(kend < f.cols ? kend : f.cols);
        const int nx = (k1 - k0) * BT;
        // contiguous X: the slice is X[k0*BT .. k1*BT); bulk-copy its 16-byte
        // multiple (k0 is a multiple of 8, so the start is aligned), load the rest
        const int nbulk = (MODE == kModeY && x_contig) ? (nx & ~3) : 0;
        if (tid == 0) {
            if (r > 0) fence_proxy_async_smem();   // last round's generic reads before async writes
            if (!(early && r == 0)) issue_handle(rc0, rc1);
            mbar_arrive_expect_tx(bar, uint32_t(nbulk) * 4);
            if (nbulk > 0) bulk_g2s(s_x, X + int64_t(k0) * BT, uint32_t(nbulk) * 4, bar);
        }
        if (MODE == kModeY && x_contig) {
            for (int idx = nbulk + tid; idx < nx; idx += kWarps * 32) s_x[idx] = __ldg(X + int64_t(k0) * BT + idx);
        } else {
            // strided X or the stacked RNN input: 8 independent loads in flight per thread
            for (int base = 0; base < nx; base += 8 * kWarps * 32) {
                float tmp[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int idx = base + u * kWarps * 32 + tid;
                    const int k = k0 + idx / BT, t = idx % BT;
                    float v = 0.0f;
                    if (idx < nx && t < nb) {
                        if constexpr (MODE == kModeY) v = __ldg(X + int64_t(k) * ldx + t);
                        else v = k < ra.I ? __ldg(ra.x + int64_t(k) * ra.B + t) : __ldg(ra.h + int64_t(k - ra.I) * ra.B + t);
                    }
                    tmp[u] = v;
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int idx = base + u * kWarps * 32 + tid;
                    if (idx < nx) s_x[idx] = tmp[u];
                }
            }
        }
        __syncthreads();
        ok = __syncthreads_and(mbar_wait(bar, r & 1));
        if (ok && lane < g.nrows) {
            const int nrc = rc1 - rc0, cpw = (nrc + kWarps - 1) / kWarps;
            const int lb = min(nrc, warp * cpw), le = min(nrc, lb + cpw);
            constexpr bool kSplit = MODE == kModeGru;
            if (g.nib)
                chunks<BF16, true, BT, kSplit>(g, rc0, lb, le, lane, k0, split, s_vals, s_offs, s_x, acc, acc2);
            else
                chunks<BF16, false, BT, kSplit>(g, rc0, lb, le, lane, k0, split, s_vals, s_offs, s_x, acc, acc2);
        }
        __syncthreads();
    }
    if (!ok) {
        // a copy did not land in time: record it, give in-flight copies one more
        // bounded wait, and finish without trusting the sums
        if (tid == 0) atomicOr(f.status, kStatusTimeout);
        mbar_wait(bar, r_fail & 1);
    }
#pragma unroll
    for (int t = 0; t < BT; ++t) {
        s_red[(warp * kSlots + lane) * kPb + t] = acc[t];
        if constexpr (kParts == 2) s_red[(warp * kSlots + lane) * kPb + BT + t] = acc2[t];
    }
    __syncthreads();
    if (warp == 0) {
#pragma unroll
        for (int t = 0; t < kPb; ++t) {
            float s = s_red[lane * kPb + t];
#pragma unroll
            for (int w = 1; w < kWarps; ++w) s += s_red[(w * kSlots + lane) * kPb + t];
            s_part[lane * kPb + t] = s;
        }
    }
    if (ksc > 1) cluster.sync();
    else __syncthreads();
    // rank q finishes slots [s0, s1) of the group, adding the ranks in a fixed order
    const int per = (kSlots + ksc - 1) / ksc;
    const int s0 = min(g.nrows, q * per), s1 = min(g.nrows, s0 + per);
    for (int idx = tid; idx < (s1 - s0) * kPb; idx += kWarps * 32) {
        const int slot = s0 + idx / kPb, t = idx % kPb;
        // every rank's partial sum requested before any is added: one round trip
        // through distributed shared memory, not one per rank
        float pv[8];
#pragma unroll
        for (int r = 0; r < 8; ++r)
            if (r < ksc) pv[r] = (ksc > 1 ? cluster.map_shared_rank(s_part, r) : s_part)[slot * kPb + t];
        const int row = f.rowmap[gi * kSlots + slot];
        float s = 0.0f;
#pragma unroll
        for (int r = 0; r < 8; ++r)
            if (r < ksc) s += pv[r];
        if constexpr (MODE == kModeY) {
            if (t < nb) Y[int64_t(row) * ldy + t] = s;
        } else {
            const int tt = t % BT;
            if (tt < nb) (t < BT ? ra.gx : ra.gh)[int64_t(row) * ra.B + tt] = s;
        }
    }
    if constexpr (MODE != kModeY) {
        for (int i = tid; i < s1 - s0; i += kWarps * 32) s_rows[i] = f.rowmap[gi * kSlots + s0 + i];
        __syncthreads();
        rnn_finish<MODE>(ra, s_rows, s1 - s0, 0, 1, 0, nb, s_units, s_nunits);
    }
    if (ksc > 1) cluster.sync();
}

// Cluster size: split each group over up to 8 CTAs, but keep the grid within
// about two CTAs per SM so that it runs in one wave and leaves room for the
// next kernel's prologue (PDL).
inline unsigned cluster_size(const Format &f) {
    unsigned ksc = 1;
    while (ksc < 8 && int64_t(f.ngroups) * ksc * 2 <= 2 * int64_t(sm_count())) ksc *= 2;
    return ksc;
}

template <bool BF16, int BT, int MODE>
cudaError_t launch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy,
                   const RnnArgs &ra, bool early, cudaStream_t stream) {
    constexpr size_t smem = smem_bytes<BF16, BT, MODE>();
    const cudaError_t attr = allow_smem(rowlane_kernel<BF16, BT, MODE>, smem);
    if (attr != cudaSuccess) return attr;
    const unsigned ksc = cluster_size(f);
    const dim3 grid(static_cast<unsigned>(f.ngroups) * ksc);
    // X rows are the slice's BT-wide rows back to back: one bulk copy per round
    const int x_contig = (MODE == kModeY && batch == BT && ldx == BT && reinterpret_cast<uintptr_t>(X) % 16 == 0) ? 1 : 0;
    return launch_ex(rowlane_kernel<BF16, BT, MODE>, grid, dim3(kWarps * 32), smem, stream, ksc, true, f, X, ldx, batch,
                     Y, ldy, ra, early ? 1 : 0, x_contig);
}

// Batch 1, 2 or 3-4 columns.
template <bool BF16, int MODE>
cudaError_t launch_any(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy,
                       const RnnArgs &ra, bool early, cudaStream_t stream) {
    if (batch == 1) return launch<BF16, 1, MODE>(f, X, ldx, batch, Y, ldy, ra, early, stream);
    if (batch == 2) return launch<BF16, 2, MODE>(f, X, ldx, batch, Y, ldy, ra, early, stream);
    return launch<BF16, 4, MODE>(f, X, ldx, batch, Y, ldy, ra, early, stream);
}

}  // namespace rowlane
}  // namespace darb
