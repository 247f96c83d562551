// spmm.cu -- y = W_darb X on the GPU (Sec. 3.2, Fig. 6(b)).
//
// Two kernels, chosen by batch width:
//
//  * row-per-lane (batch <= 8): lane i of every warp owns slot i of a 32-row
//    group and keeps BT accumulators; the 8 warps of a CTA split the group's
//    chunks and add their partial sums in shared memory in a fixed order.  The
//    32 lanes gather activations from one window [j*m, j*m+m) at a time, so
//    the L1 serves a whole warp's gather with one or two line reads.  This is
//    the HBM-bound regime: values and offsets stream once at 16 bytes per lane.
//
//  * batch-per-lane (batch > 8): LPR lanes share one row and each owns 4
//    consecutive batch columns, so a gather is one contiguous 16*LPR-byte read
//    of an activation row, and each kept value is reused across the 4*LPR
//    columns held in registers.  Every thread walks its rows' blocks in order;
//    with fewer than 8 lanes per row the CTA's extra warps take a second half
//    of the blocks and the halves are added in shared memory.
//
// Both kernels accumulate in fp32, add partial sums in a fixed order (results
// are deterministic), and write every output element exactly once.
#include "kernels_common.cuh"
#include "launch.cuh"
#include "tma.cuh"

#include <cooperative_groups.h>

namespace cg = cooperative_groups;

namespace darb {
namespace {

// ---------------------------------------------------------------------------
// Row-per-lane kernel with a cluster split of the blocks (batch <= 4).
//
// A cluster of KSC CTAs works on one 32-row group; CTA q of the cluster takes
// the q-th contiguous range of the group's chunks.  Per round of at most kCpr
// chunks, one thread starts two bulk (TMA) copies -- the chunks' kept values
// and packed offsets, contiguous in HBM -- into shared memory, while all
// threads stage the activation rows those chunks can select, [j*m, j*m+m) for
// every block j, with coalesced loads.  Warps then split the round's chunks,
// lane i computing slot i from shared memory.  Partial sums meet first in
// shared memory (8 warps, fixed order) and then across the cluster through
// distributed shared memory (fixed rank order), and CTA 0 of the cluster
// writes Y.
//
// The handle's values and offsets never change after encoding, so when the
// caller allows it (`early`) the first round's copies are issued before
// griddepcontrol.wait and overlap the previous kernel on the stream; X and Y
// are touched only after that wait.
constexpr int kCpr = 32;        // chunks per round, at most
constexpr int kXcap = 8192;     // activation floats staged per round, at most

template <bool BF16, int BT>
__host__ __device__ constexpr size_t rowlane2_smem() {
    return 128 + size_t(kCpr) * kSlots * kChunk * (BF16 ? 2 : 4) + size_t(kCpr) * kSlots * 2 * 4 +
           size_t(kXcap) * 4 + size_t(kWarps) * kSlots * BT * 4 + size_t(kSlots) * BT * 4;
}

template <bool BF16, bool NIB, int BT>
__device__ __forceinline__ void rowlane2_chunks(const Group &g, int rc0, int lc_begin, int lc_end,
                                                int lane, int k0, const unsigned char *s_vals,
                                                const uint32_t *s_offs, const float *s_x,
                                                float (&acc)[BT]) {
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
                const int k = j * m + unpack_offset<NIB>(ow, e) - k0;
#pragma unroll
                for (int t = 0; t < BT; ++t) acc[t] = fmaf(v[e], s_x[k * BT + t], acc[t]);
            }
        }
    }
}

template <bool BF16, int BT>
__global__ void __launch_bounds__(kWarps * 32)
spmm_rowlane2(Format f, const float *__restrict__ X, int64_t ldx, int64_t batch,
              float *__restrict__ Y, int64_t ldy, int early, int x_contig) {
    extern __shared__ __align__(128) unsigned char sm[];
    constexpr int kEsz = BF16 ? 2 : 4;
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm);
    unsigned char *s_vals = sm + 128;
    uint32_t *s_offs = reinterpret_cast<uint32_t *>(s_vals + size_t(kCpr) * kSlots * kChunk * kEsz);
    float *s_x = reinterpret_cast<float *>(s_offs + size_t(kCpr) * kSlots * 2);
    float *s_red = s_x + kXcap;
    float *s_part = s_red + kWarps * kSlots * BT;

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
    const unsigned char *vals_g =
        static_cast<const unsigned char *>(f.vals) + size_t(g.val_off) * kEsz;
    const uint32_t *offs_g = f.offs + g.off_off;
    const int64_t b0 = 0;
    const int nb = batch < BT ? static_cast<int>(batch) : BT;

    if (tid == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    __syncthreads();
    // Round r's copies all complete one phase of `bar`: the handle's values and
    // offsets (issued before the PDL wait when `early`), plus the activation
    // slice when it is one contiguous, 16-byte aligned run of X.
    auto issue_handle = [&](int rc0, int rc1, bool arrive) {
        const uint32_t bv = uint32_t(rc1 - rc0) * kSlots * kChunk * kEsz;
        const uint32_t bo = uint32_t(rc1 - rc0) * kSlots * rw * 4;
        if (arrive) mbar_arrive_expect_tx(bar, bv + bo);
        else mbar_expect_tx(bar, bv + bo);
        bulk_g2s(s_vals, vals_g + size_t(rc0) * kSlots * kChunk * kEsz, bv, bar);
        bulk_g2s(s_offs, offs_g + size_t(rc0) * kSlots * rw, bo, bar);
    };
    const int rounds = (c1 - c0 + cpr - 1) / cpr;
    if (early && rounds > 0 && tid == 0) issue_handle(c0, min(c1, c0 + cpr), false);
    pdl_wait_previous();

    float acc[BT];
#pragma unroll
    for (int t = 0; t < BT; ++t) acc[t] = 0.0f;
    bool ok = true;
    int r_fail = 0;
    for (int r = 0; r < rounds && ok; ++r) {
        r_fail = r;
        const int rc0 = c0 + r * cpr, rc1 = min(c1, rc0 + cpr);
        const int k0 = rc0 * kChunk * m;
        const int64_t kend = int64_t(rc1) * kChunk * m;
        const int k1 = static_cast<int>(kend < f.cols ? kend : f.cols);
        const int nx = (k1 - k0) * BT;
        // contiguous: the slice is X[k0*BT .. k1*BT); bulk-copy its 16-byte
        // multiple (k0 is a multiple of 8, so the start is aligned), load the rest
        const int nbulk = x_contig ? (nx & ~3) : 0;
        if (tid == 0) {
            if (r > 0) fence_proxy_async_smem();   // last round's generic reads before async writes
            if (!(early && r == 0)) issue_handle(rc0, rc1, false);
            mbar_arrive_expect_tx(bar, uint32_t(nbulk) * 4);
            if (nbulk > 0) bulk_g2s(s_x, X + int64_t(k0) * BT, uint32_t(nbulk) * 4, bar);
        }
        if (x_contig) {
            for (int idx = nbulk + tid; idx < nx; idx += kWarps * 32) s_x[idx] = __ldg(X + int64_t(k0) * BT + idx);
        } else {
            // strided X: 8 independent loads in flight per thread
            for (int base = 0; base < nx; base += 8 * kWarps * 32) {
                float tmp[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int idx = base + u * kWarps * 32 + tid;
                    const int kk = idx / BT, t = idx % BT;
                    tmp[u] = (idx < nx && t < nb) ? __ldg(X + int64_t(k0 + kk) * ldx + b0 + t) : 0.0f;
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
            if (g.nib)
                rowlane2_chunks<BF16, true, BT>(g, rc0, lb, le, lane, k0, s_vals, s_offs, s_x, acc);
            else
                rowlane2_chunks<BF16, false, BT>(g, rc0, lb, le, lane, k0, s_vals, s_offs, s_x, acc);
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
    for (int t = 0; t < BT; ++t) s_red[(warp * kSlots + lane) * BT + t] = acc[t];
    __syncthreads();
    if (warp == 0) {
#pragma unroll
        for (int t = 0; t < BT; ++t) {
            float s = s_red[lane * BT + t];
#pragma unroll
            for (int w = 1; w < kWarps; ++w) s += s_red[(w * kSlots + lane) * BT + t];
            s_part[lane * BT + t] = s;
        }
    }
    if (ksc > 1) cluster.sync();
    if (q == 0 && warp == 0 && lane < g.nrows) {
        const int row = f.rowmap[gi * kSlots + lane];
        float *yr = Y + int64_t(row) * ldy + b0;
#pragma unroll
        for (int t = 0; t < BT; ++t) {
            float s = s_part[lane * BT + t];
            for (int r = 1; r < ksc; ++r) s += cluster.map_shared_rank(s_part, r)[lane * BT + t];
            if (t < nb) yr[t] = s;
        }
    }
    if (ksc > 1) cluster.sync();
}

__device__ __forceinline__ float4 load_x4(const float *p, int nb, bool vec) {
    if (vec && nb >= 4) return __ldg(reinterpret_cast<const float4 *>(p));
    float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
    if (nb > 0) r.x = __ldg(p);
    if (nb > 1) r.y = __ldg(p + 1);
    if (nb > 2) r.z = __ldg(p + 2);
    if (nb > 3) r.w = __ldg(p + 3);
    return r;
}

__device__ __forceinline__ void store_y4(float *p, float4 v, int nb) {
    if (nb > 0) p[0] = v.x;
    if (nb > 1) p[1] = v.y;
    if (nb > 2) p[2] = v.z;
    if (nb > 3) p[3] = v.w;
}

template <bool BF16, bool NIB, int LPR>
__device__ __forceinline__ float4 batchlane_accumulate(const Format &f, const Group &g, int slot,
                                                       int c_begin, int c_end, const float *xb,
                                                       int64_t ldx, int nb, bool vec) {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    const int m = g.m, n = g.n;
    for (int c = c_begin; c < c_end; ++c) {
        float v[kChunk];
        load_chunk<BF16>(f.vals, g.val_off + (static_cast<int64_t>(c) * kSlots + slot) * kChunk, v);
        const uint2 ow = load_offsets<NIB>(f.offs + g.off_off, static_cast<int64_t>(c) * kSlots + slot);
        const bool full = (c + 1) * kChunk <= n;
#pragma unroll
        for (int e = 0; e < kChunk; ++e) {
            const int j = c * kChunk + e;
            if (full || j < n) {
                const int k = j * m + unpack_offset<NIB>(ow, e);
                const float4 xv = load_x4(xb + static_cast<int64_t>(k) * ldx, nb, vec);
                acc.x = fmaf(v[e], xv.x, acc.x);
                acc.y = fmaf(v[e], xv.y, acc.y);
                acc.z = fmaf(v[e], xv.z, acc.z);
                acc.w = fmaf(v[e], xv.w, acc.w);
            }
        }
    }
    return acc;
}

template <bool BF16, int LPR>
__global__ void __launch_bounds__(kWarps * 32)
spmm_batchlane(Format f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy,
               bool vec) {
    constexpr int kRpw = 32 / LPR;                  // rows per warp at a time
    constexpr int kPar = kWarps * kRpw;             // row slots worked at a time by the CTA
    constexpr int kKs = kPar > kSlots ? kPar / kSlots : 1;       // block-range splits
    constexpr int kPasses = kPar < kSlots ? kSlots / kPar : 1;   // rows per thread
    __shared__ float4 red[kKs][kSlots][LPR];
    pdl_launch_dependents();
    pdl_wait_previous();
    const int gi = blockIdx.x;
    const Group g = f.groups[gi];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int q = lane % LPR;
    const int s = warp * kRpw + lane / LPR;
    const int ks = s / kSlots;
    const int slot0 = s % kSlots;
    const int64_t b = static_cast<int64_t>(blockIdx.y) * (4 * LPR) + 4 * q;
    const int nb = batch - b >= 4 ? 4 : (batch - b > 0 ? static_cast<int>(batch - b) : 0);
    const int nch = (g.n + kChunk - 1) / kChunk;
    const int cps = (nch + kKs - 1) / kKs;
    const int c_begin = min(nch, ks * cps), c_end = min(nch, c_begin + cps);
#pragma unroll 1
    for (int p = 0; p < kPasses; ++p) {
        const int slot = slot0 + p * kPar;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        if (slot < g.nrows && nb > 0) {
            acc = g.nib ? batchlane_accumulate<BF16, true, LPR>(f, g, slot, c_begin, c_end, X + b, ldx, nb, vec)
                        : batchlane_accumulate<BF16, false, LPR>(f, g, slot, c_begin, c_end, X + b, ldx, nb, vec);
        }
        if constexpr (kKs == 1) {
            if (slot < g.nrows && nb > 0) {
                const int row = f.rowmap[gi * kSlots + slot];
                store_y4(Y + static_cast<int64_t>(row) * ldy + b, acc, nb);
            }
        } else {
            red[ks][slot][q] = acc;
        }
    }
    if constexpr (kKs > 1) {
        __syncthreads();
        if (ks == 0 && slot0 < g.nrows && nb > 0) {
            float4 a = red[0][slot0][q];
#pragma unroll
            for (int w = 1; w < kKs; ++w) {
                const float4 o = red[w][slot0][q];
                a.x += o.x; a.y += o.y; a.z += o.z; a.w += o.w;
            }
            const int row = f.rowmap[gi * kSlots + slot0];
            store_y4(Y + static_cast<int64_t>(row) * ldy + b, a, nb);
        }
    }
}

template <bool BF16, int BT>
cudaError_t launch_rowlane2(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                            int64_t ldy, bool early, cudaStream_t stream) {
    constexpr size_t smem = rowlane2_smem<BF16, BT>();
    static const cudaError_t attr = allow_smem(spmm_rowlane2<BF16, BT>, smem);
    if (attr != cudaSuccess) return attr;
    // split each group over up to 8 CTAs, but keep the grid within about two
    // CTAs per SM so that it runs in one wave and leaves room for the next
    // kernel's prologue (PDL)
    unsigned ksc = 1;
    while (ksc < 8 && int64_t(f.ngroups) * ksc * 2 <= 2 * int64_t(sm_count())) ksc *= 2;
    const dim3 grid(static_cast<unsigned>(f.ngroups) * ksc);
    // X rows are the slice's BT-wide rows back to back: one bulk copy per round
    const int x_contig = (batch == BT && ldx == BT && reinterpret_cast<uintptr_t>(X) % 16 == 0) ? 1 : 0;
    return launch_ex(spmm_rowlane2<BF16, BT>, grid, dim3(kWarps * 32), smem, stream, ksc, true, f, X,
                     ldx, batch, Y, ldy, early ? 1 : 0, x_contig);
}

template <bool BF16>
cudaError_t launch_small_batch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                               int64_t ldy, bool early, cudaStream_t stream) {
    if (batch == 1) return launch_rowlane2<BF16, 1>(f, X, ldx, batch, Y, ldy, early, stream);
    if (batch == 2) return launch_rowlane2<BF16, 2>(f, X, ldx, batch, Y, ldy, early, stream);
    return launch_rowlane2<BF16, 4>(f, X, ldx, batch, Y, ldy, early, stream);
}

template <bool BF16>
cudaError_t launch_batchlane(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                             int64_t ldy, cudaStream_t stream) {
    const bool vec = (reinterpret_cast<uintptr_t>(X) % 16 == 0) && (ldx % 4 == 0);
    const dim3 block(kWarps * 32);
    const unsigned ng = static_cast<unsigned>(f.ngroups);
    const int64_t q = (batch + 3) / 4;   // 4-column lane slices needed
    if (q <= 4)
        return launch_ex(spmm_batchlane<BF16, 4>, dim3(ng, 1), block, 0, stream, 1, true, f, X, ldx, batch, Y, ldy, vec);
    if (q <= 8)
        return launch_ex(spmm_batchlane<BF16, 8>, dim3(ng, 1), block, 0, stream, 1, true, f, X, ldx, batch, Y, ldy, vec);
    if (q <= 16)
        return launch_ex(spmm_batchlane<BF16, 16>, dim3(ng, 1), block, 0, stream, 1, true, f, X, ldx, batch, Y, ldy, vec);
    const unsigned tiles = static_cast<unsigned>((q + 31) / 32);
    return launch_ex(spmm_batchlane<BF16, 32>, dim3(ng, tiles), block, 0, stream, 1, true, f, X, ldx, batch, Y, ldy, vec);
}

}  // namespace

cudaError_t launch_spmm(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                        int64_t ldy, bool early, cudaStream_t stream) {
    if (batch <= 4)
        return f.bf16 ? launch_small_batch<true>(f, X, ldx, batch, Y, ldy, early, stream)
                      : launch_small_batch<false>(f, X, ldx, batch, Y, ldy, early, stream);
    return f.bf16 ? launch_batchlane<true>(f, X, ldx, batch, Y, ldy, stream)
                  : launch_batchlane<false>(f, X, ldx, batch, Y, ldy, stream);
}

int sm_count() {
    static int n = [] {
        int dev = 0, v = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
            cudaGetLastError();
            return 148;
        }
        return v;
    }();
    return n;
}

}  // namespace darb
