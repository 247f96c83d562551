// spmm.cu -- y = W_darb X on the GPU (Sec. 3.2, Fig. 6(b)), batch <= 4.
//
// Row per lane: lane i of every warp owns slot i of a 32-row group and keeps
// one accumulator per batch column.  At a given block j the 32 lanes select
// activations from one window [j*m, j*m+m) of X, so the gathers from the
// staged slice are (nearly) free of bank conflicts, and the values and
// offsets stream from HBM exactly once: the HBM-bound regime.  Batch > 4 goes
// to spmm_batch.cu.  Both accumulate in fp32, add partial sums in a fixed order
// (results are deterministic) and write every output element exactly once.
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

}  // namespace

cudaError_t launch_spmm(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                        int64_t ldy, bool early, cudaStream_t stream) {
    if (batch <= 4)
        return f.bf16 ? launch_small_batch<true>(f, X, ldx, batch, Y, ldy, early, stream)
                      : launch_small_batch<false>(f, X, ldx, batch, Y, ldy, early, stream);
    return launch_spmm_batch(f, X, ldx, batch, Y, ldy, early, stream);
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
