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

namespace darb {
namespace {

template <bool BF16, int BT>
__global__ void __launch_bounds__(kWarps * 32)
spmm_rowlane(Format f, XPlain xs, int64_t batch, float *Y, int64_t ldy) {
    __shared__ float red[kWarps][kSlots][BT];
    const int gi = blockIdx.x;
    const Group g = f.groups[gi];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t b0 = static_cast<int64_t>(blockIdx.y) * BT;
    const int nb = batch - b0 < BT ? static_cast<int>(batch - b0) : BT;
    const int nch = (g.n + kChunk - 1) / kChunk;
    const int cpw = (nch + kWarps - 1) / kWarps;
    const int c_begin = min(nch, warp * cpw), c_end = min(nch, c_begin + cpw);
    float acc[BT], acc2[BT];
#pragma unroll
    for (int t = 0; t < BT; ++t) acc[t] = acc2[t] = 0.0f;
    if (lane < g.nrows) {
        if (g.nib)
            rowlane_accumulate<BF16, true, BT, false>(f, g, lane, c_begin, c_end, xs, b0, nb, acc, acc2);
        else
            rowlane_accumulate<BF16, false, BT, false>(f, g, lane, c_begin, c_end, xs, b0, nb, acc, acc2);
    }
#pragma unroll
    for (int t = 0; t < BT; ++t) red[warp][lane][t] = acc[t];
    __syncthreads();
    if (warp == 0 && lane < g.nrows) {
        const int row = f.rowmap[gi * kSlots + lane];
        float *yr = Y + static_cast<int64_t>(row) * ldy + b0;
#pragma unroll
        for (int t = 0; t < BT; ++t) {
            float s = red[0][lane][t];
#pragma unroll
            for (int w = 1; w < kWarps; ++w) s += red[w][lane][t];
            if (t < nb) yr[t] = s;
        }
    }
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

template <bool BF16>
cudaError_t launch_rowlane(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                           int64_t ldy, cudaStream_t stream) {
    XPlain xs{X, ldx};
    const dim3 block(kWarps * 32);
    const unsigned ng = static_cast<unsigned>(f.ngroups);
    if (batch == 1) {
        spmm_rowlane<BF16, 1><<<dim3(ng, 1), block, 0, stream>>>(f, xs, batch, Y, ldy);
    } else if (batch == 2) {
        spmm_rowlane<BF16, 2><<<dim3(ng, 1), block, 0, stream>>>(f, xs, batch, Y, ldy);
    } else if (batch <= 4) {
        spmm_rowlane<BF16, 4><<<dim3(ng, 1), block, 0, stream>>>(f, xs, batch, Y, ldy);
    } else {
        const unsigned tiles = static_cast<unsigned>((batch + 7) / 8);
        spmm_rowlane<BF16, 8><<<dim3(ng, tiles), block, 0, stream>>>(f, xs, batch, Y, ldy);
    }
    return cudaGetLastError();
}

template <bool BF16>
cudaError_t launch_batchlane(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                             int64_t ldy, cudaStream_t stream) {
    const bool vec = (reinterpret_cast<uintptr_t>(X) % 16 == 0) && (ldx % 4 == 0);
    const dim3 block(kWarps * 32);
    const unsigned ng = static_cast<unsigned>(f.ngroups);
    const int64_t q = (batch + 3) / 4;   // 4-column lane slices needed
    if (q <= 4) {
        spmm_batchlane<BF16, 4><<<dim3(ng, 1), block, 0, stream>>>(f, X, ldx, batch, Y, ldy, vec);
    } else if (q <= 8) {
        spmm_batchlane<BF16, 8><<<dim3(ng, 1), block, 0, stream>>>(f, X, ldx, batch, Y, ldy, vec);
    } else if (q <= 16) {
        spmm_batchlane<BF16, 16><<<dim3(ng, 1), block, 0, stream>>>(f, X, ldx, batch, Y, ldy, vec);
    } else {
        const unsigned tiles = static_cast<unsigned>((q + 31) / 32);
        spmm_batchlane<BF16, 32><<<dim3(ng, tiles), block, 0, stream>>>(f, X, ldx, batch, Y, ldy, vec);
    }
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_spmm(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                        int64_t ldy, cudaStream_t stream) {
    if (batch <= 8)
        return f.bf16 ? launch_rowlane<true>(f, X, ldx, batch, Y, ldy, stream)
                      : launch_rowlane<false>(f, X, ldx, batch, Y, ldy, stream);
    return f.bf16 ? launch_batchlane<true>(f, X, ldx, batch, Y, ldy, stream)
                  : launch_batchlane<false>(f, X, ldx, batch, Y, ldy, stream);
}

}  // namespace darb
