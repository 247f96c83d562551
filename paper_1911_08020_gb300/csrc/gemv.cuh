// gemv.cuh -- y = W_darb x for a single activation column (batch 1): the
// HBM-bound, latency-bound regime of Sec. 3.2 / Fig. 6(b).
//
// One CTA per 32-row group, sixteen warps.  Warp w takes the group's chunks
// w, w + 16, ...; lane i is slot i, so a warp's load of one chunk's kept
// values (16 bytes per lane for bf16) and packed offsets is 32 contiguous
// records: HBM streams each value and offset exactly once.  The whole of x
// (cols floats) is first copied into shared memory by all threads; at block j
// the 32 lanes select x[j*m + off_i] from one window of m activations, so the
// gathers hardly conflict.  The first chunks' loads are in flight while x is
// staged -- and, when the handle's data is known to be complete (`early`),
// even before the previous kernel on the stream has finished (PDL).  Each
// lane keeps one partial sum per batch of chunks; the sixteen partial sums of
// a row meet in shared memory and are added in warp order (deterministic).
//
// Compared with the row-per-lane kernel (rowlane.cuh) it needs no cluster,
// no distributed shared memory and no per-round staging of the values.
//
// gemv_bulk_kernel is the same product with the whole group in shared memory:
// at the start one thread bulk-copies the group's values and offsets (one
// contiguous run each) and, once the previous kernel is done, x; the warps
// then read their chunks from shared memory.  Every byte of a call is in
// flight after one issue, so a call costs one round trip to HBM (the W copies
// even start while the previous kernel drains), where the register kernel
// needs one per batch of chunks plus one for x.  It is used when the largest
// group and x fit in shared memory and the arrays are 16-byte aligned.
#pragma once

#include "kernels_common.cuh"
#include "launch.cuh"
#include "tma.cuh"

namespace darb {
namespace gemv {

constexpr int kWarpsG = 16;
constexpr int kThreadsG = kWarpsG * 32;
// Chunks a lane has in flight at once.  Three keeps the kernel near 60
// registers a thread: a CTA then fits beside the CTAs of the kernel before it
// on the stream (the encoder's, say), so with PDL it starts its loads while
// that kernel drains.  Four chunks run a lone launch ~15% faster but need ~84
// registers, and the bench step (encode, then the products) came out ~3%
// slower for it.
constexpr int kBatchChunks = 3;
constexpr size_t kMaxCols = 48 * 1024;   // x in shared memory: 192 KB at most

template <bool BF16>
struct ChunkData {
    uint4 v[BF16 ? 1 : 2];   // 8 values
    uint2 o;                 // packed offsets (nibbles in .x, or bytes in .x/.y)
};

template <bool BF16>
__device__ __forceinline__ void load_chunk_rec(const Format &f, const Group &g, int c, int lane, ChunkData<BF16> &d) {
    const int64_t rec = int64_t(c) * kSlots + lane;
    if constexpr (BF16) {
        d.v[0] = __ldg(reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(f.vals) + g.val_off + rec * kChunk));
    } else {
        const uint4 *p = reinterpret_cast<const uint4 *>(static_cast<const float *>(f.vals) + g.val_off + rec * kChunk);
        d.v[0] = __ldg(p);
        d.v[1] = __ldg(p + 1);
    }
    if (g.nib) d.o = make_uint2(__ldg(f.offs + g.off_off + rec), 0u);
    else d.o = __ldg(reinterpret_cast<const uint2 *>(f.offs + g.off_off) + rec);
}

template <bool BF16>
__device__ __forceinline__ float chunk_dot(const Group &g, int c, const ChunkData<BF16> &d, const float *s_x) {
    float v[kChunk];
    if constexpr (BF16) {
        const uint32_t w[4] = {d.v[0].x, d.v[0].y, d.v[0].z, d.v[0].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            v[2 * e] = __uint_as_float(w[e] << 16);
            v[2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
        }
    } else {
        v[0] = __uint_as_float(d.v[0].x); v[1] = __uint_as_float(d.v[0].y);
        v[2] = __uint_as_float(d.v[0].z); v[3] = __uint_as_float(d.v[0].w);
        v[4] = __uint_as_float(d.v[1].x); v[5] = __uint_as_float(d.v[1].y);
        v[6] = __uint_as_float(d.v[1].z); v[7] = __uint_as_float(d.v[1].w);
    }
    const int m = g.m, n = g.n;
    const bool full = (c + 1) * kChunk <= n;
    float acc = 0.0f;
#pragma unroll
    for (int e = 0; e < kChunk; ++e) {
        const int j = c * kChunk + e;
        if (full || j < n) {
            const uint32_t o = g.nib ? (d.o.x >> (4 * e)) & 15u : ((e < 4 ? d.o.x : d.o.y) >> (8 * (e & 3))) & 255u;
            acc = fmaf(v[e], s_x[j * m + int(o)], acc);
        }
    }
    return acc;
}

template <bool BF16>
__global__ void __launch_bounds__(kThreadsG)
gemv_kernel(Format f, const float *X, int64_t ldx, float *Y, int64_t ldy, int early) {
    extern __shared__ float s_x[];   // cols floats
    __shared__ float s_part[kWarpsG][kSlots];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gi = blockIdx.x;
    const Group g = f.groups[gi];
    const int nch = (g.n + kChunk - 1) / kChunk;

    pdl_launch_dependents();
    // the first batch of this warp's chunks: the handle's data never changes
    // after encoding, so with `early` it is read before the previous kernel ends
    ChunkData<BF16> d[kBatchChunks];
    int c0 = warp;
    auto load_batch = [&](int cfirst) {
#pragma unroll
        for (int k = 0; k < kBatchChunks; ++k) {
            const int c = cfirst + k * kWarpsG;
            if (c < nch) load_chunk_rec<BF16>(f, g, c, lane, d[k]);
        }
    };
    if (early) load_batch(c0);
    pdl_wait_previous();   // x may come from the previous kernel, and Y may still be read by it
    if (!early) load_batch(c0);
    // x -> shared memory (16-byte loads when x is one aligned contiguous run)
    const int64_t cols = f.cols;
    if (ldx == 1 && (reinterpret_cast<uintptr_t>(X) & 15) == 0) {
        const int64_t nq = cols / 4;
        for (int64_t i = tid; i < nq; i += kThreadsG)
            reinterpret_cast<float4 *>(s_x)[i] = __ldg(reinterpret_cast<const float4 *>(X) + i);
        for (int64_t k = nq * 4 + tid; k < cols; k += kThreadsG) s_x[k] = __ldg(X + k);
    } else {
        for (int64_t k = tid; k < cols; k += kThreadsG) s_x[k] = __ldg(X + k * ldx);
    }
    __syncthreads();
    float acc = 0.0f;
    while (c0 < nch) {
#pragma unroll
        for (int k = 0; k < kBatchChunks; ++k) {
            const int c = c0 + k * kWarpsG;
            if (c < nch) acc += chunk_dot<BF16>(g, c, d[k], s_x);
        }
        c0 += kBatchChunks * kWarpsG;
        if (c0 < nch) load_batch(c0);
    }
    s_part[warp][lane] = acc;
    __syncthreads();
    if (warp == 0 && lane < g.nrows) {
        float s = 0.0f;
#pragma unroll
        for (int w = 0; w < kWarpsG; ++w) s += s_part[w][lane];
        Y[int64_t(f.rowmap[gi * kSlots + lane]) * ldy] = s;
    }
}

// Shared memory of gemv_bulk_kernel: [0, 128) the two mbarriers, then vcap
// bytes for a group's values, ocap for its offsets, then x.
template <bool BF16>
__global__ void __launch_bounds__(kThreadsG)
gemv_bulk_kernel(Format f, const float *X, int64_t ldx, float *Y, int64_t ldy, int early, int vcap, int ocap) {
    constexpr int kEsz = BF16 ? 2 : 4;
    extern __shared__ __align__(128) unsigned char sm[];
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm);   // [0]: values and offsets, [1]: x
    unsigned char *const s_val = sm + 128;
    uint32_t *const s_off = reinterpret_cast<uint32_t *>(s_val + vcap);
    float *const s_x = reinterpret_cast<float *>(reinterpret_cast<unsigned char *>(s_off) + ocap);
    __shared__ float s_part[kWarpsG][kSlots];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gi = blockIdx.x;
    const Group g = f.groups[gi];
    const int nch = (g.n + kChunk - 1) / kChunk;
    const uint32_t vbytes = uint32_t(nch) * kSlots * kChunk * kEsz;
    const uint32_t obytes = uint32_t(nch) * kSlots * (g.nib ? 4u : 8u);
    const int64_t cols = f.cols;
    // x in one copy when it is one aligned run of whole 16-byte units
    const bool xbulk = ldx == 1 && (reinterpret_cast<uintptr_t>(X) & 15) == 0 && (cols & 3) == 0;
    auto copy_w = [&] {
        mbar_arrive_expect_tx(&bar[0], vbytes + obytes);
        bulk_g2s(s_val, static_cast<const unsigned char *>(f.vals) + g.val_off * kEsz, vbytes, &bar[0]);
        bulk_g2s(s_off, f.offs + g.off_off, obytes, &bar[0]);
    };

    pdl_launch_dependents();
    if (tid == 0) {
        mbar_init(&bar[0], 1);
        mbar_init(&bar[1], 1);
        fence_mbar_init();
        if (early) copy_w();   // the handle's data never changes after encoding
    }
    pdl_wait_previous();   // x may come from the previous kernel, and Y may still be read by it
    if (tid == 0) {
        if (!early) copy_w();
        if (xbulk) {
            mbar_arrive_expect_tx(&bar[1], uint32_t(cols) * 4u);
            bulk_g2s(s_x, X, uint32_t(cols) * 4u, &bar[1]);
        }
    }
    if (!xbulk)
        for (int64_t k = tid; k < cols; k += kThreadsG) s_x[k] = __ldg(X + k * ldx);
    __syncthreads();   // the barriers' initialisation and the plain copy of x are seen by all threads
    const bool ok = __syncthreads_and(mbar_wait(&bar[0], 0) && (!xbulk || mbar_wait(&bar[1], 0)));
    float acc = 0.0f;
    if (ok) {
        for (int c = warp; c < nch; c += kWarpsG) {
            const int rec = c * kSlots + lane;
            ChunkData<BF16> d;
            if constexpr (BF16) {
                d.v[0] = reinterpret_cast<const uint4 *>(s_val)[rec];
            } else {
                d.v[0] = reinterpret_cast<const uint4 *>(s_val)[2 * rec];
                d.v[1] = reinterpret_cast<const uint4 *>(s_val)[2 * rec + 1];
            }
            d.o = g.nib ? make_uint2(s_off[rec], 0u) : reinterpret_cast<const uint2 *>(s_off)[rec];
            acc += chunk_dot<BF16>(g, c, d, s_x);
        }
    } else if (tid == 0) {
        // a copy did not land in time: record it, and give the copies still in
        // flight a second bounded wait before the CTA (and its shared memory) ends
        atomicOr(f.status, kStatusTimeout);
        mbar_wait(&bar[0], 0);
        if (xbulk) mbar_wait(&bar[1], 0);
    }
    s_part[warp][lane] = acc;
    __syncthreads();
    if (ok && warp == 0 && lane < g.nrows) {
        float sum = 0.0f;
#pragma unroll
        for (int w = 0; w < kWarpsG; ++w) sum += s_part[w][lane];
        Y[int64_t(f.rowmap[gi * kSlots + lane]) * ldy] = sum;
    }
}

constexpr size_t kBulkSmemLimit = 225 * 1024;   // dynamic: 227 KB a block, less the static partial sums

template <bool BF16>
cudaError_t launch(const Format &f, const float *X, int64_t ldx, float *Y, int64_t ldy, bool early,
                   cudaStream_t stream) {
    // the largest group is one of the smallest block size
    if (f.m_min > 0 && (reinterpret_cast<uintptr_t>(f.vals) & 15) == 0 &&
        (reinterpret_cast<uintptr_t>(f.offs) & 15) == 0) {
        const int64_t nch = ((f.cols + f.m_min - 1) / f.m_min + kChunk - 1) / kChunk;
        const int64_t vcap = nch * kSlots * kChunk * (BF16 ? 2 : 4);
        // any group (m >= m_min) has at most nch chunks; room for 8-byte offset
        // records, which groups of m > 16 use
        const int64_t ocap = nch * kSlots * 8;
        const int64_t smem = 128 + vcap + ocap + f.cols * 4;
        if (smem <= int64_t(kBulkSmemLimit)) {
            const cudaError_t attr = allow_smem(gemv_bulk_kernel<BF16>, kBulkSmemLimit);
            if (attr != cudaSuccess) return attr;
            return launch_ex(gemv_bulk_kernel<BF16>, dim3(static_cast<unsigned>(f.ngroups)), dim3(kThreadsG),
                             size_t(smem), stream, 1, true, f, X, ldx, Y, ldy, early ? 1 : 0, int(vcap), int(ocap));
        }
    }
    const size_t smem = size_t(f.cols) * 4;
    const cudaError_t attr = allow_smem(gemv_kernel<BF16>, kMaxCols * 4);
    if (attr != cudaSuccess) return attr;
    return launch_ex(gemv_kernel<BF16>, dim3(static_cast<unsigned>(f.ngroups)), dim3(kThreadsG), smem, stream, 1, true,
                     f, X, ldx, Y, ldy, early ? 1 : 0);
}

}  // namespace gemv
}  // namespace darb
