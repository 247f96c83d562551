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

#include <type_traits>

#include "kernels_common.cuh"
#include "launch.cuh"
#include "tma.cuh"

namespace darb {
namespace gemv {

constexpr int kWarpsG = 16;
constexpr int kThreadsG = kWarpsG * 32;
// Chunks a lane has in flight at once (bf16 records).  Three keeps the kernel
// near 60 registers a thread: a CTA then fits beside the CTAs of the kernel
// before it on the stream (the encoder's, say), so with PDL it starts its
// loads while that kernel drains.  Four chunks run a lone launch ~15% faster
// but need ~84 registers, and the bench step (encode, then the products) came
// out ~3% slower for it.  fp32 records are twice the size: two chunks.
template <bool BF16>
__host__ __device__ constexpr int batch_chunks() { return BF16 ? 3 : 2; }
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

// A chunk's products for one slot (lane): block e selects xb[e m + offset],
// xb = x + 8 c m.  The offset width and, for every chunk but a row's last, the
// 8 blocks' existence are known at compile time, so an element costs an
// extract, an address, a gather and an FMA; two accumulators (even and odd
// blocks) keep independent gathers in flight.
template <bool BF16, bool NIB, bool FULL>
__device__ __forceinline__ float chunk_sum(const ChunkData<BF16> &d, const float *xb, int m, int nvalid) {
    float a0 = 0.0f, a1 = 0.0f;
#pragma unroll
    for (int e = 0; e < kChunk; ++e) {
        if (FULL || e < nvalid) {
            const uint32_t o = NIB ? (d.o.x >> (4 * e)) & 15u : ((e < 4 ? d.o.x : d.o.y) >> (8 * (e & 3))) & 255u;
            const uint4 &q = d.v[BF16 ? 0 : e >> 2];
            const uint32_t word = BF16 ? ((e >> 1) == 0 ? q.x : (e >> 1) == 1 ? q.y : (e >> 1) == 2 ? q.z : q.w)
                                       : ((e & 3) == 0 ? q.x : (e & 3) == 1 ? q.y : (e & 3) == 2 ? q.z : q.w);
            const float v = BF16 ? __uint_as_float((e & 1) ? (word & 0xFFFF0000u) : (word << 16)) : __uint_as_float(word);
            const float x = xb[e * m + int(o)];
            if ((e & 1) && BF16) a1 = fmaf(v, x, a1);   // fp32 records: one chain (register pressure)
            else a0 = fmaf(v, x, a0);
        }
    }
    return a0 + a1;
}

// Chunk c's products for one slot: a row's last chunk may hold fewer than 8 blocks.
template <bool BF16, bool NIB>
__device__ __forceinline__ float chunk_at(const ChunkData<BF16> &d, int c, int n, int m, const float *xs) {
    const float *xb = xs + c * kChunk * m;
    return (c + 1) * kChunk <= n ? chunk_sum<BF16, NIB, true>(d, xb, m, kChunk)
                                 : chunk_sum<BF16, NIB, false>(d, xb, m, n - c * kChunk);
}

// The record of chunk `rec` (lane = slot) from the shared-memory copies of a
// group's values and offsets.
template <bool BF16, bool NIB>
__device__ __forceinline__ ChunkData<BF16> smem_chunk(const unsigned char *s_val, const uint32_t *s_off, int rec) {
    ChunkData<BF16> d;
    if constexpr (BF16) {
        d.v[0] = reinterpret_cast<const uint4 *>(s_val)[rec];
    } else {
        d.v[0] = reinterpret_cast<const uint4 *>(s_val)[2 * rec];
        d.v[1] = reinterpret_cast<const uint4 *>(s_val)[2 * rec + 1];
    }
    d.o = NIB ? make_uint2(s_off[rec], 0u) : reinterpret_cast<const uint2 *>(s_off)[rec];
    return d;
}

// Warp `warp`'s share of a group held in shared memory: chunks warp, warp +
// WARPS, ..., two at a time.
template <bool BF16, bool NIB, int WARPS>
__device__ __forceinline__ float group_sum(const unsigned char *s_val, const uint32_t *s_off, const float *xs,
                                           int nch, int n, int m, int warp, int lane) {
    float acc0 = 0.0f, acc1 = 0.0f;
    int c = warp;
    auto one = [&](int cc, float &acc) {
        acc += chunk_at<BF16, NIB>(smem_chunk<BF16, NIB>(s_val, s_off, cc * kSlots + lane), cc, n, m, xs);
    };
    for (; c + WARPS < nch; c += 2 * WARPS) {
        one(c, acc0);
        one(c + WARPS, acc1);
    }
    if (c < nch) one(c, acc0);
    return acc0 + acc1;
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
    ChunkData<BF16> d[batch_chunks<BF16>()];
    int c0 = warp;
    auto load_batch = [&](int cfirst) {
#pragma unroll
        for (int k = 0; k < batch_chunks<BF16>(); ++k) {
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
    auto run = [&](auto nib) {   // the offset width fixed for the whole loop
        constexpr bool NIB = decltype(nib)::value;
        while (c0 < nch) {
#pragma unroll
            for (int k = 0; k < batch_chunks<BF16>(); ++k) {
                const int c = c0 + k * kWarpsG;
                if (c < nch) acc += chunk_at<BF16, NIB>(d[k], c, g.n, g.m, s_x);
            }
            c0 += batch_chunks<BF16>() * kWarpsG;
            if (c0 < nch) load_batch(c0);
        }
    };
    if (g.nib) run(std::true_type{});
    else run(std::false_type{});
    s_part[warp][lane] = acc;
    __syncthreads();
    if (warp == 0 && lane < g.nrows) {
        float s = 0.0f;
#pragma unroll
        for (int w = 0; w < kWarpsG; ++w) s += s_part[w][lane];
        Y[int64_t(f.rowmap[gi * kSlots + lane]) * ldy] = s;
    }
}

// Warps of gemv_bulk_kernel (32 split a group's chunks twice as finely but ran
// FC6 at batch 1 in 3.4 us against 3.2 for 16).
constexpr int kWarpsB = 16;
constexpr int kThreadsB = kWarpsB * 32;

// Shared memory of gemv_bulk_kernel: [0, 128) the two mbarriers, then vcap
// bytes for a group's values, ocap for its offsets, then x.
template <bool BF16>
__global__ void __launch_bounds__(kThreadsB)
gemv_bulk_kernel(Format f, const float *X, int64_t ldx, float *Y, int64_t ldy, int early, int vcap, int ocap) {
    constexpr int kEsz = BF16 ? 2 : 4;
    extern __shared__ __align__(128) unsigned char sm[];
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm);   // [0]: values and offsets, [1]: x
    unsigned char *const s_val = sm + 128;
    uint32_t *const s_off = reinterpret_cast<uint32_t *>(s_val + vcap);
    float *const s_x = reinterpret_cast<float *>(reinterpret_cast<unsigned char *>(s_off) + ocap);
    __shared__ float s_part[kWarpsB][kSlots];
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
        for (int64_t k = tid; k < cols; k += kThreadsB) s_x[k] = __ldg(X + k * ldx);
    __syncthreads();   // the barriers' initialisation and the plain copy of x are seen by all threads
    const bool ok = __syncthreads_and(mbar_wait(&bar[0], 0) && (!xbulk || mbar_wait(&bar[1], 0)));
    float acc = 0.0f;
    if (ok) {
        acc = g.nib ? group_sum<BF16, true, kWarpsB>(s_val, s_off, s_x, nch, g.n, g.m, warp, lane)
                    : group_sum<BF16, false, kWarpsB>(s_val, s_off, s_x, nch, g.n, g.m, warp, lane);
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
        for (int w = 0; w < kWarpsB; ++w) sum += s_part[w][lane];
        Y[int64_t(f.rowmap[gi * kSlots + lane]) * ldy] = sum;
    }
}

constexpr size_t kBulkSmemLimit = 225 * 1024;   // dynamic: 227 KB a block, less the static partial sums

template <bool BF16>
cudaError_t launch(const Format &f, const float *X, int64_t ldx, float *Y, int64_t ldy, bool early,
                   cudaStream_t stream) {
    // the largest group is one of the smallest block size
    const bool aligned = (reinterpret_cast<uintptr_t>(f.vals) & 15) == 0 && (reinterpret_cast<uintptr_t>(f.offs) & 15) == 0;
    if (f.m_min > 0 && aligned) {
        const int64_t nch = ((f.cols + f.m_min - 1) / f.m_min + kChunk - 1) / kChunk;
        const int64_t vcap = nch * kSlots * kChunk * (BF16 ? 2 : 4);
        // any group (m >= m_min) has at most nch chunks; room for 8-byte offset
        // records, which groups of m > 16 use
        const int64_t ocap = nch * kSlots * 8;
        const int64_t smem = 128 + vcap + ocap + f.cols * 4;
        if (smem <= int64_t(kBulkSmemLimit)) {
            const cudaError_t attr = allow_smem(gemv_bulk_kernel<BF16>, kBulkSmemLimit);
            if (attr != cudaSuccess) return attr;
            return launch_ex(gemv_bulk_kernel<BF16>, dim3(static_cast<unsigned>(f.ngroups)), dim3(kThreadsB),
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
