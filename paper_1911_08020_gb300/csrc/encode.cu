// encode.cu -- block-max weight masking (BMWM) on the GPU.
//
// Sec. 3.1 steps (1)-(3) with the per-row block size of Sec. 3.2: split row r
// into blocks of m_r columns, keep the weight of largest magnitude in each
// block (lowest column on a tie), store its value and its offset in the block.
//
// One CTA per matrix row.  The CTA streams the row (or a tile of whole blocks
// of it) from HBM into shared memory with 16-byte loads, widening bf16 to fp32
// (exact), and flags NaNs on the way.  Then each thread scans one block.  Blocks
// are m words apart, so a straight scan would make lanes collide on shared
// memory banks whenever m is even; each lane instead starts its scan at a
// rotated position s(lane) = (lane * 2^a) / 32, a = min(v2(m), 5), and wraps
// around.  Lanes that share a bank offset t*m mod 32 then start 1..2^a-1 words
// apart, which makes every scan step conflict-free for any m.  Because the scan
// order is rotated, a tie is resolved explicitly by the smaller offset.
//
// The kernel is bound by the HBM read of W: it reads rows*cols elements once
// and writes one value and 4-8 bits per block.
#include "darb_internal.h"

#include <cuda_bf16.h>

namespace darb {
namespace {

constexpr int kEncThreads = 256;
constexpr int kEncTileElems = 12288;   // 48 KB of fp32 staging per CTA

template <bool BF16>
__device__ __forceinline__ float load_w(const void *row, int64_t c) {
    if constexpr (BF16) {
        uint32_t b = static_cast<const uint16_t *>(row)[c];
        return __uint_as_float(b << 16);
    } else {
        return static_cast<const float *>(row)[c];
    }
}

// Stage columns [c0, c1) of one row into smem (as fp32); returns true if a NaN was seen.
template <bool BF16>
__device__ __forceinline__ bool stage_row(const void *row, int64_t c0, int64_t c1, float *tile) {
    bool nan = false;
    const int tid = threadIdx.x;
    constexpr int kEsz = BF16 ? 2 : 4;
    constexpr int kPerVec = 16 / kEsz;
    const char *base = static_cast<const char *>(row);
    // head: up to the first 16-byte aligned column
    int64_t a0 = c0;
    uintptr_t addr0 = reinterpret_cast<uintptr_t>(base + c0 * kEsz);
    int64_t mis = (addr0 & 15) ? (16 - (addr0 & 15)) / kEsz : 0;
    if ((addr0 & (kEsz - 1)) != 0) mis = c1 - c0;   // not even element-aligned for vectors
    int64_t head_end = min(c1, a0 + mis);
    for (int64_t c = c0 + tid; c < head_end; c += kEncThreads) {
        float v = load_w<BF16>(row, c);
        nan |= isnan(v);
        tile[c - c0] = v;
    }
    int64_t nvec = (c1 - head_end) / kPerVec;
    const uint4 *vp = reinterpret_cast<const uint4 *>(base + head_end * kEsz);
    for (int64_t i = tid; i < nvec; i += kEncThreads) {
        uint4 q = __ldcs(vp + i);   // streamed once: evict-first
        uint32_t w[4] = {q.x, q.y, q.z, q.w};
        float *dst = tile + (head_end - c0) + i * kPerVec;
        if constexpr (BF16) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                float lo = __uint_as_float(w[e] << 16);
                float hi = __uint_as_float(w[e] & 0xFFFF0000u);
                nan |= isnan(lo) | isnan(hi);
                dst[2 * e] = lo;
                dst[2 * e + 1] = hi;
            }
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                float v = __uint_as_float(w[e]);
                nan |= isnan(v);
                dst[e] = v;
            }
        }
    }
    for (int64_t c = head_end + nvec * kPerVec + tid; c < c1; c += kEncThreads) {
        float v = load_w<BF16>(row, c);
        nan |= isnan(v);
        tile[c - c0] = v;
    }
    return nan;
}

template <bool BF16>
__global__ void __launch_bounds__(kEncThreads)
encode_kernel(EncodeTarget t, const void *W, int64_t ldw, int32_t *err_flag) {
    __shared__ float tile[kEncTileElems];
    const int64_t r = blockIdx.x;
    const int m = t.row_m[r];
    const int loc = t.rowloc[r];
    const Group grp = t.groups[loc / kSlots];
    const int slot = loc % kSlots;
    const int n = grp.n;
    const int64_t cols = t.cols;
    const int lane = threadIdx.x & 31;
    const char *row = static_cast<const char *>(W) + r * ldw * (BF16 ? 2 : 4);

    // blocks per tile: whole blocks, a multiple of the chunk so offset records
    // never straddle two tiles
    const int tb = (kEncTileElems / m) / kChunk * kChunk;
    // rotation that makes the per-thread scans bank-conflict-free
    const int a = min(__ffs(m) - 1, 5);
    const int rot = (lane << a) >> 5;

    bool nan = false;
    for (int jt = 0; jt < n; jt += tb) {
        const int nb = min(tb, n - jt);
        const int64_t c0 = static_cast<int64_t>(jt) * m;
        const int64_t c1 = min(cols, c0 + static_cast<int64_t>(nb) * m);
        __syncthreads();   // previous tile fully consumed
        nan |= stage_row<BF16>(row, c0, c1, tile);
        __syncthreads();
        const int span = static_cast<int>(c1 - c0);
        // uniform trip count so every lane reaches the shuffles below
        for (int base = 0; base < nb; base += kEncThreads) {
            const int jj = base + threadIdx.x;
            const int j = jt + jj;
            uint32_t best_o = 0;
            if (jj < nb) {
                const int lo = jj * m;
                const int len = min(m, span - lo);
                uint32_t best_a = 0;
                best_o = m;   // sentinel: any element (|w| >= 0) replaces it
                int o = rot >= m ? rot % m : rot;
                for (int k = 0; k < m; ++k) {
                    if (o < len) {
                        const uint32_t av = __float_as_uint(tile[lo + o]) & 0x7FFFFFFFu;
                        if (av > best_a || (av == best_a && static_cast<uint32_t>(o) < best_o)) {
                            best_a = av;
                            best_o = o;
                        }
                    }
                    o = (o + 1 == m) ? 0 : o + 1;
                }
                const float kept = tile[lo + best_o];
                const int64_t vi = grp.val_off +
                                   (static_cast<int64_t>(j / kChunk) * kSlots + slot) * kChunk +
                                   (j % kChunk);
                if constexpr (BF16) {
                    static_cast<uint16_t *>(t.vals)[vi] =
                        static_cast<uint16_t>(__float_as_uint(kept) >> 16);
                } else {
                    static_cast<float *>(t.vals)[vi] = kept;
                }
            }
            // pack the 8 offsets of a chunk: lanes 8q..8q+7 hold blocks 8c..8c+7
            const int e = j % kChunk;
            uint32_t lo_w, hi_w;
            if (grp.nib) {
                lo_w = (jj < nb) ? (best_o << (4 * e)) : 0u;
                hi_w = 0u;
            } else {
                lo_w = (jj < nb && e < 4) ? (best_o << (8 * e)) : 0u;
                hi_w = (jj < nb && e >= 4) ? (best_o << (8 * (e - 4))) : 0u;
            }
#pragma unroll
            for (int d = 1; d < kChunk; d <<= 1) {
                lo_w |= __shfl_xor_sync(0xFFFFFFFFu, lo_w, d);
                hi_w |= __shfl_xor_sync(0xFFFFFFFFu, hi_w, d);
            }
            if (e == 0 && jj < nb) {
                const int64_t rec = static_cast<int64_t>(j / kChunk) * kSlots + slot;
                if (grp.nib) {
                    t.offs[grp.off_off + rec] = lo_w;
                } else {
                    reinterpret_cast<uint2 *>(t.offs + grp.off_off)[rec] = make_uint2(lo_w, hi_w);
                }
            }
        }
    }
    if (__syncthreads_or(nan) && threadIdx.x == 0) atomicExch(err_flag, 1);
}

}  // namespace

cudaError_t launch_encode(const EncodeTarget &t, const void *W, int64_t ldw, int32_t *err_flag,
                          cudaStream_t stream) {
    dim3 grid(static_cast<unsigned>(t.rows));
    if (t.bf16) {
        encode_kernel<true><<<grid, kEncThreads, 0, stream>>>(t, W, ldw, err_flag);
    } else {
        encode_kernel<false><<<grid, kEncThreads, 0, stream>>>(t, W, ldw, err_flag);
    }
    return cudaGetLastError();
}

}  // namespace darb
