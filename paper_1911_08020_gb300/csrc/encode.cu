// encode.cu -- block-max weight masking (BMWM) on the GPU.
//
// Sec. 3.1 steps (1)-(3) with the per-row block size of Sec. 3.2: split row r
// into blocks of m_r columns, keep the weight of largest magnitude in each
// block (lowest column on a tie), store its value and its offset in the block.
//
// The work is a list of tiles (a row, or a run of whole blocks of a long row),
// each resolved on the host into a 32-byte descriptor (position in W, block
// size, destination in the format), so that a tile costs one load to find.
// A persistent grid (as many CTAs per SM as their two tile buffers allow)
// walks the list; each CTA keeps the bulk (TMA) copy of its next tile in
// flight in a second shared-memory buffer while it scans the current one, so
// the HBM read of W -- the only large traffic -- streams without stalls.  Tiles are scanned where the copy
// put them; positions past the row's end are zero-filled, which can never beat
// a real element of the block (it comes later, and ties go to the lowest
// column).  A NaN anywhere in a block would be that block's largest magnitude,
// so checking each block's winner finds every NaN at no extra cost.
//
// Scan: each thread takes one block (for bf16 with power-of-two m >= 8, in
// 16-byte units of 8 elements, see the kernel).  Blocks are m words apart, so a straight
// scan makes lanes collide on shared-memory banks whenever m is even; each lane
// instead starts at a rotated position s(lane) = (lane * 2^a) / 32,
// a = min(v2(m), 5), and wraps around.  Lanes that share a bank offset
// t*m mod 32 then start 1..2^a-1 words apart, so every scan step is
// conflict-free for any m.  Because the order is rotated, ties are resolved
// explicitly by the smaller offset: for bf16, key = |w| << 16 | (0xFFFF - offset)
// and one unsigned max per element does both (two per 32-bit word when m is
// even, the rotation then counted in words); fp32 compares (|w|, offset).
#include "darb_internal.h"
#include "launch.cuh"
#include "tma.cuh"

#include <algorithm>
#include <type_traits>

namespace darb {
namespace {

constexpr int kEncThreads = 128;   // small CTAs: more of them (and their copies) per SM; 256 was 5-17% slower

// Bytes of one stage: the largest tile of the handle plus room for its
// 16-byte-misaligned start, in 128-byte units.  Sizing the ring to the
// handle (not to the largest possible tile) lets short rows run with more
// CTAs per SM, i.e. with more tiles in flight.
inline int stage_bytes(const EncodeTarget &t) {
    const int esz = t.bf16 ? 2 : 4;
    return (t.max_tile * esz + 16 + 127) / 128 * 128;
}

// Two stages a CTA: one tile scanned while the next lands.  More CTAs per SM
// (six for FC6's 18 KB tiles) beat a deeper ring (three stages, four CTAs:
// FC6 22.8 us against 21.6).
template <bool BF16>
__host__ __device__ constexpr int enc_stages() { return 2; }

// shared memory: [0, 32) one mbarrier per stage, [32, 128) the descriptor of
// the tile in each stage, then the stages' raw buffers
template <bool BF16>
inline size_t encode_smem(int sbytes) {
    return 128 + size_t(enc_stages<BF16>()) * sbytes;
}
static_assert(enc_stages<true>() * sizeof(EncTile) <= 96 && enc_stages<false>() * sizeof(EncTile) <= 96,
              "tile descriptors must fit in the shared-memory header");

__device__ __forceinline__ EncTile load_tile(const EncTile *p) {
    union {
        int4 v[2];
        EncTile t;
    } u;
    const int4 *q = reinterpret_cast<const int4 *>(p);
    u.v[0] = __ldg(q);
    u.v[1] = __ldg(q + 1);
    return u.t;
}

// Where a tile sits in W and which of its bytes the bulk copy moves.
struct TileGeo {
    const char *gaddr;   // first byte of the tile in W
    int off0;            // gaddr - (gaddr rounded down to 16 bytes)
    int blo, bhi;        // bulk-copied byte range, relative to the rounded-down address
};

template <bool BF16>
__device__ __forceinline__ TileGeo tile_geo(const EncTile &d, const void *W, int64_t ldw) {
    constexpr int kEsz = BF16 ? 2 : 4;
    TileGeo g;
    g.gaddr = static_cast<const char *>(W) + (int64_t(d.row) * ldw + d.c0) * kEsz;
    g.off0 = static_cast<int>(reinterpret_cast<uintptr_t>(g.gaddr) & 15);
    g.blo = (g.off0 + 15) & ~15;
    g.bhi = (g.off0 + d.span * kEsz) & ~15;
    if (g.bhi < g.blo) g.bhi = g.blo;
    return g;
}

template <bool BF16>
__global__ void __launch_bounds__(kEncThreads)
encode_kernel(EncodeTarget t, const void *W, int64_t ldw, int32_t *status, int sbytes) {
    constexpr int kEsz = BF16 ? 2 : 4;
    constexpr int kStages = enc_stages<BF16>();
    using elem_t = typename std::conditional<BF16, uint16_t, uint32_t>::type;
    extern __shared__ __align__(128) unsigned char sm[];
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm);        // one per stage
    EncTile *s_tile = reinterpret_cast<EncTile *>(sm + 32);   // the tile in each stage
    unsigned char *const raw0 = sm + 128;                    // stage s at raw0 + s * sbytes
    const int tid = threadIdx.x, lane = tid & 31;

    pdl_launch_dependents();
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(&bar[s], 1);
        fence_mbar_init();
    }
    __syncthreads();
    pdl_wait_previous();   // W may come from the previous kernel; outputs may still be read by it

    // thread 0 only: record tile d in stage s and start its bulk copy
    auto issue = [&](const EncTile &d, int s) {
        s_tile[s] = d;
        const TileGeo g = tile_geo<BF16>(d, W, ldw);
        const uint32_t bytes = uint32_t(g.bhi - g.blo);
        mbar_arrive_expect_tx(&bar[s], bytes);
        if (bytes > 0) bulk_g2s(raw0 + s * sbytes + g.blo, g.gaddr - g.off0 + g.blo, bytes, &bar[s]);
    };

    bool nan = false, ok = true;
    uint32_t phases = 0u;   // bit s: parity of stage s's next phase
    int it = 0;
    EncTile next{};         // thread 0: descriptor of the next tile to issue, loaded one iteration early
    if (tid == 0) {
        for (int k = 0; k < kStages - 1; ++k) {
            const int i = blockIdx.x + k * gridDim.x;
            if (i < t.ntiles) issue(load_tile(t.tiles + i), k);
        }
        const int i = blockIdx.x + (kStages - 1) * gridDim.x;
        if (i < t.ntiles) next = load_tile(t.tiles + i);
    }
    for (int i = blockIdx.x; i < t.ntiles; i += gridDim.x, ++it) {
        const int s = it % kStages;
        const int iahead = i + (kStages - 1) * gridDim.x;
        if (iahead < t.ntiles && tid == 0) {
            fence_proxy_async_smem();   // earlier generic accesses to that stage come first
            issue(next, (it + kStages - 1) % kStages);
            if (iahead + int(gridDim.x) < t.ntiles) next = load_tile(t.tiles + iahead + gridDim.x);
        }
        ok = __syncthreads_and(mbar_wait(&bar[s], (phases >> s) & 1u));
        phases ^= 1u << s;
        if (!ok) break;
        const EncTile d = s_tile[s];
        const TileGeo g = tile_geo<BF16>(d, W, ldw);
        const int m = d.m, nb = d.nb;
        const bool nib = m <= 16;
        const int padded = nb * m;   // <= t.max_tile
        // element c of the tile sits at word c of `e`; fill the bytes the bulk
        // copy did not cover (unaligned head and tail) and zero the padding
        elem_t *e = reinterpret_cast<elem_t *>(raw0 + s * sbytes + g.off0);
        const int ehead = (g.blo - g.off0) / kEsz, etail = (g.bhi - g.off0) / kEsz;
        if (ehead > 0 || etail < padded) {   // the same for every thread
            const elem_t *src = reinterpret_cast<const elem_t *>(g.gaddr);
            for (int c = tid; c < ehead && c < padded; c += kEncThreads) e[c] = c < d.span ? __ldg(src + c) : elem_t(0);
            for (int c = etail + tid; c < padded; c += kEncThreads) e[c] = c < d.span ? __ldg(src + c) : elem_t(0);
            __syncthreads();
        }
        // ---- general path: one block per thread
        const int a = min(__ffs(m) - 1, 5);
        const int rot = (lane << a) >> 5;
        // bf16 with an even block size and a 4-byte aligned tile: scan two
        // elements per 32-bit word, rotating in word units (m/2 words per block)
        const bool pairs = BF16 && (m % 2 == 0) && (g.off0 % 4 == 0);
        const int mw = m >> 1;
        const int aw = mw > 0 ? min(__ffs(mw) - 1, 5) : 0;
        const int rotw = (lane << aw) >> 5;
        // bf16, m a power of two >= 8 and a 16-byte aligned tile: 16-byte units of
        // 8 elements (U = m / 8 per block).  Per unit, the largest magnitude by
        // packed 16-bit maxima (no per-element key); per block, the unit that
        // first reaches the block's largest magnitude (ties to the lowest unit,
        // through the unit number in the key); then, in that unit alone, the
        // lowest element with that magnitude.  Lanes start at rotated units
        // (lane & 7 for U >= 8, else (lane & 7) * U / 8: a quarter-warp's 16-byte
        // loads then meet 8 distinct bank groups) and run all U units (no divergence).
        const int U = m >> 3;
        const bool units = BF16 && m >= 8 && (m & (m - 1)) == 0 && (g.off0 % 16 == 0);
        const int rotu = !units ? 0 : U >= 8 ? (lane & 7) : ((lane & 7) * U) >> 3;
        for (int base = 0; base < nb; base += kEncThreads) {
            const int jj = base + tid;
            uint32_t best_o = 0;
            if (jj < nb) {
                const elem_t *blk = e + jj * m;
                int o = rot;
                if constexpr (BF16) {
                    uint32_t best = 0;
                    if (units) {
                        const uint4 *ublk = reinterpret_cast<const uint4 *>(blk);
                        const uint32_t umsk = uint32_t(U) - 1u;
                        uint32_t ukey = 0;   // (largest magnitude << 16) | (0xFFFF - unit)
#pragma unroll 4
                        for (int k = 0; k < U; ++k) {
                            const uint32_t u = (uint32_t(rotu) + uint32_t(k)) & umsk;
                            const uint4 q = ublk[u];
                            const uint32_t m01 = __vmaxu2(q.x & 0x7FFF7FFFu, q.y & 0x7FFF7FFFu);
                            const uint32_t m23 = __vmaxu2(q.z & 0x7FFF7FFFu, q.w & 0x7FFF7FFFu);
                            const uint32_t mm = __vmaxu2(m01, m23);
                            const uint32_t mx = max(mm >> 16, mm & 0xFFFFu);   // the unit's largest magnitude
                            ukey = max(ukey, (mx << 16) | (0xFFFFu - u));
                        }
                        const uint32_t mag = ukey >> 16, u = 0xFFFFu - (ukey & 0xFFFFu);
                        const uint4 q = ublk[u];
                        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
                        uint32_t first = 8;   // lowest element of the unit with that magnitude
#pragma unroll
                        for (int j = 7; j >= 0; --j)
                            if (((w[j >> 1] >> (16 * (j & 1))) & 0x7FFFu) == mag) first = uint32_t(j);
                        best = (mag << 16) | (0xFFFFu - (8u * u + first));
                    } else if (pairs) {
                        const uint32_t *wblk = reinterpret_cast<const uint32_t *>(blk);
                        int qw = rotw;
#pragma unroll 2
                        for (int k = 0; k < mw; ++k) {
                            const uint32_t w = wblk[qw];
                            const uint32_t i0 = 0xFFFFu - 2u * uint32_t(qw);   // key of element 2*qw
                            best = max(best, ((w << 16) & 0x7FFF0000u) | i0);
                            best = max(best, (w & 0x7FFF0000u) | (i0 - 1u));
                            qw = (qw + 1 == mw) ? 0 : qw + 1;
                        }
                    } else {
                        for (int k = 0; k < m; ++k) {
                            best = max(best, ((uint32_t(blk[o]) & 0x7FFFu) << 16) | (0xFFFFu - uint32_t(o)));
                            o = (o + 1 == m) ? 0 : o + 1;
                        }
                    }
                    best_o = 0xFFFFu - (best & 0xFFFFu);
                    nan |= (best >> 16) > 0x7F80u;
                } else {
                    uint32_t best_a = 0;
                    best_o = uint32_t(m);
                    for (int k = 0; k < m; ++k) {
                        const uint32_t av = blk[o] & 0x7FFFFFFFu;
                        if (av > best_a || (av == best_a && uint32_t(o) < best_o)) {
                            best_a = av;
                            best_o = uint32_t(o);
                        }
                        o = (o + 1 == m) ? 0 : o + 1;
                    }
                    nan |= best_a > 0x7F800000u;
                }
                static_cast<elem_t *>(t.vals)[d.val_base + int64_t(jj / kChunk) * (kSlots * kChunk) + jj % kChunk] =
                    blk[best_o];
            }
            // pack the 8 offsets of a chunk: lanes 8q..8q+7 hold blocks 8c..8c+7
            // (tiles start on a chunk boundary, so block jj is at position jj % 8)
            const int q = jj % kChunk;
            uint32_t lo_w, hi_w;
            if (nib) {
                lo_w = (jj < nb) ? (best_o << (4 * q)) : 0u;
                hi_w = 0u;
            } else {
                lo_w = (jj < nb && q < 4) ? (best_o << (8 * q)) : 0u;
                hi_w = (jj < nb && q >= 4) ? (best_o << (8 * (q - 4))) : 0u;
            }
#pragma unroll
            for (int dd = 1; dd < kChunk; dd <<= 1) {
                lo_w |= __shfl_xor_sync(0xFFFFFFFFu, lo_w, dd);
                hi_w |= __shfl_xor_sync(0xFFFFFFFFu, hi_w, dd);
            }
            if (q == 0 && jj < nb) {
                const int64_t c = jj / kChunk;
                if (nib) t.offs[d.off_base + c * kSlots] = lo_w;
                else reinterpret_cast<uint2 *>(t.offs + d.off_base)[c * kSlots] = make_uint2(lo_w, hi_w);
            }
        }
        __syncthreads();   // this stage is free for the copy issued next iteration
    }
    if (!ok) {
        // a copy did not land in time: record it and let the copies still in flight settle
        if (tid == 0) atomicOr(status, kStatusTimeout);
        for (int k = 1; k < kStages; ++k) {
            const int s = (it + k) % kStages;
            mbar_wait(&bar[s], (phases >> s) & 1u);
        }
    }
    if (__syncthreads_or(nan) && tid == 0) atomicOr(status, kStatusNaN);
}

// Largest dynamic shared memory any handle can ask for (tiles of kEncTileElems).
template <bool BF16>
inline size_t encode_smem_max() {
    return encode_smem<BF16>((kEncTileElems * (BF16 ? 2 : 4) + 16 + 127) / 128 * 128);
}

template <bool BF16>
cudaError_t launch_encode_t(const EncodeTarget &t, const void *W, int64_t ldw, int32_t *status,
                            cudaStream_t stream) {
    const cudaError_t a = allow_smem(encode_kernel<BF16>, encode_smem_max<BF16>());
    if (a != cudaSuccess) return a;
    const int sbytes = stage_bytes(t);
    const size_t smem = encode_smem<BF16>(sbytes);
    // resident CTAs per SM at this handle's ring size (shared memory or threads bound it)
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, encode_kernel<BF16>, kEncThreads, smem) != cudaSuccess ||
        per_sm <= 0) {
        cudaGetLastError();
        per_sm = 1;
    }
    const unsigned grid = static_cast<unsigned>(std::min<int64_t>(t.ntiles, per_sm * int64_t(sm_count())));
    if (grid == 0) return cudaSuccess;
    return launch_ex(encode_kernel<BF16>, dim3(grid), dim3(kEncThreads), smem, stream, 1, true, t, W, ldw, status,
                     sbytes);
}

}  // namespace

cudaError_t launch_encode(const EncodeTarget &t, const void *W, int64_t ldw, int32_t *status,
                          cudaStream_t stream) {
    return t.bf16 ? launch_encode_t<true>(t, W, ldw, status, stream) : launch_encode_t<false>(t, W, ldw, status, stream);
}

}  // namespace darb
