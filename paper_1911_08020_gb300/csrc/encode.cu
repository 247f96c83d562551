// encode.cu -- block-max weight masking (BMWM) on the GPU.
//
// Sec. 3.1 steps (1)-(3) with the per-row block size of Sec. 3.2: split row r
// into blocks of m_r columns, keep the weight of largest magnitude in each
// block (lowest column on a tie), store its value and its offset in the block.
//
// Two kernels.  bf16 weights whose block sizes are all powers of two from 8
// to 256 (16-byte units of 8 weights never straddle a block) take the row
// path below (encode_rows_kernel): warps that work alone on 2048-column
// tiles, one 16-byte unit per lane and step.  Everything else (fp32 weights,
// other block sizes, unaligned rows) takes encode_kernel, described here.
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
        ok = __syncthreads_and(mbar_wait(&bar[s], (phases >> s) & 1u, true));
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

// ---------------------------------------------------------------------------
// Row path: bf16 weights, every block size a power of two from 8 to 256,
// 16-byte aligned rows.  Its tiles are kRowPassElems columns (whole records,
// starting on 16-byte boundaries), so that the work spreads evenly over the
// warps whatever the row lengths.  Each warp works alone: it takes every
// kRowWarps * gridDim.x-th tile and keeps kRowStages of them in flight as bulk
// copies into its own shared-memory ring, each completing on the warp's own
// mbarrier -- no CTA barrier, so a warp never waits for another.
//
// Every lane scans 8 of a tile's 16-byte units (8 weights each), whatever m
// is: for m <= 64 it takes 8 / U whole blocks (U = m / 8 units; block
// i * 32 + lane in step i), for m > 64 a slice of 8 units of one block shared
// by L = U / 8 lanes, whose keys meet by xor shuffles.  Per unit, the largest
// magnitude by packed 16-bit maxima and the key |w| << 16 | (0xFFFF - unit),
// one unsigned max per unit keeping the lowest unit on a tie; then, in the
// winning unit alone, the lowest element with that magnitude.  Kept values
// and offsets go through per-warp buffers and leave as whole records (16
// bytes of values, 4 or 8 bytes of offsets), one per lane.
constexpr int kRowWarps = 4;                    // warps per CTA
constexpr int kRowStages = 2;                   // tiles a warp has in flight
constexpr int kRowCtas = 6;                     // CTAs per SM: registers capped to fit them
constexpr int kPassUnits = kRowPassElems / 8;   // 16-byte units of a tile, 8 per lane

struct __align__(128) RowWarp {
    uint4 stage[kRowStages][kPassUnits];
    EncTile desc[kRowStages];    // the tile in each stage
    uint16_t vbuf[kPassUnits];   // a tile's kept values by block (at most kPassUnits blocks, m = 8)
    uint8_t obuf[kPassUnits];    // and their offsets
    uint64_t bar[kRowStages];
};
constexpr size_t kRowSmem = sizeof(RowWarp) * kRowWarps;

// Packed unsigned 16-bit maximum of each half (PTX max.u16x2).
__device__ __forceinline__ uint32_t vmax_u16x2(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("max.u16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

// prmt.b32 in its default mode: byte n of the result is byte (sel >> 4n) & 7 of
// b:a, or, where bit 3 of that nibble is set, that byte's top bit copied to all 8.
__device__ __forceinline__ uint32_t prmt_sign(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t r;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
    return r;
}

// The lowest j in 0..7 whose bf16 element j of unit q (half j & 1 of word
// j >> 1) has magnitude mx, given mx in both halves of mx2 and no element
// above it.  Per half, 0x8000 + |w| - mx keeps bit 15 exactly when |w| == mx
// and never borrows from the other half; prmt with a sign-replicating
// selector turns each such bit into a byte of ones, element 0 in the top
// byte, so the count of leading zero bytes is the index.
__device__ __forceinline__ uint32_t first_max_index(const uint4 &q, uint32_t mx2) {
    const uint32_t d0 = (q.x | 0x80008000u) - mx2, d1 = (q.y | 0x80008000u) - mx2;
    const uint32_t d2 = (q.z | 0x80008000u) - mx2, d3 = (q.w | 0x80008000u) - mx2;
    const uint32_t e0123 = prmt_sign(d0, d1, 0x9BDF);   // byte 3 - j = element j's flag
    const uint32_t e4567 = prmt_sign(d2, d3, 0x9BDF);
    return uint32_t(__clzll((uint64_t(e0123) << 32) | e4567)) >> 3;
}

// 16 bytes of shared memory at a 32-bit shared address (volatile: never moved
// across the mbarrier wait that makes them valid).
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

// One tile with block size 8U in stage s (pu units, whole blocks) -> its kept
// values and offset records.  True if a block's largest magnitude is a NaN.
template <int U>
__device__ __forceinline__ bool row_scan(RowWarp &rw, int s, int pu, int lane, uint16_t *vals, uint32_t *offs) {
    constexpr int S = U < 8 ? U : 8;        // units a lane scans per block (or slice)
    constexpr int L = U > 8 ? U / 8 : 1;    // lanes per block
    constexpr int NSEG = 8 / S;             // blocks a lane takes
    constexpr bool kNib = U <= 2;           // m <= 16: 4-bit offsets
    const uint32_t st = smem_addr(rw.stage[s]);
    // The lane scans units rot ^ k, k = 0..S-1, of its block (or slice): each
    // block (slice) starts on a multiple of S units, so the XOR stays inside
    // it, and the 8 lanes of a quarter-warp meet 8 distinct bank groups.  The
    // key's low half 0xFFFF - (unit in the block) is then lowbase ^ k, as the
    // slice offset is a multiple of 8 and rot ^ k < 8.
    const uint32_t rot = U >= 8 ? uint32_t(lane & 7) : ((uint32_t(lane & 7) * U) >> 3);
    const uint32_t soff = uint32_t(lane & (L - 1)) * 8u;
    const uint32_t lowbase = (0xFFFFu - soff) ^ rot;
    uint32_t key[NSEG];   // (largest magnitude << 16) | (0xFFFF - unit in the block)
#pragma unroll
    for (int i = 0; i < NSEG; ++i) {
        const uint32_t seg = st + ((uint32_t((i * 32 + lane) / L) * U + soff + rot) << 4);
        key[i] = 0u;
#pragma unroll
        for (int k = 0; k < S; ++k) {
            const uint4 q = lds128(seg ^ uint32_t(k << 4));
            const uint32_t mm = vmax_u16x2(vmax_u16x2(q.x & 0x7FFF7FFFu, q.y & 0x7FFF7FFFu),
                                           vmax_u16x2(q.z & 0x7FFF7FFFu, q.w & 0x7FFF7FFFu));
            const uint32_t mx2 = vmax_u16x2(mm, __byte_perm(mm, 0u, 0x1032));   // the unit's largest, both halves
            key[i] = max(key[i], __byte_perm(lowbase ^ uint32_t(k), mx2, 0x7610));
        }
    }
    bool nan = false;
#pragma unroll
    for (int i = 0; i < NSEG; ++i) {
        uint32_t kk = key[i];
#pragma unroll
        for (int sft = 1; sft < L; sft <<= 1) kk = max(kk, __shfl_xor_sync(0xFFFFFFFFu, kk, sft));
        const int blk = (i * 32 + lane) / L;   // block of the tile
        const uint32_t wu = 0xFFFFu - (kk & 0xFFFFu);
        const uint32_t ua = st + ((uint32_t(blk) * U + wu) << 4);   // the winning unit
        const uint32_t j0 = first_max_index(lds128(ua), __byte_perm(kk, 0u, 0x3232));
        if ((lane & (L - 1)) == 0) {
            const bool real = blk * U < pu;
            uint16_t v = 0;
            asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(ua + 2u * j0));
            nan |= real && (kk >> 16) > 0x7F80u;
            rw.vbuf[blk] = real ? v : uint16_t(0);   // blocks past the row's end: zero
            rw.obuf[blk] = real ? uint8_t(wu * 8u + j0) : uint8_t(0);
        }
    }
    __syncwarp();
    // record c (blocks 8c..8c+7) from lane c
    if (lane * kChunk < pu / U) {
        const uint4 vv = *reinterpret_cast<const uint4 *>(rw.vbuf + lane * kChunk);
        const uint2 oo = *reinterpret_cast<const uint2 *>(rw.obuf + lane * kChunk);
        *reinterpret_cast<uint4 *>(vals + int64_t(lane) * (kSlots * kChunk)) = vv;
        if (kNib) {   // bytes b0..b7 (each < 16) -> nibbles: b0 | b1 << 4 | ... | b7 << 28
            offs[lane * kSlots] = __byte_perm(oo.x | (oo.x >> 4), oo.y | (oo.y >> 4), 0x6420);
        } else {
            reinterpret_cast<uint2 *>(offs)[lane * kSlots] = oo;
        }
    }
    __syncwarp();   // the buffers are read before the next tile writes them
    return nan;
}

__global__ void __launch_bounds__(kRowWarps * 32, kRowCtas)
encode_rows_kernel(EncodeTarget t, const uint16_t *W, int64_t ldw, int32_t *status) {
    extern __shared__ __align__(128) unsigned char sm[];
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    RowWarp &rw = reinterpret_cast<RowWarp *>(sm)[wl];
    const int n = t.n_row_tiles, stride = int(gridDim.x) * kRowWarps;
    pdl_launch_dependents();
    if (lane == 0) {
        for (int s = 0; s < kRowStages; ++s) mbar_init(&rw.bar[s], 1);
        fence_mbar_init();
    }
    __syncwarp();
    pdl_wait_previous();   // W may come from the previous kernel; outputs may still be read by it

    // lane 0: record tile d in stage s and start the copy of its whole units
    // (the stage's mbarrier phase also publishes the descriptor to the warp)
    auto issue = [&](const EncTile &d, int s) {
        rw.desc[s] = d;
        const uint32_t bytes = uint32_t(d.span >> 3) * 16u;
        mbar_arrive_expect_tx(&rw.bar[s], bytes);
        if (bytes > 0) bulk_g2s(rw.stage[s], W + int64_t(d.row) * ldw + d.c0, bytes, &rw.bar[s]);
    };
    int pt = blockIdx.x * kRowWarps + wl;   // the next tile to issue
    EncTile nd{};                           // lane 0: its descriptor, loaded a step early
    if (lane == 0 && pt < n) nd = load_tile(t.row_tiles + pt);
    int issued = 0, consumed = 0;
    for (; issued < kRowStages && pt < n; ++issued, pt += stride) {
        if (lane == 0) {
            issue(nd, issued);
            if (pt + stride < n) nd = load_tile(t.row_tiles + pt + stride);
        }
    }
    uint32_t phases = 0u;   // bit s: parity of stage s's pending phase
    bool nan = false, ok = true;
    while (consumed < issued) {
        const int s = consumed % kRowStages;
        ok = __all_sync(0xFFFFFFFFu, mbar_wait(&rw.bar[s], (phases >> s) & 1u));
        if (!ok) break;
        phases ^= 1u << s;
        const EncTile d = rw.desc[s];
        const int U = d.m >> 3;
        const int pu = int(d.nb) * U;         // units of the tile: whole blocks
        const int full_units = d.span >> 3;   // units entirely inside the row: copied
        if (pu > full_units) {
            // the row's ragged end and the zero padding of its last block
            uint4 *st = rw.stage[s];
            const uint16_t *src = W + int64_t(d.row) * ldw + d.c0;
            for (int un = full_units + lane; un < pu; un += 32) {
                uint32_t w[4] = {0u, 0u, 0u, 0u};
                for (int j = 0; j < 8; ++j) {
                    const int c = un * 8 + j;
                    if (c < d.span) w[j >> 1] |= uint32_t(src[c]) << (16 * (j & 1));
                }
                st[un] = make_uint4(w[0], w[1], w[2], w[3]);
            }
            __syncwarp();
        }
        uint16_t *vals = static_cast<uint16_t *>(t.vals) + d.val_base;
        uint32_t *offs = t.offs + d.off_base;
        switch (U) {
            case 1: nan |= row_scan<1>(rw, s, pu, lane, vals, offs); break;
            case 2: nan |= row_scan<2>(rw, s, pu, lane, vals, offs); break;
            case 4: nan |= row_scan<4>(rw, s, pu, lane, vals, offs); break;
            case 8: nan |= row_scan<8>(rw, s, pu, lane, vals, offs); break;
            case 16: nan |= row_scan<16>(rw, s, pu, lane, vals, offs); break;
            default: nan |= row_scan<32>(rw, s, pu, lane, vals, offs); break;
        }
        ++consumed;
        if (pt < n) {   // refill stage s (row_scan ended with a warp barrier: the stage is free)
            if (lane == 0) {
                fence_proxy_async_smem();   // the scan's reads of the stage come first
                issue(nd, s);
                if (pt + stride < n) nd = load_tile(t.row_tiles + pt + stride);
            }
            pt += stride;
            ++issued;
        }
    }
    if (!ok) {
        // a copy did not land in time: record it and let the copies still in flight settle
        if (lane == 0) atomicOr(status, kStatusTimeout);
        for (int k = consumed; k < issued; ++k) {
            const int s = k % kRowStages;
            mbar_wait(&rw.bar[s], (phases >> s) & 1u);
        }
    }
    if (__any_sync(0xFFFFFFFFu, nan) && lane == 0) atomicOr(status, kStatusNaN);
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
    // the row path when its tiles exist and every one starts on a 16-byte
    // boundary (tiles start at multiples of 2048 columns of 16-byte aligned rows)
    if (t.n_row_tiles > 0 && (reinterpret_cast<uintptr_t>(W) & 15) == 0 && (ldw * 2) % 16 == 0) {
        const cudaError_t a = allow_smem(encode_rows_kernel, kRowSmem);
        if (a != cudaSuccess) return a;
        const int per_sm = static_cast<int>(per_device(reinterpret_cast<const void *>(encode_rows_kernel), 0, [] {
            int n = 0;
            if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, encode_rows_kernel, kRowWarps * 32, kRowSmem) !=
                    cudaSuccess || n <= 0) {
                cudaGetLastError();
                n = 1;
            }
            return static_cast<long long>(n);
        }));
        const unsigned grid = static_cast<unsigned>(
            std::min<int64_t>((t.n_row_tiles + kRowWarps - 1) / kRowWarps, per_sm * int64_t(sm_count())));
        return launch_ex(encode_rows_kernel, dim3(grid), dim3(kRowWarps * 32), kRowSmem, stream, 1, true, t,
                         static_cast<const uint16_t *>(W), ldw, status);
    }
    return t.bf16 ? launch_encode_t<true>(t, W, ldw, status, stream) : launch_encode_t<false>(t, W, ldw, status, stream);
}

}  // namespace darb
