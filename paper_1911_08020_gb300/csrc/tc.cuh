// tc.cuh -- Y = W_darb X on the tensor cores (tcgen05, kind::f16) for bf16
// weights and wide batches.
//
// Past a few dozen batch columns the CUDA-core product is bound by gathering
// one activation operand from shared memory per (kept weight, column) pair.
// This path instead densifies a slice of W_darb in shared memory and hands
// the contraction to the tensor cores: the zeros cost m times the multiplies
// of the sparse product, but a GB300 SM does them far faster than it can
// gather.
//
// Two kernels per call:
//  * split_kernel writes X once as two bf16 arrays, x = hi + lo, into
//    stream-ordered workspace (the tensor cores take bf16 X only with bf16
//    weights, and one bf16 copy would be too coarse);
//  * tc_kernel.  Work unit: 256 rows (eight consecutive 32-row groups, any
//    block sizes) x one batch tile of N = 32..256 columns x one split-K
//    rank's share of the columns of W, walked in stages of 32 columns (64
//    for N <= 64):
//      - a TMA warp copies the stage's rows of hi and lo for the batch tile
//        straight into two MN-major B tiles (128-byte swizzle; rows and
//        columns past the ends read as zeros);
//      - sixteen producer warps, two per 32-row group taking alternate
//        stages (one thread per row; all lanes of a warp share the group's
//        block size and walk the blocks in lockstep), zero the row's 64 bytes
//        of the stage and write the row's kept values that fall in it (bf16,
//        exact) into two 128 x 32 A tiles (K-major, 64-byte swizzle); for
//        m >= 16 at most three blocks meet a stage and are decoded in
//        straight-line code;
//      - an MMA warp issues, per stage and 128-row half, A*B_hi + A*B_lo for
//        two K=16 steps into that half's TMEM accumulator (128 lanes x N fp32
//        columns) and releases the stage with tcgen05.commit.
//    At the end the ranks of a tile add their partial accumulators: every
//    rank writes its partial tile to workspace (L2-resident, coalesced),
//    the ranks meet -- on the tile's arrival counter (bounded wait) when they
//    are CTAs of one cooperative launch, at a cluster barrier when they are
//    a cluster -- and each rank adds the partials of its slice of the rows
//    in rank order (deterministic) and writes them to Y.  (Pushing the rows
//    through distributed shared memory instead moved only ~10 bytes/clock
//    per SM.)
// Per stage the shared memory moves the MMA operands (96 KB at N = 256), the
// copied B tiles and the A rows; with the split done beforehand that stays
// near what the tensor cores need for the stage's multiplies.
//
// Numerics: weights are exact; |x - hi - lo| <= 2^-16 |x| (two round-to-
// nearest bf16 steps), products are exact and accumulate in fp32, so
// |Y - Y_exact| <= 2^-16 * sum |val * x| plus fp32 accumulation error.
// Non-finite activations are multiplied by the zeros of the dense tile (and
// an infinity has no finite low part), so a NaN or infinity in X can turn
// rows that do not select it into NaN; |x| must stay below the largest bf16.
#pragma once

#include "darb_internal.h"
#include "launch.cuh"
#include "tcgen05.cuh"
#include "tma.cuh"

#include <cooperative_groups.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cstring>

namespace darb {
namespace tc {

namespace cg = cooperative_groups;

constexpr int kRows = 256;                       // rows per CTA
constexpr int kCtaGroups = kRows / kSlots;       // 32-row groups per CTA
// Columns of W per stage, KW: 32, or 64 for narrow batch tiles (N <= 64),
// where the tensor cores finish a stage so fast that the per-stage hand-offs
// would dominate.
constexpr int kRowWarps = kRows / 32;            // warps that cover the CTA's rows once
constexpr int kProducerWarps = 2 * kRowWarps;    // kept values -> A: two warps per group, alternate stages
constexpr int kTmaWarp = kProducerWarps;         // activation copies
constexpr int kMmaWarp = kTmaWarp + 1;           // TMEM owner, MMA issue
constexpr int kThreads = (kMmaWarp + 1) * 32;
constexpr int kBox = 64;                         // batch columns of one B box (128 bytes of bf16)
constexpr int kMaxStages = 8;
constexpr int kStageOff = 1024;                  // after the barriers; 1024-byte aligned
constexpr size_t kSmemLimit = 227 * 1024;

// Layout of one stage width KW.  A rows are KW bf16 (64 or 128 bytes, with the
// swizzle of that width: 8-row atoms of 512 or 1024 bytes); a B tile is made
// of boxes of 64 batch columns x KW rows, i.e. KW/8 K groups of 8-row x
// 128-byte atoms per 64 columns.
template <int KW>
struct Geo {
    static constexpr int kARow = KW * 2;                     // bytes of one A row
    static constexpr int kAHalf = 128 * kARow;               // one 128-row A tile
    static constexpr int kAtom = 8 * kARow;                  // 8-row A atom
    static constexpr uint32_t kALayout = KW == 32 ? kLayoutSw64 : kLayoutSw128;
    static constexpr int kBCol = KW * 128;                   // one 64-column group of a B tile
    static constexpr int kWindow = (KW - 1) / 16 + 2;        // blocks meeting a stage when m >= 16
    static_assert(KW == 32 || KW == 64, "stage width");
    // A row r (0..127) of a tile starts at row(r); kept value column p of it
    // sits at row(r) + ((2p) ^ swz(r)): the swizzle XORs the 16-byte chunk bits
    static __device__ __forceinline__ int row(int r) { return (r >> 3) * kAtom + (r & 7) * kARow; }
    static __device__ __forceinline__ int swz(int r) { return KW == 32 ? ((r >> 1) & 3) << 4 : (r & 7) << 4; }
    static __host__ __device__ constexpr int b_tile_bytes(int N) { return (N + kBox - 1) / kBox * kBCol; }
    // an MMA stage: the two A halves, B_hi and B_lo
    static __host__ __device__ constexpr int stage_bytes(int N) { return 2 * kAHalf + 2 * b_tile_bytes(N); }
};

__host__ __device__ constexpr int stage_width(int N) { return N <= 64 ? 64 : 32; }

__host__ __device__ constexpr uint32_t tmem_cols(int N) { return 2 * N < 32 ? 32u : uint32_t(2 * N); }

struct Plan {
    int N;          // batch tile width: 32, 64, 128 or 256
    int KW;         // stage width
    int nstages;    // MMA stages in the ring
    size_t smem;    // dynamic shared memory, including 1024 bytes of alignment slack
};

inline Plan plan_for(int N) {
    Plan p{};
    p.N = N;
    p.KW = stage_width(N);
    const int sb = p.KW == 64 ? Geo<64>::stage_bytes(N) : Geo<32>::stage_bytes(N);
    const size_t budget = kSmemLimit - 1024 - kStageOff;
    p.nstages = static_cast<int>(budget / sb);
    if (p.nstages > kMaxStages) p.nstages = kMaxStages;
    p.smem = 1024 + kStageOff + size_t(p.nstages) * sb;
    return p;
}

// x -> (hi, lo) as bf16 bits: hi = bf16(x), lo = bf16(x - hi), both rounded to nearest.
__device__ __forceinline__ void split2(float a, float b, uint32_t *hi, uint32_t *lo) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    const __nv_bfloat162 l = __floats2bfloat162_rn(a - __low2float(h), b - __high2float(h));
    *hi = *reinterpret_cast<const uint32_t *>(&h);
    *lo = *reinterpret_cast<const uint32_t *>(&l);
}

// hi, lo: cols x batch bf16 with row pitch ldw (a multiple of 8).  Item i is
// four consecutive batch columns of one row; a thread takes kSplitItems items
// a gridDim.x * 256 apart and issues all their loads before it converts any
// (one round trip to HBM instead of one per item).  cols * ceil(batch / 4)
// < 2^30 (checked by the caller), so no item index overflows an int.
constexpr int kSplitItems = 4;
__global__ void __launch_bounds__(256)
split_kernel(const float *X, int64_t ldx, int64_t batch, int64_t cols, uint16_t *hi, uint16_t *lo, int64_t ldw,
             int *arrive, int narrive) {
    pdl_launch_dependents();
    pdl_wait_previous();   // X may come from the previous kernel; the workspace may still be read by it
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < narrive; i += gridDim.x * blockDim.x) arrive[i] = 0;
    const int q4 = static_cast<int>((batch + 3) / 4), nb = static_cast<int>(batch);
    const int items = static_cast<int>(cols) * q4;
    const bool vec = (ldx & 3) == 0 && (reinterpret_cast<uintptr_t>(X) & 15) == 0;
    const int stride = gridDim.x * blockDim.x;
    for (int i0 = blockIdx.x * blockDim.x + threadIdx.x; i0 < items; i0 += kSplitItems * stride) {
        float4 v[kSplitItems];
#pragma unroll
        for (int u = 0; u < kSplitItems; ++u) {
            const int i = i0 + u * stride;
            v[u] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if (i < items) {
                const int k = i / q4, b = (i - k * q4) * 4;
                const float *x = X + int64_t(k) * ldx + b;
                if (vec && b + 4 <= nb) {
                    v[u] = __ldg(reinterpret_cast<const float4 *>(x));
                } else {
                    v[u].x = __ldg(x);
                    if (b + 1 < nb) v[u].y = __ldg(x + 1);
                    if (b + 2 < nb) v[u].z = __ldg(x + 2);
                    if (b + 3 < nb) v[u].w = __ldg(x + 3);
                }
            }
        }
#pragma unroll
        for (int u = 0; u < kSplitItems; ++u) {
            const int i = i0 + u * stride;
            if (i < items) {
                const int k = i / q4, b = (i - k * q4) * 4;
                uint2 h, l;
                split2(v[u].x, v[u].y, &h.x, &l.x);
                split2(v[u].z, v[u].w, &h.y, &l.y);
                // ldw is a multiple of 8 and b of 4, so b + 4 <= ldw: 8-byte aligned, inside the row
                *reinterpret_cast<uint2 *>(hi + int64_t(k) * ldw + b) = h;
                *reinterpret_cast<uint2 *>(lo + int64_t(k) * ldw + b) = l;
            }
        }
    }
}

template <int KW>
__global__ void __launch_bounds__(kThreads, 1)
tc_kernel(const __grid_constant__ CUtensorMap hmap, const __grid_constant__ CUtensorMap lmap, Format f, int ksplit,
          int nstages, int N, int64_t batch, float *Y, int64_t ldy, float *part, int *arrive, int early) {
    using G = Geo<KW>;
    constexpr int kK = KW;
    constexpr int kARow = G::kARow, kAHalf = G::kAHalf;
    extern __shared__ unsigned char sm_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) &
                                                          ~uintptr_t(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(sm);     // MMA stage written (producers, TMA)
    uint64_t *empty = full + kMaxStages;                   // MMA stage consumed (commit)
    uint64_t *done = empty + kMaxStages;
    uint32_t *s_tmem = reinterpret_cast<uint32_t *>(done + 1);
    unsigned char *const stages = sm + kStageOff;
    const int sbytes = G::stage_bytes(N), bbytes = G::b_tile_bytes(N);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int tile = blockIdx.x / ksplit, rank = blockIdx.x % ksplit;
    const int64_t n0 = int64_t(blockIdx.y) * N;
    const int KS = static_cast<int>((f.cols + kK - 1) / kK);
    const int ks0 = static_cast<int>(int64_t(KS) * rank / ksplit);
    const int nst = static_cast<int>(int64_t(KS) * (rank + 1) / ksplit) - ks0;
    const uint32_t tcols = tmem_cols(N);

    pdl_launch_dependents();
    if (tid == 0) {
        for (int s = 0; s < kMaxStages; ++s) {
            mbar_init(&full[s], kRowWarps + 1);   // the stage's producer warps and the TMA thread
            mbar_init(&empty[s], 1);
        }
        mbar_init(done, 1);
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(s_tmem, tcols);
        tmem_relinquish();
    }
    if (warp == kTmaWarp && lane == 0) {
        prefetch_tensormap(&hmap);
        prefetch_tensormap(&lmap);
    }
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem = *s_tmem;
    bool ok = true;

    if (warp < kProducerWarps) {
        // ---- producers: warp w covers group tile*8 + (w % 8), so m is uniform
        // across it, on the stages of parity w / 8; thread t owns row t % 256
        // of the CTA (half (t % 256) / 128 of the tile)
        if (!early) pdl_wait_previous();
        const int t = tid & (kRows - 1), r = t & 127, par = warp / kRowWarps;
        const int g = tile * kCtaGroups + (warp & (kRowWarps - 1));
        int m = 1, n = 0, nib = 1, nrows = 0;
        int64_t val_off = 0, off_off = 0;
        if (g < f.ngroups) {
            const Group G = f.groups[g];
            m = G.m;
            n = G.n;
            nib = G.nib;
            nrows = G.nrows;
            val_off = G.val_off;
            off_off = G.off_off;
        }
        const bool valid = lane < nrows;
        const uint16_t *vals = static_cast<const uint16_t *>(f.vals);
        auto load_chunk = [&](int c, uint4 &v, uint2 &o) {
            const int64_t rec = int64_t(c) * kSlots + lane;
            if (valid && c * kChunk < n) {
                v = __ldg(reinterpret_cast<const uint4 *>(vals + val_off + rec * kChunk));
                if (nib) o = make_uint2(__ldg(f.offs + off_off + rec), 0u);
                else o = __ldg(reinterpret_cast<const uint2 *>(f.offs + off_off) + rec);
            }
        };
        // blocks of this warp's first stage start at jb = floor(k0 / m), rem = k0 - jb*m;
        // each next stage of the warp moves k0 by 64 = q64*m + r64
        const int k0first = (ks0 + par) * kK;
        int jb = k0first / m, rem = k0first - jb * m;
        const int q64 = 2 * kK / m, r64 = 2 * kK - q64 * m;   // two stages: 2*KW columns
        // chunk cc in (cv, co), cc+1 and cc+2 prefetched
        int cc = jb >> 3;
        uint4 cv = make_uint4(0, 0, 0, 0), v1 = cv, v2 = cv;
        uint2 co = make_uint2(0, 0), o1 = co, o2 = co;
        load_chunk(cc, cv, co);
        load_chunk(cc + 1, v1, o1);
        load_chunk(cc + 2, v2, o2);
        unsigned char *const row0 = stages + (t >> 7) * kAHalf + G::row(r);   // this row in stage 0
        const int swz = G::swz(r);
        auto value = [](const uint4 &v, int q) -> uint16_t {
            const uint32_t w = (q >> 1) == 0 ? v.x : (q >> 1) == 1 ? v.y : (q >> 1) == 2 ? v.z : v.w;
            return static_cast<uint16_t>((q & 1) ? w >> 16 : w);
        };
        auto offset = [nib](const uint2 &o, int q) -> uint32_t {
            return nib ? (o.x >> (4 * q)) & 15u : ((q < 4 ? o.x : o.y) >> (8 * (q & 3))) & 255u;
        };
        int s = par % nstages;
        uint32_t phase = par >= nstages ? 1u : 0u;   // parity of the current use of stage s
        for (int it = par; it < nst; it += 2) {
            if (it >= nstages && !__all_sync(0xFFFFFFFFu, mbar_wait(&empty[s], phase ^ 1u, false))) {
                ok = false;   // the whole warp leaves together
                break;
            }
            unsigned char *const row = row0 + size_t(s) * sbytes;
#pragma unroll
            for (int c = 0; c < kARow / 16; ++c)   // rotated by lane: spread over the banks
                reinterpret_cast<uint4 *>(row)[(c + lane) & (kARow / 16 - 1)] = make_uint4(0, 0, 0, 0);
            const int k0 = (ks0 + it) * kK;
            if (m >= 16) {
                // blocks jb .. jb + kWindow - 1 (in chunk cc or cc+1) cover the stage
#pragma unroll
                for (int b = 0; b < G::kWindow; ++b) {
                    const int j = jb + b;
                    const bool in1 = (j >> 3) != cc;
                    const int q = j & 7;
                    const int p = j * m + static_cast<int>(offset(in1 ? o1 : co, q)) - k0;
                    if (valid && j < n && static_cast<unsigned>(p) < static_cast<unsigned>(kK))
                        *reinterpret_cast<uint16_t *>(row + ((2 * p) ^ swz)) = value(in1 ? v1 : cv, q);
                }
            } else {
                // blocks j with j*m < k0 + 32, from jb on: the same for every lane
                for (int j = jb; j < n && j * m < k0 + kK; ++j) {
                    while ((j >> 3) != cc) {   // step through to j's chunk, prefetch two ahead
                        ++cc;
                        cv = v1;
                        co = o1;
                        v1 = v2;
                        o1 = o2;
                        load_chunk(cc + 2, v2, o2);
                    }
                    const int q = j & 7;
                    const int p = j * m + static_cast<int>(offset(co, q)) - k0;
                    if (valid && static_cast<unsigned>(p) < static_cast<unsigned>(kK))
                        *reinterpret_cast<uint16_t *>(row + ((2 * p) ^ swz)) = value(cv, q);
                }
            }
            jb += q64;
            rem += r64;
            if (rem >= m) {
                rem -= m;
                ++jb;
            }
            if (m >= 16 && (jb >> 3) != cc) {   // at most one chunk per step when m >= 16
                cc = jb >> 3;
                cv = v1;
                co = o1;
                v1 = v2;
                o1 = o2;
                load_chunk(cc + 2, v2, o2);
            }
            fence_proxy_async_smem();   // the tensor core reads A through the async proxy
            __syncwarp();
            if (lane == 0) mbar_arrive(&full[s]);
            s += 2;
            while (s >= nstages) {
                s -= nstages;
                phase ^= 1u;
            }
        }
    } else if (warp == kTmaWarp) {
        // ---- the stage's rows of hi and lo, straight into the B tiles
        if (lane == 0) {
            pdl_wait_previous();   // the split is the previous kernel
            const int nbox = (N + kBox - 1) / kBox;
            int s = 0;
            uint32_t phase = 0;
            for (int it = 0; it < nst; ++it) {
                if (it >= nstages && !mbar_wait(&empty[s], phase ^ 1u, false)) {
                    ok = false;
                    break;
                }
                unsigned char *bhi = stages + size_t(s) * sbytes + 2 * kAHalf, *blo = bhi + bbytes;
                mbar_arrive_expect_tx(&full[s], static_cast<uint32_t>(2 * bbytes));
                const int k0 = (ks0 + it) * kK;
                for (int b = 0; b < nbox; ++b) {
                    tensor2d_g2s(bhi + b * G::kBCol, &hmap, static_cast<int>(n0) + kBox * b, k0, &full[s]);
                    tensor2d_g2s(blo + b * G::kBCol, &lmap, static_cast<int>(n0) + kBox * b, k0, &full[s]);
                }
                if (++s == nstages) {
                    s = 0;
                    phase ^= 1u;
                }
            }
        }
        __syncwarp();
    } else {
        // ---- MMA issue: D_h += A_h * B_hi + A_h * B_lo, two K=16 steps per stage
        const uint32_t idesc = idesc_bf16(128, N, false, true);
        const uint32_t sa0 = smem_addr(stages);
        // descriptors of stage 0; a stage is sbytes further on (the start
        // address field counts 16-byte units)
        const uint64_t a0 = smem_desc(sa0, 16, G::kAtom, G::kALayout);
        const uint64_t bh0 = smem_desc(sa0 + 2 * kAHalf, G::kBCol, 1024, kLayoutSw128);
        const uint64_t bl0 = smem_desc(sa0 + 2 * kAHalf + bbytes, G::kBCol, 1024, kLayoutSw128);
        int s = 0;
        uint32_t phase = 0;
        for (int it = 0; it < nst; ++it) {
            if (!__all_sync(0xFFFFFFFFu, mbar_wait(&full[s], phase, false))) {
                ok = false;
                break;
            }
            tc_fence_after_sync();
            if (lane == 0) {
                const uint64_t so = uint64_t(s) * uint64_t(sbytes >> 4);
#pragma unroll
                for (int kk = 0; kk < kK / 16; ++kk) {
                    const uint64_t bh = bh0 + so + kk * (2048 >> 4), bl = bl0 + so + kk * (2048 >> 4);
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh) {
                        const uint64_t ad = a0 + so + (hh * kAHalf + kk * 32) / 16;
                        mma_bf16(tmem + hh * N, ad, bh, idesc, (it | kk) != 0 ? 1u : 0u);
                        mma_bf16(tmem + hh * N, ad, bl, idesc, 1u);
                    }
                }
                mma_commit(&empty[s]);
            }
            __syncwarp();
            if (++s == nstages) {
                s = 0;
                phase ^= 1u;
            }
        }
        if (lane == 0) mma_commit(done);   // fires once every MMA above has completed
        __syncwarp();
    }

    // ---- epilogue: accumulators -> Y (through a cluster reduction when split)
    if (warp < kRowWarps) {
        if (!__all_sync(0xFFFFFFFFu, mbar_wait(done, 0, false))) ok = false;
        tc_fence_after_sync();
    }
    pdl_wait_previous();   // Y may still be read by the previous kernel
    const bool vec = (ldy & 3) == 0 && (reinterpret_cast<uintptr_t>(Y) & 15) == 0;
    if (ksplit == 1) {
        if (warp < kRowWarps) {
            // as for the partial tiles below: turn each 32 x 32 block around in
            // shared memory so that 8 lanes write 32 consecutive columns of a row
            const int g = tile * kCtaGroups + warp;
            float *tb = reinterpret_cast<float *>(stages) + warp * (32 * 36);
            const uint32_t tl = tmem + (uint32_t(32 * (warp & 3)) << 16) + uint32_t((warp >> 2) * N);
            int64_t rows8[8];   // matrix rows of the block rows this lane writes
#pragma unroll
            for (int i = 0; i < 8; ++i) rows8[i] = g < f.ngroups ? f.rowmap[g * kSlots + 4 * i + (lane >> 3)] : -1;
#pragma unroll 1
            for (int cb = 0; cb < N / 32; ++cb) {   // 32 registers of accumulator at a time
                uint32_t v[32];
                tmem_ld32(tl + cb * 32, v);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    reinterpret_cast<uint4 *>(tb + lane * 36)[i] = make_uint4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                __syncwarp();
                const int64_t c0 = n0 + cb * 32 + 4 * (lane & 7);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int rr = 4 * i + (lane >> 3);
                    const float4 a4 = reinterpret_cast<const float4 *>(tb + rr * 36)[lane & 7];
                    if (rows8[i] >= 0 && c0 < batch) {
                        float *y = Y + rows8[i] * ldy + c0;
                        if (vec && c0 + 4 <= batch) {
                            *reinterpret_cast<float4 *>(y) = a4;
                        } else {
                            const float f4[4] = {a4.x, a4.y, a4.z, a4.w};
                            for (int q = 0; q < 4 && c0 + q < batch; ++q) y[q] = f4[q];
                        }
                    }
                }
                __syncwarp();
            }
        }
    } else {
        // partial tiles [tile of the grid][rank][256 rows][N] in workspace
        float *const mine = part + ((size_t(blockIdx.y) * (gridDim.x / ksplit) + tile) * ksplit + rank) *
                                       size_t(kRows) * N;
        if (warp < kRowWarps) {
            // a lane holds one row; turn each 32 x 32 block around in shared memory
            // (rows padded to 36 floats: conflict-free) so that every store
            // instruction writes four whole 128-byte row segments
            float *tb = reinterpret_cast<float *>(stages) + warp * (32 * 36);   // the rings are free now
            const uint32_t tl = tmem + (uint32_t(32 * (warp & 3)) << 16) + uint32_t((warp >> 2) * N);
#pragma unroll 1
            for (int cb = 0; cb < N / 32; ++cb) {   // 32 registers of accumulator at a time
                uint32_t v[32];
                tmem_ld32(tl + cb * 32, v);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    reinterpret_cast<uint4 *>(tb + lane * 36)[i] = make_uint4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                __syncwarp();
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int rr = 4 * i + (lane >> 3), c4 = lane & 7;   // row of the block, float4 in the row
                    __stcg(reinterpret_cast<float4 *>(mine + size_t(warp * 32 + rr) * N + cb * 32) + c4,
                           reinterpret_cast<const float4 *>(tb + rr * 36)[c4]);
                }
                __syncwarp();
            }
        }
        if (arrive == nullptr) {
            cg::this_cluster().sync();   // release/acquire: every rank's partial tile is visible
        } else {
            // the ranks of the tile are CTAs of a cooperative launch: count in, then
            // wait (bounded) until every rank has published its partial tile
            __shared__ int s_go;
            __syncthreads();
            if (tid == 0) {
                int *ctr = arrive + blockIdx.y * (gridDim.x / ksplit) + tile;
                __threadfence();
                atomicAdd(ctr, 1);
                const unsigned long long t0 = global_timer_ns();
                int go = 1;
                while (true) {
                    int v;
                    asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
                    if (v >= ksplit) break;
                    if (global_timer_ns() - t0 > kWaitLimitNs) {
                        go = 0;
                        break;
                    }
                    __nanosleep(32);
                }
                __threadfence();
                s_go = go;
            }
            __syncthreads();
            if (!s_go) {
                if (tid == 0) atomicOr(f.status, kStatusTimeout);
                goto finish;
            }
        }
        const float *first = mine - size_t(rank) * kRows * N;   // rank 0's tile
        const int own = (kRows + ksplit - 1) / ksplit;       // rows each rank adds up
        const int r0 = rank * own, r1 = min(kRows, r0 + own);
        const int nq = N / 4;
        const size_t sstride = size_t(kRows) * N / 4;         // float4s between two ranks' tiles
#pragma unroll 1
        for (int e = tid; e < (r1 - r0) * nq; e += kThreads) {
            const int crow = r0 + e / nq, c4 = e % nq;
            const float4 *src4 = reinterpret_cast<const float4 *>(first + size_t(crow) * N) + c4;
            float4 v[8];   // every rank's partial in flight at once (ksplit <= 8), added in rank order
#pragma unroll
            for (int i = 0; i < 8; ++i)
                if (i < ksplit) v[i] = __ldcg(src4 + i * sstride);
            float4 acc = v[0];
#pragma unroll
            for (int i = 1; i < 8; ++i)
                if (i < ksplit) {
                    acc.x += v[i].x;
                    acc.y += v[i].y;
                    acc.z += v[i].z;
                    acc.w += v[i].w;
                }
            const int g = tile * kCtaGroups + crow / kSlots;
            const int64_t row = g < f.ngroups ? f.rowmap[g * kSlots + crow % kSlots] : -1;
            const int64_t c0 = n0 + 4 * c4;
            if (row >= 0 && c0 < batch) {
                float *y = Y + row * ldy + c0;
                if (vec && c0 + 4 <= batch) {
                    *reinterpret_cast<float4 *>(y) = acc;
                } else {
                    const float a4[4] = {acc.x, acc.y, acc.z, acc.w};
                    for (int i = 0; i < 4 && c0 + i < batch; ++i) y[i] = a4[i];
                }
            }
        }
    }

finish:
    if (!ok) atomicOr(f.status, kStatusTimeout);
    tc_fence_before_sync();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after_sync();
        tmem_dealloc(tmem, tcols);
    }
}

// Tensor map over one bf16 part of X (cols x batch, row pitch ldw elements)
// with 64-column x kw-row boxes and 128-byte swizzle.
inline bool make_part_map(CUtensorMap *map, const uint16_t *part, int64_t ldw, int64_t batch, int64_t cols, int kw) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (enc == nullptr) return false;
    const cuuint64_t dims[2] = {cuuint64_t(batch), cuuint64_t(cols)};
    const cuuint64_t strides[1] = {cuuint64_t(ldw) * 2};
    const cuuint32_t box[2] = {cuuint32_t(kBox), cuuint32_t(kw)};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t *>(part), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

inline int tile_width(int64_t batch) {
    int N = 32;
    while (N < 256 && N < batch) N <<= 1;
    return N;
}

// Clusters of `ksplit` CTAs of this kernel that can be resident at once (-1 if unknown).
template <int KW>
inline int active_clusters(int ksplit, const Plan &p) {
    const void *key = reinterpret_cast<const void *>(tc_kernel<KW>);
    return static_cast<int>(per_device(key, 16ll * p.N + ksplit, [&]() -> long long {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(ksplit * 64, 1);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = p.smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = ksplit;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, tc_kernel<KW>, &cfg) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
    }
    return n > 0 ? n : -1;
    }));
}

// CTAs of this kernel that fit on the device at once (for a cooperative launch).
template <int KW>
inline int64_t coop_capacity(const Plan &p) {
    const void *key = reinterpret_cast<const void *>(tc_kernel<KW>);
    const long long n = per_device(key, -1000ll - p.N, [&]() -> long long {
        int per_sm = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, tc_kernel<KW>, kThreads, p.smem) != cudaSuccess) {
            cudaGetLastError();
            per_sm = 0;
        }
        return per_sm > 0 ? static_cast<long long>(per_sm) * sm_count() : -1;
    });
    return n > 0 ? n : 0;
}

// Cluster split: fewest waves per unit of work, i.e. the smallest
// ceil(units / resident clusters) / ksplit, never more ranks than stages.
template <int KW>
inline int pick_split(int64_t units, int KS, const Plan &p) {
    int best = 1;
    double best_cost = 1e30;
    for (int s = 1; s <= 8 && s <= KS; ++s) {
        int act = active_clusters<KW>(s, p);
        if (act <= 0) act = sm_count() / s;
        if (act <= 0) continue;
        const int64_t waves = (units + act - 1) / act;
        const double cost = double(waves) / s;
        if (cost < best_cost - 1e-9) {
            best_cost = cost;
            best = s;
        }
    }
    return best;
}

template <int KW>
cudaError_t launch_kw(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy, bool early,
                      const Plan &p, cudaStream_t stream) {
    const cudaError_t a = [] {
        size_t most = 0;
        for (int w = 32; w <= 256; w *= 2)
            if (stage_width(w) == KW) most = plan_for(w).smem > most ? plan_for(w).smem : most;
        return allow_smem(tc_kernel<KW>, most);
    }();
    if (a != cudaSuccess) return a;
    const int T = (f.ngroups + kCtaGroups - 1) / kCtaGroups;
    const int64_t NT = (batch + p.N - 1) / p.N;
    const int KS = static_cast<int>((f.cols + KW - 1) / KW);
    const int64_t units = int64_t(T) * NT;
    int ksplit = pick_split<KW>(units, KS, p);
    // A cooperative launch (every CTA resident at once) lets the ranks of a tile
    // meet on a counter instead of a cluster barrier, so the split is not held
    // to the cluster shapes a GPC can place: up to 8 ranks as long as one wave
    // of CTAs holds every tile.
    const int coop_split = static_cast<int>(std::min<int64_t>({8, int64_t(KS), coop_capacity<KW>(p) / units}));
    const bool coop = coop_split > ksplit;
    const int kmax = coop ? coop_split : ksplit;
    // workspace: hi and lo parts of X, the partial tiles of a split, the tiles' arrival counters
    const int64_t ldw = (batch + 7) / 8 * 8;
    const size_t part = (size_t(f.cols) * size_t(ldw) * 2 + 255) / 256 * 256;
    const size_t partials = kmax > 1 ? size_t(kmax) * units * kRows * p.N * 4 : 0;
    const size_t counters = coop ? size_t(units) * 4 : 0;
    void *ws = nullptr;
    cudaError_t e = stream_alloc(&ws, 2 * part + partials + counters, stream);
    if (e != cudaSuccess) return e;
    uint16_t *hi = static_cast<uint16_t *>(ws), *lo = hi + part / 2;
    float *pt = kmax > 1 ? reinterpret_cast<float *>(static_cast<char *>(ws) + 2 * part) : nullptr;
    int *arrive = coop ? reinterpret_cast<int *>(static_cast<char *>(ws) + 2 * part + partials) : nullptr;
    CUtensorMap hmap, lmap;
    std::memset(&hmap, 0, sizeof(hmap));
    std::memset(&lmap, 0, sizeof(lmap));
    if (!make_part_map(&hmap, hi, ldw, batch, f.cols, KW) || !make_part_map(&lmap, lo, ldw, batch, f.cols, KW)) {
        cudaFreeAsync(ws, stream);
        return cudaErrorNotSupported;
    }
    const int64_t items = f.cols * ((batch + 3) / 4);
    if (items >= (int64_t(1) << 30)) {   // 16 GB of X and more: the CUDA-core path
        cudaFreeAsync(ws, stream);
        return cudaErrorNotSupported;
    }
    const int64_t per_cta = 256 * kSplitItems;
    const unsigned sgrid = static_cast<unsigned>(std::max<int64_t>(1, std::min<int64_t>((items + per_cta - 1) / per_cta,
                                                                                      int64_t(sm_count()) * 8)));
    e = launch_ex(split_kernel, dim3(sgrid), dim3(256), 0, stream, 1, true, X, ldx, batch, f.cols, hi, lo, ldw,
                  arrive, static_cast<int>(counters / 4));
    if (e == cudaSuccess && coop) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(T * coop_split), static_cast<unsigned>(NT));
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = p.smem;
        cfg.stream = stream;
        cudaLaunchAttribute attr[2];
        attr[0].id = cudaLaunchAttributeCooperative;
        attr[0].val.cooperative = 1;
        attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[1].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = pdl_enabled() ? 2 : 1;
        e = cudaLaunchKernelEx(&cfg, tc_kernel<KW>, hmap, lmap, f, coop_split, p.nstages, p.N, batch, Y, ldy, pt,
                               arrive, early ? 1 : 0);
        if (e != cudaSuccess) {   // not launchable cooperatively here: the cluster split instead
            cudaGetLastError();
            e = cudaSuccess;
            arrive = nullptr;
        } else {
            ksplit = 0;   // launched
        }
    }
    if (e == cudaSuccess && ksplit > 0) {
        const dim3 grid(static_cast<unsigned>(T * ksplit), static_cast<unsigned>(NT));
        e = launch_ex(tc_kernel<KW>, grid, dim3(kThreads), p.smem, stream, static_cast<unsigned>(ksplit), true, hmap,
                      lmap, f, ksplit, p.nstages, p.N, batch, Y, ldy, pt, static_cast<int *>(nullptr),
                      early ? 1 : 0);
    }
    const cudaError_t ef = cudaFreeAsync(ws, stream);
    return e != cudaSuccess ? e : ef;
}

// cudaErrorNotSupported when the call does not fit this path (fp32 weights);
// the caller then takes the CUDA-core path.  The split of X lives in
// stream-ordered workspace from the device's default memory pool, taken and
// returned on `stream` around the two kernels.
inline cudaError_t launch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy,
                          bool early, cudaStream_t stream) {
    if (!f.bf16 || f.ngroups <= 0 || f.cols > (int64_t(1) << 31) - 1) return cudaErrorNotSupported;
    const Plan p = plan_for(tile_width(batch));
    return p.KW == 64 ? launch_kw<64>(f, X, ldx, batch, Y, ldy, early, p, stream)
                      : launch_kw<32>(f, X, ldx, batch, Y, ldy, early, p, stream);
}

}  // namespace tc
}  // namespace darb
