// tc.cuh -- Y = W_darb X on the tensor cores (tcgen05, kind::f16) for bf16
// weights and wide batches.
//
// Past a few dozen batch columns the CUDA-core product is bound by gathering
// one activation operand from shared memory per (kept weight, column) pair.
// This kernel instead densifies a slice of W_darb in shared memory and hands
// the contraction to the tensor cores: the zeros cost m times the multiplies
// of the sparse product, but a GB300 SM does them far faster than it can
// gather.
//
// Work unit: 256 rows (eight consecutive 32-row groups, any block sizes) x
// one batch tile of N = 32..256 columns x one cluster rank's share of the
// columns of W.  The rank walks its share in stages of 32 columns:
//  * a TMA warp copies the activation rows, X[k0 .. k0+32R) for the batch
//    tile, into a ring of 32 KB fp32 staging slots, each holding R = 256/N
//    stages (rows and columns past the ends read as zeros): about 64-96 KB of
//    activations stay in flight per SM whatever the tile width;
//  * four converter warps split the staged activations into two bf16 parts,
//    x = hi + lo, written as two MN-major B tiles (128-byte swizzle);
//  * eight producer warps (one thread per row; a warp is one 32-row group,
//    so all its lanes share a block size and walk the blocks in lockstep)
//    zero the row's 64 bytes of the stage and write the row's kept values
//    that fall in it (bf16, exact) into two 128 x 32 A tiles (K-major,
//    64-byte swizzle); for m >= 16 at most three blocks meet a stage and
//    are decoded in straight-line code;
//  * an MMA warp issues, per stage and 128-row half, A*B_hi + A*B_lo for two
//    K=16 steps into that half's TMEM accumulator (128 lanes x N fp32
//    columns) and releases the stage with tcgen05.commit.
// At the end the ranks of a cluster add their partial accumulators: each rank
// owns a slice of the rows, every rank stores its partial rows of that slice
// into the owner's shared memory (distributed shared memory, no waiting on
// remote loads), and the owner adds them in rank order (deterministic) and
// writes its rows of Y.
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

#include <cstring>

namespace darb {
namespace tc {

namespace cg = cooperative_groups;

constexpr int kRows = 256;                       // rows per CTA
constexpr int kCtaGroups = kRows / kSlots;       // 32-row groups per CTA
constexpr int kK = 32;                           // columns of W per stage
constexpr int kProducerWarps = 8;                // kept values -> A, one thread per row
constexpr int kConverterWarps = 12;              // staged activations -> B_hi, B_lo
constexpr int kConverters = kConverterWarps * 32;
constexpr int kTmaWarp = kProducerWarps + kConverterWarps;   // activation copies
constexpr int kMmaWarp = kTmaWarp + 1;           // TMEM owner, MMA issue
constexpr int kThreads = (kMmaWarp + 1) * 32;
constexpr int kARow = kK * 2;                    // bytes of one A row (bf16, 64-byte swizzle)
constexpr int kAHalf = 128 * kARow;              // one 128-row A tile
constexpr int kMaxStages = 6;
constexpr int kMaxX = 3;
constexpr int kXSlot = 32 * 1024;                // bytes of one staging slot
constexpr int kStageOff = 1024;                  // after the barriers; 1024-byte aligned
constexpr size_t kSmemLimit = 227 * 1024;

static_assert(kStageOff % 1024 == 0, "stages must start on a swizzle-atom boundary");

// One bf16 B tile: 64-column x 8-row atoms of 1 KB, four K groups per 64 columns.
__host__ __device__ constexpr int b_tile_bytes(int N) { return (N + 63) / 64 * 4096; }
// An MMA stage: the two A halves, B_hi and B_lo.
__host__ __device__ constexpr int mma_stage_bytes(int N) { return 2 * kAHalf + 2 * b_tile_bytes(N); }
// Stages per staging slot: a slot holds 32 columns x 32R rows per 32-column box.
__host__ __device__ constexpr int x_stages(int N) { return kXSlot / (N * kK * 4); }

__host__ __device__ constexpr uint32_t tmem_cols(int N) { return 2 * N < 32 ? 32u : uint32_t(2 * N); }

struct Plan {
    int N;          // batch tile width: 32, 64, 128 or 256
    int nstages;    // MMA stages in the ring
    int nx;         // staging slots in the ring
    int prows;      // rows of the partial-sum buffer per reduction round (256 or 128)
    size_t smem;    // dynamic shared memory, including 1024 bytes of alignment slack
};

inline Plan plan_for(int N) {
    Plan p{};
    p.N = N;
    const size_t budget = kSmemLimit - 1024 - kStageOff;
    // three staging slots when that leaves room for four MMA stages, else two
    p.nx = size_t(4) * mma_stage_bytes(N) + size_t(kMaxX) * kXSlot <= budget ? kMaxX : 2;
    p.nstages = static_cast<int>((budget - size_t(p.nx) * kXSlot) / mma_stage_bytes(N));
    if (p.nstages > kMaxStages) p.nstages = kMaxStages;
    const size_t area = size_t(p.nstages) * mma_stage_bytes(N) + size_t(p.nx) * kXSlot;
    // the partial-sum buffer holds ksplit * ceil(prows / ksplit) <= prows + 7 rows
    p.prows = size_t(kRows + 8) * (N + 4) * 4 <= area ? kRows : 128;
    p.smem = 1024 + kStageOff + area;
    return p;
}

// An A tile row r (0..127) starts at a_row(r); kept value column p (0..31)
// of it sits at a_row(r) + ((2p) ^ a_swz(r)): 2p is the byte offset, whose
// 16-byte chunk bits the 64-byte swizzle XORs with (r / 2) % 4.
__device__ __forceinline__ int a_row(int r) { return (r >> 3) * 512 + (r & 7) * kARow; }
__device__ __forceinline__ int a_swz(int r) { return ((r >> 1) & 3) << 4; }

__device__ __forceinline__ uint32_t pack_hi_lo(float a, float b, uint32_t *lo) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    const __nv_bfloat162 l = __floats2bfloat162_rn(a - __low2float(h), b - __high2float(h));
    *lo = *reinterpret_cast<const uint32_t *>(&l);
    return *reinterpret_cast<const uint32_t *>(&h);
}

__global__ void __launch_bounds__(kThreads, 1)
tc_kernel(const __grid_constant__ CUtensorMap xmap, Format f, int ksplit, int nstages, int nx, int N, int prows,
          int64_t batch, float *Y, int64_t ldy, int early) {
    extern __shared__ unsigned char sm_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) &
                                                          ~uintptr_t(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(sm);     // MMA stage written (producers, converters)
    uint64_t *empty = full + kMaxStages;                   // MMA stage consumed (commit)
    uint64_t *xfull = empty + kMaxStages;                  // staging slot landed (TMA)
    uint64_t *xempty = xfull + kMaxX;                      // staging slot converted (converters)
    uint64_t *done = xempty + kMaxX;
    uint32_t *s_tmem = reinterpret_cast<uint32_t *>(done + 1);
    unsigned char *const stages = sm + kStageOff;
    const int sbytes = mma_stage_bytes(N), bbytes = b_tile_bytes(N);
    unsigned char *const xring = stages + size_t(nstages) * sbytes;
    const int R = x_stages(N);                             // stages per staging slot
    const int xbox = R * kK * 128;                         // bytes of one 32-column box of a slot

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
            mbar_init(&full[s], kProducerWarps + kConverterWarps);
            mbar_init(&empty[s], 1);
        }
        for (int x = 0; x < kMaxX; ++x) {
            mbar_init(&xfull[x], 1);
            mbar_init(&xempty[x], kConverterWarps);
        }
        mbar_init(done, 1);
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(s_tmem, tcols);
        tmem_relinquish();
    }
    if (warp == kTmaWarp && lane == 0) prefetch_tensormap(&xmap);
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem = *s_tmem;
    bool ok = true;

    if (warp < kProducerWarps) {
        // ---- producers: thread t owns row t of the CTA (half t / 128 of the tile);
        // warp w is group tile*8 + w, so m is uniform across the warp
        if (!early) pdl_wait_previous();
        const int t = tid, r = t & 127;
        const int g = tile * kCtaGroups + warp;
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
        // blocks of this rank's first stage start at jb = floor(k0 / m), rem = k0 - jb*m;
        // each next stage moves k0 by 32 = q32*m + r32
        const int k0first = ks0 * kK;
        int jb = k0first / m, rem = k0first - jb * m;
        const int q32 = kK / m, r32 = kK - q32 * m;
        // chunk cc in (cv, co), cc+1 and cc+2 prefetched
        int cc = jb >> 3;
        uint4 cv = make_uint4(0, 0, 0, 0), v1 = cv, v2 = cv;
        uint2 co = make_uint2(0, 0), o1 = co, o2 = co;
        load_chunk(cc, cv, co);
        load_chunk(cc + 1, v1, o1);
        load_chunk(cc + 2, v2, o2);
        unsigned char *const row0 = stages + (t >> 7) * kAHalf + a_row(r);   // this row in stage 0
        const int swz = a_swz(r);
        auto value = [](const uint4 &v, int q) -> uint16_t {
            const uint32_t w = (q >> 1) == 0 ? v.x : (q >> 1) == 1 ? v.y : (q >> 1) == 2 ? v.z : v.w;
            return static_cast<uint16_t>((q & 1) ? w >> 16 : w);
        };
        auto offset = [nib](const uint2 &o, int q) -> uint32_t {
            return nib ? (o.x >> (4 * q)) & 15u : ((q < 4 ? o.x : o.y) >> (8 * (q & 3))) & 255u;
        };
        int s = 0;
        uint32_t phase = 0;   // parity of the current use of stage s
        for (int it = 0; it < nst; ++it) {
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
                // blocks jb, jb+1, jb+2 (in chunk cc or cc+1) cover the stage
#pragma unroll
                for (int b = 0; b < 3; ++b) {
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
                    if ((j >> 3) != cc) {   // step into the next chunk, prefetch two ahead
                        cc = j >> 3;
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
            jb += q32;
            rem += r32;
            if (rem >= m) {
                rem -= m;
                ++jb;
            }
            if (m >= 16 && (jb >> 3) != cc) {   // at most one chunk per stage when m >= 16
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
            if (++s == nstages) {
                s = 0;
                phase ^= 1u;
            }
        }
    } else if (warp < kTmaWarp) {
        // ---- converters: staged fp32 (32-column boxes) -> B_hi, B_lo (64-column atoms)
        const int ct = tid - kProducerWarps * 32;
        const int units = N * (kK / 8);   // (row k of the stage, 8 batch columns)
        int s = 0, x = 0, sub = 0;
        uint32_t phase = 0, xphase = 0;
        for (int it = 0; it < nst; ++it) {
            if (it >= nstages && !__all_sync(0xFFFFFFFFu, mbar_wait(&empty[s], phase ^ 1u, false))) {
                ok = false;
                break;
            }
            if (!__all_sync(0xFFFFFFFFu, mbar_wait(&xfull[x], xphase, false))) {
                ok = false;
                break;
            }
            const unsigned char *xs = xring + size_t(x) * kXSlot + sub * (kK * 128);
            unsigned char *bhi = stages + size_t(s) * sbytes + 2 * kAHalf, *blo = bhi + bbytes;
            for (int u = ct; u < units; u += kConverters) {
                const int k = u & (kK - 1), nc = u >> 5;   // lanes: consecutive rows k, conflict-free
                const unsigned char *src = xs + (nc >> 2) * xbox + k * 128;
                const int c4 = (nc & 3) * 2;
                const float4 a4 = *reinterpret_cast<const float4 *>(src + ((c4 ^ (k & 7)) << 4));
                const float4 b4 = *reinterpret_cast<const float4 *>(src + (((c4 + 1) ^ (k & 7)) << 4));
                uint4 hv, lv;
                hv.x = pack_hi_lo(a4.x, a4.y, &lv.x);
                hv.y = pack_hi_lo(a4.z, a4.w, &lv.y);
                hv.z = pack_hi_lo(b4.x, b4.y, &lv.z);
                hv.w = pack_hi_lo(b4.z, b4.w, &lv.w);
                const int off = (nc >> 3) * 4096 + (k >> 3) * 1024 + (k & 7) * 128 + (((nc & 7) ^ (k & 7)) << 4);
                *reinterpret_cast<uint4 *>(bhi + off) = hv;
                *reinterpret_cast<uint4 *>(blo + off) = lv;
            }
            fence_proxy_async_smem();   // the tensor core reads B through the async proxy
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&full[s]);
                if (sub == R - 1 || it == nst - 1) mbar_arrive(&xempty[x]);
            }
            if (++s == nstages) {
                s = 0;
                phase ^= 1u;
            }
            if (++sub == R) {
                sub = 0;
                if (++x == nx) {
                    x = 0;
                    xphase ^= 1u;
                }
            }
        }
    } else if (warp == kTmaWarp) {
        // ---- activation rows into the staging ring, R stages per slot
        if (lane == 0) {
            pdl_wait_previous();   // X may come from the previous kernel
            const int nslots = (nst + R - 1) / R;
            int x = 0;
            uint32_t xphase = 0;
            for (int sl = 0; sl < nslots; ++sl) {
                if (sl >= nx && !mbar_wait(&xempty[x], xphase ^ 1u, false)) {
                    ok = false;
                    break;
                }
                unsigned char *xs = xring + size_t(x) * kXSlot;
                mbar_arrive_expect_tx(&xfull[x], static_cast<uint32_t>(kXSlot));
                for (int b = 0; b < N / 32; ++b)
                    tensor2d_g2s(xs + b * xbox, &xmap, static_cast<int>(n0) + 32 * b, (ks0 + sl * R) * kK, &xfull[x]);
                if (++x == nx) {
                    x = 0;
                    xphase ^= 1u;
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
        const uint64_t a0 = smem_desc(sa0, 16, 512, kLayoutSw64);
        const uint64_t bh0 = smem_desc(sa0 + 2 * kAHalf, 4096, 1024, kLayoutSw128);
        const uint64_t bl0 = smem_desc(sa0 + 2 * kAHalf + bbytes, 4096, 1024, kLayoutSw128);
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
    if (warp < kProducerWarps) {
        if (!__all_sync(0xFFFFFFFFu, mbar_wait(done, 0, false))) ok = false;
        tc_fence_after_sync();
    }
    pdl_wait_previous();   // Y may still be read by the previous kernel
    const bool vec = (ldy & 3) == 0 && (reinterpret_cast<uintptr_t>(Y) & 15) == 0;
    if (ksplit == 1) {
        if (warp < kProducerWarps) {
            const int g = tile * kCtaGroups + warp;
            const int64_t row = g < f.ngroups ? f.rowmap[g * kSlots + lane] : -1;
            const uint32_t tl = tmem + (uint32_t(32 * (warp & 3)) << 16) + uint32_t((warp >> 2) * N);
#pragma unroll 1
            for (int cb = 0; cb < N / 32; ++cb) {   // 32 registers of accumulator at a time
                uint32_t v[32];
                tmem_ld32(tl + cb * 32, v);
                tmem_ld_wait();
                const int64_t c0 = n0 + cb * 32;
                if (row >= 0 && c0 < batch) {
                    float *y = Y + row * ldy + c0;
                    const int64_t cnt = batch - c0;
                    if (vec && cnt >= 32) {
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            reinterpret_cast<float4 *>(y)[i] =
                                make_float4(__uint_as_float(v[4 * i]), __uint_as_float(v[4 * i + 1]),
                                            __uint_as_float(v[4 * i + 2]), __uint_as_float(v[4 * i + 3]));
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (i < cnt) y[i] = __uint_as_float(v[i]);
                    }
                }
            }
        }
    } else {
        cg::cluster_group cluster = cg::this_cluster();
        float *P = reinterpret_cast<float *>(stages);   // [source rank][owned row][pst]; free once all MMAs are done
        const int pst = N + 4;                          // padded row stride: conflict-free stores
        const int rounds = kRows / prows;
        const int own = (prows + ksplit - 1) / ksplit;  // rows each rank owns per round
        const int nq = N / 4;
        cluster.sync();   // every rank's MMAs are done: the stage rings may be overwritten
        for (int round = 0; round < rounds; ++round) {
            if (warp < kProducerWarps && (prows == kRows || (warp >> 2) == round)) {
                const int prow = (prows == kRows ? warp * 32 : (warp & 3) * 32) + lane;   // row of the round
                const int owner = prow / own;
                const uint32_t dst = cluster_addr(smem_addr(P + (rank * own + (prow - owner * own)) * pst),
                                                  static_cast<uint32_t>(owner));
                const uint32_t tl = tmem + (uint32_t(32 * (warp & 3)) << 16) + uint32_t((warp >> 2) * N);
#pragma unroll 1
                for (int cb = 0; cb < N / 32; ++cb) {   // 32 registers of accumulator at a time
                    uint32_t v[32];
                    tmem_ld32(tl + cb * 32, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        st_cluster_v4(dst + (cb * 32 + 4 * i) * 4, v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                }
            }
            cluster.sync();   // the partial rows have landed in their owners
            const int r0 = rank * own, r1 = min(prows, r0 + own);
#pragma unroll 1
            for (int e = tid; e < (r1 - r0) * nq; e += kThreads) {
                const int pr = e / nq, c4 = e % nq;
                const float4 *src4 = reinterpret_cast<const float4 *>(P + pr * pst) + c4;
                const int sstride = own * pst / 4;   // float4s between two sources' copies of the row
                float4 acc = src4[0];
#pragma unroll 1
                for (int s0 = 1; s0 < ksplit; s0 += 4) {   // four loads in flight, added in rank order
                    float4 v[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (s0 + i < ksplit) v[i] = src4[(s0 + i) * sstride];
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (s0 + i < ksplit) {
                            acc.x += v[i].x;
                            acc.y += v[i].y;
                            acc.z += v[i].z;
                            acc.w += v[i].w;
                        }
                }
                const int crow = (prows == kRows ? 0 : round * 128) + r0 + pr;   // row of the CTA
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
            cluster.sync();   // the owner has read its buffer before the next round refills it
        }
    }

    if (!ok) atomicOr(f.status, kStatusTimeout);
    tc_fence_before_sync();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after_sync();
        tmem_dealloc(tmem, tcols);
    }
}

// Tensor map over X (cols x batch fp32, row pitch ldx floats) with boxes of
// 32 columns x 32R rows and 128-byte swizzle; false if X cannot be described
// (alignment).
inline bool make_xmap(CUtensorMap *map, const float *X, int64_t ldx, int64_t batch, int64_t cols, int N) {
    if (X == nullptr || reinterpret_cast<uintptr_t>(X) % 16 != 0 || (ldx * 4) % 16 != 0) return false;
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (enc == nullptr) return false;
    const cuuint64_t dims[2] = {cuuint64_t(batch), cuuint64_t(cols)};
    const cuuint64_t strides[1] = {cuuint64_t(ldx) * 4};
    const cuuint32_t box[2] = {32, cuuint32_t(kK * x_stages(N))};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(X), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

inline int tile_width(int64_t batch) {
    int N = 32;
    while (N < 256 && N < batch) N <<= 1;
    return N;
}

// Clusters of `ksplit` CTAs of this kernel that can be resident at once (0 if unknown).
inline int active_clusters(int ksplit, const Plan &p) {
    static int cache[4][9] = {};
    const int wi = p.N == 32 ? 0 : p.N == 64 ? 1 : p.N == 128 ? 2 : 3;
    if (cache[wi][ksplit] != 0) return cache[wi][ksplit];
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
    if (cudaOccupancyMaxActiveClusters(&n, tc_kernel, &cfg) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
    }
    if (n <= 0) n = -1;
    cache[wi][ksplit] = n;
    return n;
}

// Cluster split: fewest waves per unit of work, i.e. the smallest
// ceil(units / resident clusters) / ksplit, never more ranks than stages.
inline int pick_split(int64_t units, int KS, const Plan &p) {
    int best = 1;
    double best_cost = 1e30;
    for (int s = 1; s <= 8 && s <= KS; ++s) {
        int act = active_clusters(s, p);
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

// cudaErrorNotSupported when the call does not fit this kernel (fp32 weights,
// X not describable by a tensor map); the caller then takes the CUDA-core path.
inline cudaError_t launch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy,
                          bool early, cudaStream_t stream) {
    if (!f.bf16 || f.ngroups <= 0) return cudaErrorNotSupported;
    CUtensorMap xmap;
    std::memset(&xmap, 0, sizeof(xmap));
    const Plan p = plan_for(tile_width(batch));
    if (!make_xmap(&xmap, X, ldx, batch, f.cols, p.N)) return cudaErrorNotSupported;
    static const cudaError_t a = [] {
        size_t most = 0;
        for (int w = 32; w <= 256; w *= 2) most = plan_for(w).smem > most ? plan_for(w).smem : most;
        return allow_smem(tc_kernel, most);
    }();
    if (a != cudaSuccess) return a;
    const int T = (f.ngroups + kCtaGroups - 1) / kCtaGroups;
    const int64_t NT = (batch + p.N - 1) / p.N;
    const int KS = static_cast<int>((f.cols + kK - 1) / kK);
    const int ksplit = pick_split(int64_t(T) * NT, KS, p);
    const dim3 grid(static_cast<unsigned>(T * ksplit), static_cast<unsigned>(NT));
    return launch_ex(tc_kernel, grid, dim3(kThreads), p.smem, stream, static_cast<unsigned>(ksplit), true, xmap, f,
                     ksplit, p.nstages, p.nx, p.N, p.prows, batch, Y, ldy, early ? 1 : 0);
}

}  // namespace tc
}  // namespace darb
