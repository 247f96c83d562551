// spmm_batch.cu -- y = W_darb X for batch > 4 (Sec. 3.2, Fig. 6(b)).
//
// Work unit: a row set (up to 8 consecutive 32-row groups of one block-size
// bin, so up to 256 rows), one cluster rank's share of the blocks, and one
// batch tile of 4*LPR columns.  The rank's blocks are walked in rounds.  Per
// round one thread starts the bulk (TMA) copies of the round's kept values and
// packed offsets (one contiguous run per group) and the 2-D tensor copies of
// the activation rows those blocks can select, X[j*m .. j*m+m) for the batch
// tile (out-of-range rows and columns arrive as zeros).  Then LPR lanes share
// a row and each lane owns 4 batch columns: a selected activation row is one
// 16*LPR-byte shared-memory read, and each kept value is reused across the
// tile's columns from registers.  A thread keeps its rows' partial sums in
// registers across rounds; at the end the ranks add their partial sums
// through distributed shared memory in a fixed order (deterministic), each
// rank finishing a slice of the rows and writing Y.
//
// Why row sets: an activation row staged in shared memory is selected by about
// rows/m of the set's rows, so staging traffic per FMA is 4*m/rows bytes;
// 256 rows keep it well under the on-chip bandwidth for the block sizes the
// paper uses.
#include "kernels_common.cuh"
#include "launch.cuh"
#include "tma.cuh"

#include <cooperative_groups.h>
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>

namespace cg = cooperative_groups;

namespace darb {
namespace {

constexpr int kXcapB = 8192;      // activation floats per round
constexpr int kXslack = 1024;     // room for the last tensor box of a round to run past it
constexpr int kXstage = kXcapB + kXslack;
constexpr int kRecCap = 16;       // (group, chunk) records staged per round
constexpr int kStages = 2;        // rounds in flight per CTA
constexpr int kConsumers = 8;     // consumer warps; one more warp produces
constexpr int kBatchThreads = (kConsumers + 1) * 32;

// Lanes per row LPR, columns per lane CPL: the batch tile is LPR*CPL columns.
// Wide tiles keep fewer rows per set so that the accumulators fit in registers.
template <int LPR, int CPL>
__host__ __device__ constexpr int max_set_groups() { return CPL == 8 ? 4 : 8; }

template <int LPR, int CPL>
__host__ __device__ constexpr int box_rows() { return kXslack / (LPR * CPL); }

template <bool BF16>
__host__ __device__ constexpr size_t stage_val_bytes() { return size_t(kRecCap) * kSlots * kChunk * (BF16 ? 2 : 4); }

constexpr size_t kStageOffBytes = size_t(kRecCap) * kSlots * 2 * 4;

template <bool BF16>
__host__ __device__ constexpr size_t batch_smem() {
    return 128 + kStages * (size_t(kXstage) * 4 + stage_val_bytes<BF16>() + kStageOffBytes);
}

// One chunk (8 blocks) of one row slot: decode the offsets and add the 8 kept
// values times their selected activation rows into acc.  NIB (4-bit offsets)
// and WHOLE (all 8 blocks inside the round) are compile-time so that the
// innermost loop is just offset extraction, one address, the loads and FMAs.
template <bool BF16, bool NIB, bool WHOLE, int KQ, int LPR>
__device__ __forceinline__ void batch_chunk(const unsigned char *s_vals, const uint32_t *s_offs, int rec,
                                            const float4 *xb, int m, int row_f4, int e_lo, int e_hi,
                                            float4 (&acc)[KQ]) {
    float v[kChunk];
    if constexpr (BF16) {
        const uint4 w4 = *reinterpret_cast<const uint4 *>(s_vals + size_t(rec) * 16);
        const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            v[2 * e] = __uint_as_float(w[e] << 16);
            v[2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
        }
    } else {
        const float4 *pv = reinterpret_cast<const float4 *>(s_vals + size_t(rec) * 32);
        const float4 x0 = pv[0], x1 = pv[1];
        v[0] = x0.x; v[1] = x0.y; v[2] = x0.z; v[3] = x0.w;
        v[4] = x1.x; v[5] = x1.y; v[6] = x1.z; v[7] = x1.w;
    }
    uint2 ow;
    if constexpr (NIB) ow = make_uint2(s_offs[rec], 0u);
    else ow = reinterpret_cast<const uint2 *>(s_offs)[rec];
    const int mstride = m * row_f4;
#pragma unroll
    for (int e = 0; e < kChunk; ++e) {
        if (WHOLE || (e >= e_lo && e < e_hi)) {
            int off;
            if constexpr (NIB) off = int((ow.x >> (4 * e)) & 15u);
            else off = int(((e < 4 ? ow.x : ow.y) >> (8 * (e & 3))) & 255u);
            const float4 *xr = xb + e * mstride + off * row_f4;
#pragma unroll
            for (int u = 0; u < KQ; ++u) {
                const float4 xv = xr[u * LPR];
                acc[u].x = fmaf(v[e], xv.x, acc[u].x);
                acc[u].y = fmaf(v[e], xv.y, acc[u].y);
                acc[u].z = fmaf(v[e], xv.z, acc[u].z);
                acc[u].w = fmaf(v[e], xv.w, acc[u].w);
            }
        }
    }
}

template <bool BF16, int LPR, int CPL>
__global__ void __launch_bounds__(kBatchThreads)
spmm_batch(Format f, const int2 *__restrict__ sets, const float *__restrict__ X, int64_t ldx, int64_t batch,
           float *__restrict__ Y, int64_t ldy, const __grid_constant__ CUtensorMap xmap, int use_tma,
           int early) {
    constexpr int kBt = LPR * CPL;        // batch tile
    constexpr int kQ = CPL / 4;           // float4 per lane
    constexpr int kRpw = 32 / LPR;        // rows per consumer warp at a time
    constexpr int kRptMax = max_set_groups<LPR, CPL>() * kSlots / (kConsumers * kRpw);
    constexpr int kBoxRows = box_rows<LPR, CPL>();
    constexpr int kEsz = BF16 ? 2 : 4;
    extern __shared__ __align__(128) unsigned char sm[];
    // layout: full[kStages] empty[kStages] | X stages | values stages | offsets stages
    uint64_t *full = reinterpret_cast<uint64_t *>(sm);
    uint64_t *empty = full + kStages;
    float *s_x0 = reinterpret_cast<float *>(sm + 128);
    unsigned char *s_v0 = sm + 128 + size_t(kStages) * kXstage * 4;
    unsigned char *s_o0 = s_v0 + kStages * stage_val_bytes<BF16>();

    pdl_launch_dependents();
    cg::cluster_group cluster = cg::this_cluster();
    const int ksc = static_cast<int>(cluster.num_blocks());
    const int q = static_cast<int>(cluster.block_rank());
    const int2 set = sets[blockIdx.x / ksc];
    const int ng = set.y;
    const Group g0 = f.groups[set.x];
    const int m = g0.m, n = g0.n, rw = g0.nib ? 1 : 2;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t b0 = int64_t(blockIdx.y) * kBt;
    const int nch = (n + kChunk - 1) / kChunk;
    const int cpc = (nch + ksc - 1) / ksc;
    const int c0 = min(nch, q * cpc), c1 = min(nch, c0 + cpc);
    const int J0 = c0 * kChunk, J1 = min(n, c1 * kChunk);
    // blocks per round: bounded by the activation tile and by the staged records
    const int rb = max(1, min(kXcapB / (m * kBt), (kRecCap / ng - 1) * kChunk));
    const int rounds = (J1 - J0 + rb - 1) / rb;

    if (tid == 0) {
        for (int st = 0; st < kStages; ++st) {
            mbar_init(&full[st], 1);
            mbar_init(&empty[st], kConsumers);
        }
        fence_mbar_init();
    }
    __syncthreads();

    struct Round { int jr0, jr1, cr0, nchr, kx0, kr; };
    auto round_geo = [&](int r) {
        Round g;
        g.jr0 = J0 + r * rb;
        g.jr1 = min(J1, g.jr0 + rb);
        g.cr0 = g.jr0 / kChunk;
        g.nchr = (g.jr1 + kChunk - 1) / kChunk - g.cr0;
        g.kx0 = g.jr0 * m;
        const int64_t kxe = int64_t(g.jr1) * m;
        g.kr = static_cast<int>((kxe < f.cols ? kxe : f.cols) - g.kx0);
        return g;
    };
    // Round r's copies into stage st (producer lane 0).  The handle part (kept
    // values and offsets, one contiguous run per group) may go before the PDL
    // wait; the activation part only after it.  Exactly one arrival per round
    // closes full[st] together with the transferred bytes.
    auto issue = [&](int r, int st, bool handle, bool xpart) {
        const Round g = round_geo(r);
        const uint32_t bv = uint32_t(g.nchr) * kSlots * kChunk * kEsz;
        const uint32_t bo = uint32_t(g.nchr) * kSlots * rw * 4;
        const int nbox = (g.kr + kBoxRows - 1) / kBoxRows;
        const uint32_t hbytes = handle ? uint32_t(ng) * (bv + bo) : 0u;
        const uint32_t xbytes = (xpart && use_tma) ? uint32_t(nbox) * kBoxRows * kBt * 4 : 0u;
        if (xpart) mbar_arrive_expect_tx(&full[st], hbytes + xbytes);
        else mbar_expect_tx(&full[st], hbytes);
        if (handle)
            for (int gi = 0; gi < ng; ++gi) {
                const Group gg = f.groups[set.x + gi];
                bulk_g2s(s_v0 + st * stage_val_bytes<BF16>() + size_t(gi) * bv,
                         static_cast<const unsigned char *>(f.vals) +
                             (size_t(gg.val_off) + size_t(g.cr0) * kSlots * kChunk) * kEsz,
                         bv, &full[st]);
                bulk_g2s(s_o0 + st * kStageOffBytes + size_t(gi) * bo,
                         f.offs + gg.off_off + size_t(g.cr0) * kSlots * rw, bo, &full[st]);
            }
        if (xpart && use_tma)
            for (int i = 0; i < nbox; ++i)
                tensor2d_g2s(s_x0 + size_t(st) * kXstage + size_t(i) * kBoxRows * kBt, &xmap, int(b0),
                             g.kx0 + i * kBoxRows, &full[st]);
    };
    // X without a tensor map: the producer warp loads round r's tile itself
    auto load_x_plain = [&](int r, int st) {
        const Round g = round_geo(r);
        float *s_x = s_x0 + size_t(st) * kXstage;
        const int nx = g.kr * kBt;
        for (int base = 0; base < nx; base += 8 * 32) {
            float tmp[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int idx = base + u * 32 + lane;
                const int kk = idx / kBt, t = idx % kBt;
                tmp[u] = (idx < nx && b0 + t < batch) ? __ldg(X + int64_t(g.kx0 + kk) * ldx + b0 + t) : 0.0f;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int idx = base + u * 32 + lane;
                if (idx < nx) s_x[idx] = tmp[u];
            }
        }
        __threadfence_block();
        __syncwarp();
    };

    bool ok = true;
    const int pre = min(rounds, kStages);
    if (warp == kConsumers) {
        // ---------------- producer warp
        if (early && lane == 0)
            for (int r = 0; r < pre; ++r) issue(r, r, true, false);
        pdl_wait_previous();
        for (int r = 0; r < rounds && ok; ++r) {
            const int st = r % kStages;
            if (r >= kStages) {
                // the consumers have released this stage's previous round
                ok = mbar_wait(&empty[st], ((r / kStages) - 1) & 1);
                ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
                if (!ok) break;
                if (lane == 0) fence_proxy_async_smem();
            }
            if (!use_tma) load_x_plain(r, st);
            if (lane == 0) issue(r, st, !(early && r < kStages), true);
        }
        if (!ok && lane == 0) atomicOr(f.status, kStatusTimeout);
    } else {
        pdl_wait_previous();
    }

    // ---------------- consumer warps: thread = (row slot, column quad)
    const int qd = lane % LPR, rr = lane / LPR;
    float4 acc[kRptMax][kQ];
#pragma unroll
    for (int p = 0; p < kRptMax; ++p)
#pragma unroll
        for (int u = 0; u < kQ; ++u) acc[p][u] = make_float4(0.f, 0.f, 0.f, 0.f);
    const int rpt = (ng * kSlots + kConsumers * kRpw - 1) / (kConsumers * kRpw);
    uint32_t valid_mask = 0u;
    if (warp < kConsumers) {
#pragma unroll
        for (int p = 0; p < kRptMax; ++p) {
            const int s = warp * kRpw + rr + p * kConsumers * kRpw;
            const int gi = s / kSlots;
            if (p < rpt && gi < ng && (s % kSlots) < f.groups[set.x + gi].nrows) valid_mask |= 1u << p;
        }
        for (int r = 0; r < rounds && ok; ++r) {
            const int st = r % kStages;
            ok = mbar_wait(&full[st], (r / kStages) & 1);
            ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
            if (!ok) break;
            const Round g = round_geo(r);
            const float4 *sx4 = reinterpret_cast<const float4 *>(s_x0 + size_t(st) * kXstage);
            const unsigned char *s_vals = s_v0 + st * stage_val_bytes<BF16>();
            const uint32_t *s_offs = reinterpret_cast<const uint32_t *>(s_o0 + st * kStageOffBytes);
            for (int lc = 0; lc < g.nchr; ++lc) {
                const int jc = (g.cr0 + lc) * kChunk;
                // blocks of this chunk inside the round (all 8 except at the round's ends)
                const int e_lo = max(0, g.jr0 - jc), e_hi = min(kChunk, g.jr1 - jc);
                const bool whole = e_lo == 0 && e_hi == kChunk;
                // lane qd owns float4 columns u*LPR + qd: for each u a quarter-warp
                // reads 128 contiguous bytes (no bank conflicts)
                const float4 *xb = sx4 + (jc * m - g.kx0) * (kBt / 4) + qd;
#pragma unroll
                for (int p = 0; p < kRptMax; ++p) {
                    if (valid_mask & (1u << p)) {
                        const int s = warp * kRpw + rr + p * kConsumers * kRpw;
                        const int rec = ((s / kSlots) * g.nchr + lc) * kSlots + (s % kSlots);
                        if (rw == 1) {
                            if (whole)
                                batch_chunk<BF16, true, true, kQ, LPR>(s_vals, s_offs, rec, xb, m, kBt / 4, 0, kChunk, acc[p]);
                            else
                                batch_chunk<BF16, true, false, kQ, LPR>(s_vals, s_offs, rec, xb, m, kBt / 4, e_lo, e_hi, acc[p]);
                        } else {
                            if (whole)
                                batch_chunk<BF16, false, true, kQ, LPR>(s_vals, s_offs, rec, xb, m, kBt / 4, 0, kChunk, acc[p]);
                            else
                                batch_chunk<BF16, false, false, kQ, LPR>(s_vals, s_offs, rec, xb, m, kBt / 4, e_lo, e_hi, acc[p]);
                        }
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[st]);
        }
        if (!ok && lane == 0) atomicOr(f.status, kStatusTimeout);
    }
    __syncthreads();   // every round consumed: the stages are free for the partial sums
    // partial sums of every row slot of the set, slot-major: part[s][0..kBt)
    float *part = s_x0;
    float4 *part4 = reinterpret_cast<float4 *>(part);
    if (warp < kConsumers) {
#pragma unroll
        for (int p = 0; p < kRptMax; ++p) {
            const int s = warp * kRpw + rr + p * kConsumers * kRpw;
            if (p < rpt && s < ng * kSlots)
#pragma unroll
                for (int u = 0; u < kQ; ++u) part4[s * (kBt / 4) + u * LPR + qd] = acc[p][u];
        }
    }
    __syncthreads();
    if (ksc > 1) cluster.sync();
    // rank q finishes rows [s0, s1) of the set for the whole tile
    const int R = ng * kSlots;
    const int per = (R + ksc - 1) / ksc;
    const int s0 = min(R, q * per), s1 = min(R, s0 + per);
    for (int idx = tid; idx < (s1 - s0) * kBt; idx += kBatchThreads) {
        const int s = s0 + idx / kBt, t = idx % kBt;
        const int gi = s / kSlots, slot = s % kSlots;
        if (b0 + t >= batch || slot >= f.groups[set.x + gi].nrows) continue;
        float sum = 0.0f;   // ranks in a fixed order: deterministic
        for (int r = 0; r < ksc; ++r) sum += cluster.map_shared_rank(part, r)[s * kBt + t];
        const int row = f.rowmap[(set.x + gi) * kSlots + slot];
        Y[int64_t(row) * ldy + b0 + t] = sum;
    }
    if (ksc > 1) cluster.sync();
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            cudaGetLastError();
            return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
        }
        return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }();
    return fn;
}

// Tensor map over X (cols rows of `batch` floats, row pitch ldx) with a
// boxr x bt box; false if X cannot be described (alignment).
bool make_xmap(CUtensorMap *map, const float *X, int64_t ldx, int64_t batch, int64_t cols, int bt,
               int boxr) {
    if (reinterpret_cast<uintptr_t>(X) % 16 != 0 || (ldx * 4) % 16 != 0) return false;
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (enc == nullptr) return false;
    const cuuint64_t dims[2] = {cuuint64_t(batch), cuuint64_t(cols)};
    const cuuint64_t strides[1] = {cuuint64_t(ldx) * 4};
    const cuuint32_t box[2] = {cuuint32_t(bt), cuuint32_t(boxr)};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(X), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <bool BF16, int LPR, int CPL>
cudaError_t launch_batch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                         int64_t ldy, bool early, cudaStream_t stream) {
    constexpr int kBt = LPR * CPL;
    constexpr size_t smem = batch_smem<BF16>();
    static const cudaError_t attr = allow_smem(spmm_batch<BF16, LPR, CPL>, smem);
    if (attr != cudaSuccess) return attr;
    CUtensorMap map;
    std::memset(&map, 0, sizeof map);
    const int use_tma = make_xmap(&map, X, ldx, batch, f.cols, kBt, box_rows<LPR, CPL>()) ? 1 : 0;
    const int64_t tiles = (batch + kBt - 1) / kBt;
    const int64_t target = 3 * int64_t(sm_count());   // CTAs wanted
    // largest row sets (most reuse of each staged activation row) that still
    // give enough CTAs with a cluster split of at most 8
    int level = 0;
    for (int l = 3; l >= 0; --l) {
        if ((1 << l) > max_set_groups<LPR, CPL>()) continue;
        level = l;
        if (int64_t(f.nsets[l]) * tiles * 8 >= target) break;
    }
    unsigned ksc = 1;
    while (ksc < 8 && int64_t(f.nsets[level]) * tiles * ksc < target) ksc *= 2;
    const dim3 grid(static_cast<unsigned>(f.nsets[level]) * ksc, static_cast<unsigned>(tiles));
    return launch_ex(spmm_batch<BF16, LPR, CPL>, grid, dim3(kBatchThreads), smem, stream, ksc, true, f,
                     f.sets[level], X, ldx, batch, Y, ldy, map, use_tma, early ? 1 : 0);
}

}  // namespace

cudaError_t launch_spmm_batch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                              int64_t ldy, bool early, cudaStream_t stream) {
    // one block's activation rows (m_max of them) must fit a stage's tile
    if (batch <= 16 || int64_t(f.m_max) * 32 > kXcapB)
        return f.bf16 ? launch_batch<true, 4, 4>(f, X, ldx, batch, Y, ldy, early, stream)
                      : launch_batch<false, 4, 4>(f, X, ldx, batch, Y, ldy, early, stream);
    if (batch <= 32 || int64_t(f.m_max) * 64 > kXcapB)
        return f.bf16 ? launch_batch<true, 8, 4>(f, X, ldx, batch, Y, ldy, early, stream)
                      : launch_batch<false, 8, 4>(f, X, ldx, batch, Y, ldy, early, stream);
    return f.bf16 ? launch_batch<true, 8, 8>(f, X, ldx, batch, Y, ldy, early, stream)
                  : launch_batch<false, 8, 8>(f, X, ldx, batch, Y, ldy, early, stream);
}

}  // namespace darb
