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

constexpr int kXcapB = 8192;      // activation floats per round (before box slack)
constexpr int kBoxRows = 64;      // rows per 2-D tensor copy
constexpr int kRecCap = 32;       // (group, chunk) records staged per round
constexpr int kMaxSetGroups = 8;

template <bool BF16, int LPR>
__host__ __device__ constexpr size_t batch_smem() {
    return 128 + size_t(kXcapB + kBoxRows * 4 * LPR) * 4 + size_t(kRecCap) * kSlots * kChunk * (BF16 ? 2 : 4) +
           size_t(kRecCap) * kSlots * 2 * 4;
}

template <bool BF16, int LPR>
__global__ void __launch_bounds__(kWarps * 32)
spmm_batch(Format f, const int2 *__restrict__ sets, const float *__restrict__ X, int64_t ldx, int64_t batch,
           float *__restrict__ Y, int64_t ldy, const __grid_constant__ CUtensorMap xmap, int use_tma,
           int early) {
    constexpr int kBt = 4 * LPR;          // batch tile
    constexpr int kRpw = 32 / LPR;        // rows per warp at a time
    constexpr int kRptMax = kMaxSetGroups * kSlots / (kWarps * kRpw);
    constexpr int kEsz = BF16 ? 2 : 4;
    extern __shared__ __align__(128) unsigned char sm[];
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm);
    float *s_x = reinterpret_cast<float *>(sm + 128);   // activation tile, later partial sums
    unsigned char *s_vals = sm + 128 + size_t(kXcapB + kBoxRows * kBt) * 4;
    uint32_t *s_offs = reinterpret_cast<uint32_t *>(s_vals + size_t(kRecCap) * kSlots * kChunk * kEsz);

    pdl_launch_dependents();
    cg::cluster_group cluster = cg::this_cluster();
    const int ksc = static_cast<int>(cluster.num_blocks());
    const int q = static_cast<int>(cluster.block_rank());
    const int2 set = sets[blockIdx.x / ksc];
    const int ng = set.y;
    const Group g0 = f.groups[set.x];
    const int m = g0.m, n = g0.n, rw = g0.nib ? 1 : 2;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int qd = lane % LPR, rr = lane / LPR;
    const int64_t b0 = int64_t(blockIdx.y) * kBt;
    const int nch = (n + kChunk - 1) / kChunk;
    const int cpc = (nch + ksc - 1) / ksc;
    const int c0 = min(nch, q * cpc), c1 = min(nch, c0 + cpc);
    const int J0 = c0 * kChunk, J1 = min(n, c1 * kChunk);
    // blocks per round: bounded by the activation tile and by the staged records
    const int rb = max(1, min(kXcapB / (m * kBt), (kRecCap / ng - 1) * kChunk));
    const int rounds = (J1 - J0 + rb - 1) / rb;

    if (tid == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    __syncthreads();

    auto round_geo = [&](int r, int &jr0, int &jr1, int &cr0, int &nchr) {
        jr0 = J0 + r * rb;
        jr1 = min(J1, jr0 + rb);
        cr0 = jr0 / kChunk;
        nchr = (jr1 + kChunk - 1) / kChunk - cr0;
    };
    // copies of the handle's values and offsets for round r (thread 0)
    auto issue_handle = [&](int r, bool arrive, uint32_t extra) {
        int jr0, jr1, cr0, nchr;
        round_geo(r, jr0, jr1, cr0, nchr);
        const uint32_t bv = uint32_t(nchr) * kSlots * kChunk * kEsz;
        const uint32_t bo = uint32_t(nchr) * kSlots * rw * 4;
        if (arrive) mbar_arrive_expect_tx(bar, uint32_t(ng) * (bv + bo) + extra);
        else mbar_expect_tx(bar, uint32_t(ng) * (bv + bo));
        for (int gi = 0; gi < ng; ++gi) {
            const Group g = f.groups[set.x + gi];
            bulk_g2s(s_vals + size_t(gi) * bv,
                     static_cast<const unsigned char *>(f.vals) + (size_t(g.val_off) + size_t(cr0) * kSlots * kChunk) * kEsz,
                     bv, bar);
            bulk_g2s(reinterpret_cast<unsigned char *>(s_offs) + size_t(gi) * bo,
                     f.offs + g.off_off + size_t(cr0) * kSlots * rw, bo, bar);
        }
    };
    if (early && rounds > 0 && tid == 0) issue_handle(0, false, 0);
    pdl_wait_previous();

    float4 acc[kRptMax];
#pragma unroll
    for (int p = 0; p < kRptMax; ++p) acc[p] = make_float4(0.f, 0.f, 0.f, 0.f);
    const int rpt = (ng * kSlots + kWarps * kRpw - 1) / (kWarps * kRpw);
    bool ok = true;
    int r_fail = 0;
    for (int r = 0; r < rounds && ok; ++r) {
        r_fail = r;
        int jr0, jr1, cr0, nchr;
        round_geo(r, jr0, jr1, cr0, nchr);
        const int kx0 = jr0 * m;
        const int64_t kxe = int64_t(jr1) * m;
        const int kr = static_cast<int>((kxe < f.cols ? kxe : f.cols) - kx0);
        const int nbox = (kr + kBoxRows - 1) / kBoxRows;
        if (tid == 0) {
            if (r > 0) fence_proxy_async_smem();   // last round's generic reads come first
            const uint32_t xbytes = use_tma ? uint32_t(nbox) * kBoxRows * kBt * 4 : 0u;
            if (early && r == 0) {
                mbar_arrive_expect_tx(bar, xbytes);
            } else {
                issue_handle(r, true, xbytes);
            }
            if (use_tma)
                for (int i = 0; i < nbox; ++i)
                    tensor2d_g2s(s_x + size_t(i) * kBoxRows * kBt, &xmap, int(b0), kx0 + i * kBoxRows, bar);
        }
        if (!use_tma) {
            // X not addressable by a tensor map: 8 independent loads in flight per thread
            const int nx = kr * kBt;
            for (int base = 0; base < nx; base += 8 * kWarps * 32) {
                float tmp[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int idx = base + u * kWarps * 32 + tid;
                    const int kk = idx / kBt, t = idx % kBt;
                    tmp[u] = (idx < nx && b0 + t < batch) ? __ldg(X + int64_t(kx0 + kk) * ldx + b0 + t) : 0.0f;
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
        if (ok) {
            const float4 *sx4 = reinterpret_cast<const float4 *>(s_x);
            for (int lc = 0; lc < nchr; ++lc) {
                const int jc = (cr0 + lc) * kChunk;
#pragma unroll
                for (int p = 0; p < kRptMax; ++p) {
                    const int s = warp * kRpw + rr + p * kWarps * kRpw;
                    const int gi = s / kSlots, slot = s % kSlots;
                    const bool valid = p < rpt && gi < ng && slot < f.groups[set.x + min(gi, ng - 1)].nrows;
                    if (valid) {
                        const int rec = (gi * nchr + lc) * kSlots + slot;
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
                        if (rw == 1) ow = make_uint2(s_offs[rec], 0u);
                        else ow = reinterpret_cast<const uint2 *>(s_offs)[rec];
#pragma unroll
                        for (int e = 0; e < kChunk; ++e) {
                            const int j = jc + e;
                            if (j >= jr0 && j < jr1) {
                                const int off = rw == 1 ? int((ow.x >> (4 * e)) & 15u)
                                                        : int(((e < 4 ? ow.x : ow.y) >> (8 * (e & 3))) & 255u);
                                const float4 xv = sx4[(j * m + off - kx0) * LPR + qd];
                                acc[p].x = fmaf(v[e], xv.x, acc[p].x);
                                acc[p].y = fmaf(v[e], xv.y, acc[p].y);
                                acc[p].z = fmaf(v[e], xv.z, acc[p].z);
                                acc[p].w = fmaf(v[e], xv.w, acc[p].w);
                            }
                        }
                    }
                }
            }
        }
        __syncthreads();
    }
    if (!ok) {
        // a copy did not land in time: record it, let in-flight copies settle,
        // and finish without trusting the sums
        if (tid == 0) atomicOr(f.status, kStatusTimeout);
        mbar_wait(bar, r_fail & 1);
        __syncthreads();
    }
    // partial sums of every row slot of the set, slot-major: part[s][0..kBt)
    float4 *part4 = reinterpret_cast<float4 *>(s_x);
#pragma unroll
    for (int p = 0; p < kRptMax; ++p) {
        const int s = warp * kRpw + rr + p * kWarps * kRpw;
        if (p < rpt && s < ng * kSlots) part4[s * LPR + qd] = acc[p];
    }
    __syncthreads();
    if (ksc > 1) cluster.sync();
    // rank q finishes rows [s0, s1) of the set for the whole tile
    const int R = ng * kSlots;
    const int per = (R + ksc - 1) / ksc;
    const int s0 = min(R, q * per), s1 = min(R, s0 + per);
    for (int idx = tid; idx < (s1 - s0) * kBt; idx += kWarps * 32) {
        const int s = s0 + idx / kBt, t = idx % kBt;
        const int gi = s / kSlots, slot = s % kSlots;
        if (b0 + t >= batch || slot >= f.groups[set.x + gi].nrows) continue;
        float sum = 0.0f;   // ranks in a fixed order: deterministic
        for (int r = 0; r < ksc; ++r) sum += cluster.map_shared_rank(s_x, r)[s * kBt + t];
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
// kBoxRows x bt box; false if X cannot be described (alignment).
bool make_xmap(CUtensorMap *map, const float *X, int64_t ldx, int64_t batch, int64_t cols, int bt) {
    if (reinterpret_cast<uintptr_t>(X) % 16 != 0 || (ldx * 4) % 16 != 0) return false;
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (enc == nullptr) return false;
    const cuuint64_t dims[2] = {cuuint64_t(batch), cuuint64_t(cols)};
    const cuuint64_t strides[1] = {cuuint64_t(ldx) * 4};
    const cuuint32_t box[2] = {cuuint32_t(bt), cuuint32_t(kBoxRows)};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(X), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <bool BF16, int LPR>
cudaError_t launch_batch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                         int64_t ldy, bool early, cudaStream_t stream) {
    constexpr int kBt = 4 * LPR;
    constexpr size_t smem = batch_smem<BF16, LPR>();
    static const cudaError_t attr = allow_smem(spmm_batch<BF16, LPR>, smem);
    if (attr != cudaSuccess) return attr;
    CUtensorMap map;
    std::memset(&map, 0, sizeof map);
    const int use_tma = make_xmap(&map, X, ldx, batch, f.cols, kBt) ? 1 : 0;
    const int level = 3;   // sets of up to 8 groups
    const int64_t tiles = (batch + kBt - 1) / kBt;
    // cluster split so that the grid fills the GPU about twice over
    unsigned ksc = 1;
    while (ksc < 8 && int64_t(f.nsets[level]) * tiles * ksc * 2 <= 3 * int64_t(sm_count())) ksc *= 2;
    const dim3 grid(static_cast<unsigned>(f.nsets[level]) * ksc, static_cast<unsigned>(tiles));
    return launch_ex(spmm_batch<BF16, LPR>, grid, dim3(kWarps * 32), smem, stream, ksc, true, f, f.sets[level], X,
                     ldx, batch, Y, ldy, map, use_tma, early ? 1 : 0);
}

}  // namespace

cudaError_t launch_spmm_batch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                              int64_t ldy, bool early, cudaStream_t stream) {
    if (batch <= 16)
        return f.bf16 ? launch_batch<true, 4>(f, X, ldx, batch, Y, ldy, early, stream)
                      : launch_batch<false, 4>(f, X, ldx, batch, Y, ldy, early, stream);
    return f.bf16 ? launch_batch<true, 8>(f, X, ldx, batch, Y, ldy, early, stream)
                  : launch_batch<false, 8>(f, X, ldx, batch, Y, ldy, early, stream);
}

}  // namespace darb
