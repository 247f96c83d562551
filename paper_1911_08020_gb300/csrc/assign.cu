// assign.cu -- the row densities of Sec. 3.2's first step on the GPU: each
// row's count of the K weights of largest magnitude (the mask of irregular
// pruning, Sec. 2 "Irregular Pruning and Index Decoding", used only to
// measure density).
//
// The K-th largest magnitude is found by radix selection over the stored
// magnitude bits (15 for bf16, 31 for fp32: |w| orders like its bits for every
// non-NaN w), 8 bits per pass from the top: a pass histograms the next digit
// of the weights whose higher digits equal the prefix chosen so far, and a
// one-thread kernel picks the digit that holds the K-th largest and narrows
// the prefix.  No pass needs the host.  A last pass counts, per row, the
// weights whose magnitude bits are >= the threshold (every weight tied with
// the K-th largest counts).  NaN weights are reported, not ranked.
#include "darb_internal.h"
#include "launch.cuh"
#include "tma.cuh"

#include <algorithm>

namespace darb {
namespace {

constexpr int kAssignThreads = 256;

struct Select {
    uint32_t prefix;      // digits chosen so far
    int64_t remaining;    // rank of the threshold among the weights that share the prefix
};

template <bool BF16>
__device__ __forceinline__ uint32_t mag_bits(const void *W, int64_t i) {
    if constexpr (BF16) return static_cast<const uint16_t *>(W)[i] & 0x7FFFu;
    else return static_cast<const uint32_t *>(W)[i] & 0x7FFFFFFFu;
}

template <bool BF16>
__host__ __device__ constexpr uint32_t max_finite_bits() { return BF16 ? 0x7F80u : 0x7F800000u; }

// Histogram of the digit (bits >> shift) & (2^width - 1) over the weights
// whose bits above shift + width equal the prefix; flags NaNs.
// The magnitude bits of the weights of row r, 16 bytes (8 bf16 or 4 fp32) per
// load where the row allows it, handed to f(bits) one by one.
template <bool BF16, typename F>
__device__ __forceinline__ void for_row(const void *W, int64_t r, int64_t cols, int64_t ldw, F &&f) {
    constexpr int kPer = BF16 ? 8 : 4;   // weights per 16-byte load
    const char *row = static_cast<const char *>(W) + r * ldw * (BF16 ? 2 : 4);
    const int64_t lead = (reinterpret_cast<uintptr_t>(row) & 15) == 0 ? 0 : cols;   // unaligned row: plain loads
    const int64_t nvec = (cols - lead) / kPer;
    for (int64_t v = threadIdx.x; v < nvec; v += blockDim.x) {
        const uint4 q = __ldg(reinterpret_cast<const uint4 *>(row) + v);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if constexpr (BF16) {
                f(w[k] & 0x7FFFu);
                f((w[k] >> 16) & 0x7FFFu);
            } else {
                f(w[k] & 0x7FFFFFFFu);
            }
        }
    }
    for (int64_t c = nvec * kPer + threadIdx.x; c < cols; c += blockDim.x) f(mag_bits<BF16>(W, r * ldw + c));
}

template <bool BF16>
__global__ void __launch_bounds__(kAssignThreads)
digit_hist_kernel(const void *W, int64_t rows, int64_t cols, int64_t ldw, const Select *sel, int shift, int width,
                  uint32_t *hist, int32_t *nan_flag) {
    // one histogram per warp, and each thread adds a run of equal digits with
    // one atomic: magnitudes cluster (the top digit is mostly the exponent), so
    // element-by-element atomics would serialise on a few bins
    __shared__ uint32_t h[kAssignThreads / 32][256];
    for (int i = threadIdx.x; i < (kAssignThreads / 32) * 256; i += blockDim.x) (&h[0][0])[i] = 0;
    __syncthreads();
    uint32_t *hw = h[threadIdx.x >> 5];
    const uint32_t prefix = sel->prefix, dmask = (1u << width) - 1u;
    const int above = shift + width;   // <= 31: magnitude bits fit in 31
    bool nan = false;
    uint32_t run_bin = 0, run = 0;
    auto take = [&](uint32_t b) {
        nan |= b > max_finite_bits<BF16>();
        if ((b >> above) != prefix) return;
        const uint32_t d = (b >> shift) & dmask;
        if (d == run_bin) {
            ++run;
        } else {
            if (run) atomicAdd(&hw[run_bin], run);
            run_bin = d;
            run = 1;
        }
    };
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) for_row<BF16>(W, r, cols, ldw, take);
    if (run) atomicAdd(&hw[run_bin], run);
    if (nan) atomicOr(nan_flag, 1);
    __syncthreads();
    for (int i = threadIdx.x; i < 256; i += blockDim.x) {
        uint32_t v = 0;
        for (int w = 0; w < kAssignThreads / 32; ++w) v += h[w][i];
        if (v) atomicAdd(&hist[i], v);
    }
}

// The digit whose bin holds the remaining rank, counted from the top.  One
// warp: lane i sums bins [top - 8i - 7, top - 8i], a scan over the lanes finds
// the lane whose range holds the rank, and that lane walks its eight bins.
__global__ void __launch_bounds__(32) pick_digit_kernel(Select *sel, const uint32_t *hist, int width) {
    const int lane = threadIdx.x;
    const int top = (1 << width) - 1;   // 255 or 127
    const int hi = top - 8 * lane;      // this lane's highest bin (< 0: none)
    int64_t mine = 0;
#pragma unroll
    for (int k = 0; k < 8; ++k)
        if (hi - k >= 0) mine += hist[hi - k];
    int64_t incl = mine;   // bins from the top down to the end of this lane's range
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += v;
    }
    const int64_t rem = sel->remaining;
    const unsigned hit = __ballot_sync(0xFFFFFFFFu, hi >= 0 && incl >= rem);
    const int owner = hit ? __ffs(hit) - 1 : (top >> 3);   // the lowest range if the rank is past every bin
    if (lane == owner) {
        int64_t above = incl - mine;   // bins above this lane's range
        int d = hi;
        for (; d > hi - 7 && d > 0; --d) {
            if (above + hist[d] >= rem) break;
            above += hist[d];
        }
        sel->remaining = rem - above;
        sel->prefix = (sel->prefix << width) | uint32_t(d);
    }
}

// Per row: weights whose magnitude bits are >= the threshold.
template <bool BF16>
__global__ void __launch_bounds__(kAssignThreads)
row_count_kernel(const void *W, int64_t rows, int64_t cols, int64_t ldw, const Select *sel, int64_t *row_nnz) {
    __shared__ int64_t part[kAssignThreads / 32];
    const uint32_t t = sel->prefix;
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) {
        int64_t n = 0;
        for_row<BF16>(W, r, cols, ldw, [&](uint32_t b) { n += b >= t ? 1 : 0; });
        for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xFFFFFFFFu, n, o);
        if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = n;
        __syncthreads();
        if (threadIdx.x == 0) {
            int64_t s = 0;
            for (int w = 0; w < kAssignThreads / 32; ++w) s += part[w];
            row_nnz[r] = s;
        }
        __syncthreads();
    }
}

__global__ void init_select_kernel(Select *sel, int64_t keep) {
    if (threadIdx.x == 0 && blockIdx.x == 0) {
        sel->prefix = 0;
        sel->remaining = keep;
    }
}

template <bool BF16>
cudaError_t launch_topk_t(const void *W, int64_t rows, int64_t cols, int64_t ldw, int64_t keep, int64_t *row_nnz,
                          void *work, int32_t *nan_flag, cudaStream_t stream) {
    // work: Select, then one 256-bin histogram per pass
    Select *sel = static_cast<Select *>(work);
    uint32_t *hists = reinterpret_cast<uint32_t *>(static_cast<char *>(work) + 256);
    constexpr int kPasses = BF16 ? 2 : 4;
    cudaError_t e = cudaMemsetAsync(work, 0, 256 + size_t(kPasses) * 256 * 4, stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(nan_flag, 0, 4, stream);
    if (e != cudaSuccess) return e;
    init_select_kernel<<<1, 32, 0, stream>>>(sel, keep);
    const unsigned grid = static_cast<unsigned>(std::max<int64_t>(1, std::min<int64_t>(rows, 8 * int64_t(sm_count()))));
    // digits from the top: 15 bits = 8 + 7, 31 bits = 8 + 8 + 8 + 7
    int top = BF16 ? 15 : 31;
    for (int p = 0; p < kPasses; ++p) {
        const int width = top >= 8 ? 8 : top, shift = top - width;
        digit_hist_kernel<BF16><<<grid, kAssignThreads, 0, stream>>>(W, rows, cols, ldw, sel, shift, width,
                                                                     hists + 256 * p, nan_flag);
        pick_digit_kernel<<<1, 32, 0, stream>>>(sel, hists + 256 * p, width);
        top = shift;
    }
    row_count_kernel<BF16><<<grid, kAssignThreads, 0, stream>>>(W, rows, cols, ldw, sel, row_nnz);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_topk_row_nnz(const void *W, bool bf16, int64_t rows, int64_t cols, int64_t ldw, int64_t keep,
                                int64_t *row_nnz, void *work, int32_t *nan_flag, cudaStream_t stream) {
    return bf16 ? launch_topk_t<true>(W, rows, cols, ldw, keep, row_nnz, work, nan_flag, stream)
                : launch_topk_t<false>(W, rows, cols, ldw, keep, row_nnz, work, nan_flag, stream);
}

}  // namespace darb
