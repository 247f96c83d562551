// rnn.cu -- one LSTM or GRU cell step on a DARB gate matrix, in one kernel.
//
// The gate matrix (4H or 3H rows, I + H columns) multiplies the stacked input
// [x_t; h_{t-1}] read in place from the two caller buffers.  The rows of one
// hidden unit (i, f, g, o or r, z, n) generally have different block sizes and
// so sit in different 32-row groups, handled by different CTAs.  Each CTA runs
// the row-per-lane gather-FMA of the product kernel over its group, writes its
// rows' gate sums to a scratch buffer, fences, and counts the arrival on a
// per-(unit, batch tile) counter.  The CTA that brings the last gate of a unit
// applies the cell nonlinearities for that unit and resets the counter, so the
// step finishes inside the same launch with no second kernel and no waiting.
// Which CTA finishes a unit varies; the result does not, because every gate
// sum is computed in a fixed order before it is published.
//
// GRU keeps the x-part and h-part of each gate sum apart (a and bh), since the
// reset gate multiplies only the h-part of the candidate gate.
#include "kernels_common.cuh"
#include "launch.cuh"
#include "tma.cuh"

namespace darb {
namespace {

struct CellArgs {
    const float *c_prev;   // LSTM
    const float *h_prev;   // GRU: h_{t-1} again, for the interpolation
    const float *bias;     // LSTM combined bias [4H] or nullptr
    const float *b_ih;     // GRU
    const float *b_hh;     // GRU
    float *h_out;
    float *c_out;          // LSTM
};

template <bool BF16, int BT, bool GRU>
__global__ void __launch_bounds__(kWarps * 32)
rnn_step_rowlane(Format f, XStacked xs, int64_t B, int H, RnnScratch sc, CellArgs ca) {
    constexpr int kParts = GRU ? 2 : 1;
    __shared__ float red[kWarps][kSlots][BT * kParts];
    pdl_launch_dependents();
    pdl_wait_previous();
    const int gi = blockIdx.x;
    const Group g = f.groups[gi];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t b0 = static_cast<int64_t>(blockIdx.y) * BT;
    const int nb = B - b0 < BT ? static_cast<int>(B - b0) : BT;
    const int nch = (g.n + kChunk - 1) / kChunk;
    const int cpw = (nch + kWarps - 1) / kWarps;
    const int c_begin = min(nch, warp * cpw), c_end = min(nch, c_begin + cpw);
    float acc[BT], acc2[BT];
#pragma unroll
    for (int t = 0; t < BT; ++t) acc[t] = acc2[t] = 0.0f;
    if (lane < g.nrows) {
        if (g.nib)
            rowlane_accumulate<BF16, true, BT, GRU>(f, g, lane, c_begin, c_end, xs, b0, nb, acc, acc2);
        else
            rowlane_accumulate<BF16, false, BT, GRU>(f, g, lane, c_begin, c_end, xs, b0, nb, acc, acc2);
    }
#pragma unroll
    for (int t = 0; t < BT; ++t) {
        red[warp][lane][t] = acc[t];
        if constexpr (GRU) red[warp][lane][BT + t] = acc2[t];
    }
    __syncthreads();
    if (warp != 0 || lane >= g.nrows) return;

    const int row = f.rowmap[gi * kSlots + lane];
    const int64_t rows = f.rows;
    float *gx = sc.gates;                 // x part (GRU) or whole sum (LSTM)
    float *gh = sc.gates + rows * B;      // h part (GRU only)
#pragma unroll
    for (int t = 0; t < BT; ++t) {
        float s = red[0][lane][t], s2 = 0.0f;
#pragma unroll
        for (int w = 1; w < kWarps; ++w) s += red[w][lane][t];
        if constexpr (GRU) {
            s2 = red[0][lane][BT + t];
#pragma unroll
            for (int w = 1; w < kWarps; ++w) s2 += red[w][lane][BT + t];
        }
        if (t < nb) {
            gx[row * B + b0 + t] = s;
            if constexpr (GRU) gh[row * B + b0 + t] = s2;
        }
    }
    __threadfence();
    const int unit = row % H;
    int32_t *cnt = sc.counters + static_cast<int64_t>(unit) * gridDim.y + blockIdx.y;
    const int old = atomicAdd(cnt, 1);
    if (old != (GRU ? 2 : 3)) return;
    // last gate of this unit: every other gate's sums are published
    __threadfence();
    *cnt = 0;
    for (int t = 0; t < nb; ++t) {
        const int64_t b = b0 + t;
        if constexpr (!GRU) {
            float pre[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int64_t r = static_cast<int64_t>(q) * H + unit;
                pre[q] = __ldcg(gx + r * B + b) + (ca.bias ? ca.bias[r] : 0.0f);
            }
            const float c = sigmoidf_(pre[1]) * ca.c_prev[unit * B + b] + sigmoidf_(pre[0]) * tanhf(pre[2]);
            ca.c_out[unit * B + b] = c;
            ca.h_out[unit * B + b] = sigmoidf_(pre[3]) * tanhf(c);
        } else {
            float a[3], bh[3];
#pragma unroll
            for (int q = 0; q < 3; ++q) {
                const int64_t r = static_cast<int64_t>(q) * H + unit;
                a[q] = __ldcg(gx + r * B + b) + (ca.b_ih ? ca.b_ih[r] : 0.0f);
                bh[q] = __ldcg(gh + r * B + b) + (ca.b_hh ? ca.b_hh[r] : 0.0f);
            }
            const float rr = sigmoidf_(a[0] + bh[0]);
            const float zz = sigmoidf_(a[1] + bh[1]);
            const float nn = tanhf(a[2] + rr * bh[2]);
            ca.h_out[unit * B + b] = (1.0f - zz) * nn + zz * ca.h_prev[unit * B + b];
        }
    }
}

template <bool GRU>
cudaError_t launch_step(const Format &f, int64_t I, int64_t H, int64_t B, const float *x,
                        const float *h_prev, RnnScratch sc, const CellArgs &ca,
                        cudaStream_t stream) {
    XStacked xs{x, h_prev, static_cast<int>(I), B};
    const int bt = rnn_batch_tile(B);
    const dim3 grid(static_cast<unsigned>(f.ngroups), static_cast<unsigned>((B + bt - 1) / bt));
    const dim3 block(kWarps * 32);
    const int h = static_cast<int>(H);
#define DARB_STEP(BF, BTV) \
    launch_ex(rnn_step_rowlane<BF, BTV, GRU>, grid, block, 0, stream, 1, true, f, xs, B, h, sc, ca)
    if (f.bf16) {
        if (bt == 1) return DARB_STEP(true, 1);
        if (bt == 2) return DARB_STEP(true, 2);
        if (bt == 4) return DARB_STEP(true, 4);
        return DARB_STEP(true, 8);
    }
    if (bt == 1) return DARB_STEP(false, 1);
    if (bt == 2) return DARB_STEP(false, 2);
    if (bt == 4) return DARB_STEP(false, 4);
    return DARB_STEP(false, 8);
#undef DARB_STEP
}

}  // namespace

int rnn_batch_tile(int64_t B) { return B == 1 ? 1 : B == 2 ? 2 : B <= 4 ? 4 : 8; }

cudaError_t launch_lstm_step(const Format &f, int64_t I, int64_t H, int64_t B, const float *x,
                             const float *h_prev, const float *c_prev, const float *bias,
                             float *h_out, float *c_out, RnnScratch s, cudaStream_t stream) {
    CellArgs ca{c_prev, h_prev, bias, nullptr, nullptr, h_out, c_out};
    return launch_step<false>(f, I, H, B, x, h_prev, s, ca, stream);
}

cudaError_t launch_gru_step(const Format &f, int64_t I, int64_t H, int64_t B, const float *x,
                            const float *h_prev, const float *b_ih, const float *b_hh,
                            float *h_out, RnnScratch s, cudaStream_t stream) {
    CellArgs ca{nullptr, h_prev, nullptr, b_ih, b_hh, h_out, nullptr};
    return launch_step<true>(f, I, H, B, x, h_prev, s, ca, stream);
}

}  // namespace darb
