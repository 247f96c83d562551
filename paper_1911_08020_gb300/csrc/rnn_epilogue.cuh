// rnn_epilogue.cuh -- the output side of a fused RNN step (LSTM or GRU cell on
// a DARB gate matrix), shared by the row-per-lane and the batch kernels.
//
// A product kernel in RNN mode reads the stacked input [x_t; h_{t-1}] in place
// (rows [0, I) of the gate matrix's columns multiply x, rows [I, I+H) multiply
// h) and, instead of writing Y, publishes every gate row's final sum (for GRU
// the x part and the h part separately) to a gate scratch buffer.  The rows of
// one hidden unit usually sit in different CTAs, so each CTA then counts its
// rows on a per-(unit, batch tile) counter; the CTA whose count completes a
// unit applies the cell to it and resets the counter.  Nothing waits: the
// last gate to arrive does the work.
#pragma once

#include "darb_internal.h"

namespace darb {

constexpr int kModeY = 0;      // plain product, write Y
constexpr int kModeLstm = 1;   // gate rows i, f, g, o
constexpr int kModeGru = 2;    // gate rows r, z, n; x and h parts kept apart

struct RnnArgs {
    const float *x;         // I x B
    const float *h;         // H x B (h_{t-1})
    float *gx;              // rows x B: gate sums (LSTM) or their x parts (GRU)
    float *gh;              // rows x B: h parts (GRU)
    int32_t *counters;      // units x tiles, zero between launches
    const float *c_prev;    // LSTM
    const float *bias;      // LSTM combined bias [4H] or nullptr
    const float *b_ih;      // GRU [3H] or nullptr
    const float *b_hh;      // GRU [3H] or nullptr
    float *h_out;
    float *c_out;           // LSTM
    int I, H;
    int64_t B;
};

__device__ __forceinline__ float sigm(float v) { return 1.0f / (1.0f + expf(-v)); }

// The cell of `unit` for batch column b, from the published gate sums.
template <int MODE>
__device__ __forceinline__ void rnn_cell(const RnnArgs &a, int unit, int64_t b) {
    const int64_t B = a.B, H = a.H;
    if constexpr (MODE == kModeLstm) {
        float pre[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int64_t r = q * H + unit;
            pre[q] = __ldcg(a.gx + r * B + b) + (a.bias ? a.bias[r] : 0.0f);
        }
        const float c = sigm(pre[1]) * a.c_prev[unit * B + b] + sigm(pre[0]) * tanhf(pre[2]);
        a.c_out[unit * B + b] = c;
        a.h_out[unit * B + b] = sigm(pre[3]) * tanhf(c);
    } else {
        float ax[3], bh[3];
#pragma unroll
        for (int q = 0; q < 3; ++q) {
            const int64_t r = q * H + unit;
            ax[q] = __ldcg(a.gx + r * B + b) + (a.b_ih ? a.b_ih[r] : 0.0f);
            bh[q] = __ldcg(a.gh + r * B + b) + (a.b_hh ? a.b_hh[r] : 0.0f);
        }
        const float rr = sigm(ax[0] + bh[0]);
        const float zz = sigm(ax[1] + bh[1]);
        const float nn = tanhf(ax[2] + rr * bh[2]);
        a.h_out[unit * B + b] = (1.0f - zz) * nn + zz * a.h[unit * B + b];
    }
}

// Called by every thread of the CTA after it has stored the final gate sums of
// rows[0..nloc) for columns [b0, b0+nc) of batch tile `tile`.  s_units holds
// room for nloc ints and *s_nunits one.
template <int MODE>
__device__ void rnn_finish(const RnnArgs &a, const int *rows, int nloc, int tile, int ntiles, int64_t b0,
                           int nc, int *s_units, int *s_nunits) {
    constexpr int kGates = MODE == kModeLstm ? 4 : 3;
    const int tid = threadIdx.x, nthr = blockDim.x;
    __threadfence();   // this thread's gate stores are visible device-wide before any count
    if (tid == 0) *s_nunits = 0;
    __syncthreads();
    for (int i = tid; i < nloc; i += nthr) {
        const int unit = rows[i] % a.H;
        const int old = atomicAdd(a.counters + int64_t(unit) * ntiles + tile, 1);
        if (old == kGates - 1) s_units[atomicAdd(s_nunits, 1)] = unit;
    }
    __syncthreads();
    __threadfence();   // the other gates of these units were published before their counts
    const int nu = *s_nunits;
    for (int idx = tid; idx < nu * nc; idx += nthr) {
        const int64_t b = b0 + idx % nc;
        if (b < a.B) rnn_cell<MODE>(a, s_units[idx / nc], b);
    }
    for (int i = tid; i < nu; i += nthr) a.counters[int64_t(s_units[i]) * ntiles + tile] = 0;
}

}  // namespace darb
