// rnn.cu -- one LSTM or GRU cell step on a DARB gate matrix, in one kernel.
//
// The gate matrix (4H or 3H rows, I + H columns) multiplies the stacked input
// [x_t; h_{t-1}], read in place from the two caller buffers, with the same
// product kernels as darb_spmm in an RNN output mode (rnn_epilogue.cuh): each
// gate row's final sum is published to scratch, arrivals are counted per
// hidden unit, and the CTA that brings a unit's last gate applies the cell.
// Batch <= 4 uses the row-per-lane kernel (instantiated here), larger batches
// the batch-per-lane kernel (rnn_batch.cu).  GRU keeps the x part and the h
// part of each gate sum apart (a and bh), since the reset gate multiplies only
// the h part of the candidate gate.
#include "rowlane.cuh"

namespace darb {

// An upper bound on the batch tiles any RNN kernel uses for a batch of B
// (sizes the arrival counters): one tile up to 4 columns, else at most one per
// 8 columns.
int rnn_batch_tile(int64_t B) { return B == 1 ? 1 : B == 2 ? 2 : B <= 4 ? 4 : 8; }

cudaError_t launch_lstm_step(const Format &f, int64_t I, int64_t H, int64_t B, const float *x,
                             const float *h_prev, const float *c_prev, const float *bias,
                             float *h_out, float *c_out, RnnScratch s, cudaStream_t stream, bool early) {
    RnnArgs ra{};
    ra.x = x; ra.h = h_prev; ra.gx = s.gates; ra.gh = nullptr; ra.counters = s.counters;
    ra.c_prev = c_prev; ra.bias = bias; ra.h_out = h_out; ra.c_out = c_out;
    ra.I = static_cast<int>(I); ra.H = static_cast<int>(H); ra.B = B;
    if (B <= 4)
        return f.bf16 ? rowlane::launch_any<true, kModeLstm>(f, nullptr, 0, B, nullptr, 0, ra, early, stream)
                      : rowlane::launch_any<false, kModeLstm>(f, nullptr, 0, B, nullptr, 0, ra, early, stream);
    return launch_rnn_batch(f, ra, kModeLstm, early, stream);
}

cudaError_t launch_gru_step(const Format &f, int64_t I, int64_t H, int64_t B, const float *x,
                            const float *h_prev, const float *b_ih, const float *b_hh,
                            float *h_out, RnnScratch s, cudaStream_t stream, bool early) {
    RnnArgs ra{};
    ra.x = x; ra.h = h_prev; ra.gx = s.gates; ra.gh = s.gates + f.rows * B; ra.counters = s.counters;
    ra.b_ih = b_ih; ra.b_hh = b_hh; ra.h_out = h_out;
    ra.I = static_cast<int>(I); ra.H = static_cast<int>(H); ra.B = B;
    if (B <= 4)
        return f.bf16 ? rowlane::launch_any<true, kModeGru>(f, nullptr, 0, B, nullptr, 0, ra, early, stream)
                      : rowlane::launch_any<false, kModeGru>(f, nullptr, 0, B, nullptr, 0, ra, early, stream);
    return launch_rnn_batch(f, ra, kModeGru, early, stream);
}

}  // namespace darb
