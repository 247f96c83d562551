// rnn_batch.cu -- the batch > 4 RNN steps (batch.cuh in LSTM / GRU mode).
#include "batch.cuh"

namespace darb {

cudaError_t launch_rnn_batch(const Format &f, const RnnArgs &ra, int mode, bool early, cudaStream_t stream) {
    if (mode == kModeLstm)
        return f.bf16 ? batch::launch_any<true, kModeLstm>(f, nullptr, 0, ra.B, nullptr, 0, ra, early, stream)
                      : batch::launch_any<false, kModeLstm>(f, nullptr, 0, ra.B, nullptr, 0, ra, early, stream);
    return f.bf16 ? batch::launch_any<true, kModeGru>(f, nullptr, 0, ra.B, nullptr, 0, ra, early, stream)
                  : batch::launch_any<false, kModeGru>(f, nullptr, 0, ra.B, nullptr, 0, ra, early, stream);
}

}  // namespace darb
