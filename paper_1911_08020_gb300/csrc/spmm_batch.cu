// spmm_batch.cu -- the batch > 4 product (batch.cuh) for plain Y.
#include "batch.cuh"

namespace darb {

cudaError_t launch_spmm_batch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                              int64_t ldy, bool early, cudaStream_t stream) {
    const RnnArgs none{};
    return f.bf16 ? batch::launch_any<true, kModeY>(f, X, ldx, batch, Y, ldy, none, early, stream)
                  : batch::launch_any<false, kModeY>(f, X, ldx, batch, Y, ldy, none, early, stream);
}

}  // namespace darb
