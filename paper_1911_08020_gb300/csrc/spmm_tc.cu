// spmm_tc.cu -- the tensor-core product (tc.cuh) for plain Y.
#include "tc.cuh"

namespace darb {

cudaError_t launch_spmm_tc(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y, int64_t ldy,
                           bool early, cudaStream_t stream) {
    return tc::launch(f, X, ldx, batch, Y, ldy, early, stream);
}

}  // namespace darb
