// spmm.cu -- y = W_darb X on the GPU (Sec. 3.2, Fig. 6(b)): the entry the C
// ABI calls.  Batch <= 4 runs the row-per-lane kernel (rowlane.cuh: the
// HBM-bound regime, values and offsets stream once), wider batches the
// batch-per-lane kernel (batch.cuh, instantiated in spmm_batch.cu) or, for
// bf16 weights from kTensorCoreMinBatch columns on, the tensor-core kernel
// (tc.cuh, in spmm_tc.cu).  All accumulate in fp32, add partial sums in a
// fixed order (results are deterministic) and write every output element
// exactly once.
#include "rowlane.cuh"

namespace darb {

cudaError_t launch_spmm(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                        int64_t ldy, bool early, int path, cudaStream_t stream) {
    if (path == DARB_PATH_TENSOR_CORES) return launch_spmm_tc(f, X, ldx, batch, Y, ldy, early, stream);
    if (path == DARB_PATH_AUTO && f.bf16 && batch >= kTensorCoreMinBatch) {
        const cudaError_t e = launch_spmm_tc(f, X, ldx, batch, Y, ldy, early, stream);
        if (e != cudaErrorNotSupported) return e;
    }
    if (batch <= 4) {
        const RnnArgs none{};
        return f.bf16 ? rowlane::launch_any<true, kModeY>(f, X, ldx, batch, Y, ldy, none, early, stream)
                      : rowlane::launch_any<false, kModeY>(f, X, ldx, batch, Y, ldy, none, early, stream);
    }
    return launch_spmm_batch(f, X, ldx, batch, Y, ldy, early, stream);
}

int sm_count() {
    static int n = [] {
        int dev = 0, v = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
            cudaGetLastError();
            return 148;
        }
        return v;
    }();
    return n;
}

}  // namespace darb
