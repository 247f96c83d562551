// spmm.cu -- y = W_darb X on the GPU (Sec. 3.2, Fig. 6(b)): the entry the C
// ABI calls.  Batch 1 runs the one-group-per-CTA kernel (gemv.cuh) when x fits
// in shared memory, batch <= 4 otherwise the row-per-lane kernel (rowlane.cuh:
// the HBM-bound regime, values and offsets stream once), wider batches the
// batch-per-lane kernel (batch.cuh, instantiated in spmm_batch.cu).  All of
// them evaluate exactly the per-block selection and sum of Fig. 6(b) on the
// CUDA cores and allocate nothing.  The tensor-core kernel (tc.cuh, in
// spmm_tc.cu) runs only when the caller asks for it by name.  All accumulate
// in fp32, add partial sums in a fixed order (results are deterministic) and
// write every output element exactly once.
#include "gemv.cuh"
#include "launch.cuh"
#include "rowlane.cuh"

#include <mutex>
#include <set>

namespace darb {

cudaError_t launch_spmm(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                        int64_t ldy, bool early, int path, cudaStream_t stream) {
    if (path == DARB_PATH_TENSOR_CORES) return launch_spmm_tc(f, X, ldx, batch, Y, ldy, early, stream);
    if (batch == 1 && f.cols <= int64_t(gemv::kMaxCols))
        return f.bf16 ? gemv::launch<true>(f, X, ldx, Y, ldy, early, stream)
                      : gemv::launch<false>(f, X, ldx, Y, ldy, early, stream);
    if (batch <= 4) {
        const RnnArgs none{};
        return f.bf16 ? rowlane::launch_any<true, kModeY>(f, X, ldx, batch, Y, ldy, none, early, stream)
                      : rowlane::launch_any<false, kModeY>(f, X, ldx, batch, Y, ldy, none, early, stream);
    }
    return launch_spmm_batch(f, X, ldx, batch, Y, ldy, early, stream);
}

cudaError_t stream_alloc(void **p, size_t bytes, cudaStream_t stream) {
    static std::mutex mu;
    static std::set<int> raised;
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess) {
        std::lock_guard<std::mutex> lk(mu);
        if (raised.insert(dev).second) {
            cudaMemPool_t pool;
            uint64_t cur = 0;
            if (cudaDeviceGetMemPool(&pool, dev) == cudaSuccess &&
                cudaMemPoolGetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &cur) == cudaSuccess &&
                cur < kPoolKeep) {
                uint64_t v = kPoolKeep;
                cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &v);
            }
            cudaGetLastError();
        }
    } else {
        cudaGetLastError();
    }
    return cudaMallocAsync(p, bytes, stream);
}

int sm_count() {
    static const char key = 0;
    return static_cast<int>(per_device(&key, 0, [] {
        int v = 0;
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, current_device()) != cudaSuccess || v <= 0) {
            cudaGetLastError();
            return 148ll;
        }
        return static_cast<long long>(v);
    }));
}

}  // namespace darb
