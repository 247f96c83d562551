// spmm_batch.cu -- the batch > 4 product for plain Y: from 17 columns on the
// kernel with the activation tile resident in shared memory (xres.cuh) when
// the call fits it, else the streaming batch kernel (batch.cuh).  At 16
// columns or fewer the resident tile is one 16-column tile, whose 64-byte rows
// put two rows in each quarter-warp's 128-byte read (half of them conflict),
// and the streaming kernel measured faster (FC6 11.9 us against 16.8).
#include "batch.cuh"
#include "xres.cuh"

namespace darb {

cudaError_t launch_spmm_batch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                              int64_t ldy, bool early, cudaStream_t stream) {
    if (batch > 16) {
        const cudaError_t e = f.bf16 ? xres::launch<true, 32>(f, X, ldx, batch, Y, ldy, early, stream)
                                     : xres::launch<false, 32>(f, X, ldx, batch, Y, ldy, early, stream);
        if (e != cudaErrorNotSupported) return e;
        cudaGetLastError();
    }
    const RnnArgs none{};
    return f.bf16 ? batch::launch_any<true, kModeY>(f, X, ldx, batch, Y, ldy, none, early, stream)
                  : batch::launch_any<false, kModeY>(f, X, ldx, batch, Y, ldy, none, early, stream);
}

cudaError_t launch_spmm_prefix(const Format &f, int64_t col_limit, const float *X, int64_t ldx, int64_t batch,
                               float *Y, int64_t ldy, bool early, cudaStream_t stream) {
    if (batch > 16 && col_limit > 0 && col_limit < f.cols) {
        // xres on a view of the matrix `col_limit` columns wide: its column slices
        // cover [0, col_limit) only, a block that reaches past it reads rows that
        // lie outside the view's tensor map, i.e. zeros, and the blocks that start
        // past it are in no slice
        Format fx = f;
        fx.cols = col_limit;
        const cudaError_t e = f.bf16 ? xres::launch<true, 32>(fx, X, ldx, batch, Y, ldy, early, stream)
                                     : xres::launch<false, 32>(fx, X, ldx, batch, Y, ldy, early, stream);
        if (e != cudaErrorNotSupported) return e;
        cudaGetLastError();
    }
    return launch_spmm(f, X, ldx, batch, Y, ldy, early, DARB_PATH_AUTO, stream);
}

}  // namespace darb
