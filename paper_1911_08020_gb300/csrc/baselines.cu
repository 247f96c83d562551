// baselines.cu -- the comparison formats of include/darb_baselines.h: CSR
// (irregular pruning) and BSR (block pruning) products by cuSPARSE, built as
// their own library so that the DARB path never links the vendor library.
//
// Each call wraps one cusparseSpMM: the sparse matrix descriptor over the
// caller's arrays, dense descriptors over X and Y in the caller's layout
// (row-major: batch contiguous; column-major: each batch column contiguous),
// fp32 values and fp32 compute, workspace from the stream-ordered pool.
#include "darb_baselines.h"

#include <cuda_runtime.h>
#include <cusparse.h>

#include <cstdint>
#include <map>
#include <mutex>

namespace {

constexpr int64_t kI32 = int64_t(INT32_MAX);

std::mutex g_mu;                          // one call at a time per process (the handles are shared)
std::map<int, cusparseHandle_t> g_handle; // per device, created on first use

darb_status_t from_cusparse(cusparseStatus_t s) {
    switch (s) {
    case CUSPARSE_STATUS_SUCCESS: return DARB_OK;
    case CUSPARSE_STATUS_NOT_SUPPORTED:
    case CUSPARSE_STATUS_INVALID_VALUE: return DARB_ERR_UNSUPPORTED;
    case CUSPARSE_STATUS_ALLOC_FAILED: return DARB_ERR_OOM;
    default: return DARB_ERR_CUDA;
    }
}

darb_status_t handle_for_device(cusparseHandle_t *h) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return DARB_ERR_CUDA;
    }
    auto it = g_handle.find(dev);
    if (it == g_handle.end()) {
        cusparseHandle_t nh = nullptr;
        const cusparseStatus_t s = cusparseCreate(&nh);
        if (s != CUSPARSE_STATUS_SUCCESS) return s == CUSPARSE_STATUS_ALLOC_FAILED ? DARB_ERR_OOM : DARB_ERR_CUDA;
        it = g_handle.emplace(dev, nh).first;
    }
    *h = it->second;
    return DARB_OK;
}

bool dense_ok(const float *X, int64_t ldx, int64_t batch, const float *Y, int64_t ldy, int64_t rows, int64_t cols,
              darb_dense_layout_t layout) {
    if (X == nullptr || Y == nullptr || batch <= 0 || batch > kI32 || ldx > kI32 || ldy > kI32) return false;
    if (layout == DARB_DENSE_ROWS) return ldx >= batch && ldy >= batch;
    if (layout == DARB_DENSE_COLS) return ldx >= cols && ldy >= rows;
    return false;
}

// Y = A X for the sparse descriptor A (rows x cols); g_mu held.
darb_status_t spmm(cusparseSpMatDescr_t A, int64_t rows, int64_t cols, const float *X, int64_t ldx, int64_t batch,
                   float *Y, int64_t ldy, darb_dense_layout_t layout, cudaStream_t stream) {
    const cusparseOrder_t order = layout == DARB_DENSE_ROWS ? CUSPARSE_ORDER_ROW : CUSPARSE_ORDER_COL;
    cusparseHandle_t h = nullptr;
    darb_status_t st = handle_for_device(&h);
    if (st != DARB_OK) return st;
    cusparseStatus_t s = cusparseSetStream(h, stream);
    cusparseDnMatDescr_t B = nullptr, C = nullptr;
    if (s == CUSPARSE_STATUS_SUCCESS)
        s = cusparseCreateDnMat(&B, cols, batch, ldx, const_cast<float *>(X), CUDA_R_32F, order);
    if (s == CUSPARSE_STATUS_SUCCESS) s = cusparseCreateDnMat(&C, rows, batch, ldy, Y, CUDA_R_32F, order);
    const float alpha = 1.0f, beta = 0.0f;
    size_t bytes = 0;
    if (s == CUSPARSE_STATUS_SUCCESS)
        s = cusparseSpMM_bufferSize(h, CUSPARSE_OPERATION_NON_TRANSPOSE, CUSPARSE_OPERATION_NON_TRANSPOSE, &alpha, A, B,
                                    &beta, C, CUDA_R_32F, CUSPARSE_SPMM_ALG_DEFAULT, &bytes);
    st = from_cusparse(s);
    void *buf = nullptr;
    if (st == DARB_OK && bytes > 0) {
        const cudaError_t e = cudaMallocAsync(&buf, bytes, stream);
        if (e != cudaSuccess) {
            cudaGetLastError();
            st = e == cudaErrorMemoryAllocation ? DARB_ERR_OOM : DARB_ERR_CUDA;
            buf = nullptr;
        }
    }
    if (st == DARB_OK)
        st = from_cusparse(cusparseSpMM(h, CUSPARSE_OPERATION_NON_TRANSPOSE, CUSPARSE_OPERATION_NON_TRANSPOSE, &alpha,
                                        A, B, &beta, C, CUDA_R_32F, CUSPARSE_SPMM_ALG_DEFAULT, buf));
    if (buf != nullptr && cudaFreeAsync(buf, stream) != cudaSuccess) {
        cudaGetLastError();
        if (st == DARB_OK) st = DARB_ERR_CUDA;
    }
    if (B != nullptr) cusparseDestroyDnMat(B);
    if (C != nullptr) cusparseDestroyDnMat(C);
    return st;
}

}  // namespace

extern "C" {

darb_status_t darb_baseline_csr_spmm(const int32_t *row_ptr, const int32_t *col_idx, const float *vals, int64_t rows,
                                     int64_t cols, int64_t nnz, const float *X, int64_t ldx, int64_t batch, float *Y,
                                     int64_t ldy, darb_dense_layout_t layout, cudaStream_t stream) {
    if (row_ptr == nullptr || rows <= 0 || cols <= 0 || nnz < 0 || rows > kI32 || cols > kI32 || nnz > kI32 ||
        (nnz > 0 && (col_idx == nullptr || vals == nullptr)) || !dense_ok(X, ldx, batch, Y, ldy, rows, cols, layout))
        return DARB_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> lk(g_mu);
    cusparseSpMatDescr_t A = nullptr;
    const cusparseStatus_t s = cusparseCreateCsr(&A, rows, cols, nnz, const_cast<int32_t *>(row_ptr),
                                                 const_cast<int32_t *>(col_idx), const_cast<float *>(vals),
                                                 CUSPARSE_INDEX_32I, CUSPARSE_INDEX_32I, CUSPARSE_INDEX_BASE_ZERO,
                                                 CUDA_R_32F);
    darb_status_t st = from_cusparse(s);
    if (st == DARB_OK) st = spmm(A, rows, cols, X, ldx, batch, Y, ldy, layout, stream);
    if (A != nullptr) cusparseDestroySpMat(A);
    return st;
}

darb_status_t darb_baseline_bsr_spmm(const int32_t *brow_ptr, const int32_t *bcol_idx, const float *bvals,
                                     int64_t rows, int64_t cols, int64_t bs, int64_t nnzb, const float *X, int64_t ldx,
                                     int64_t batch, float *Y, int64_t ldy, darb_dense_layout_t layout,
                                     cudaStream_t stream) {
    if (brow_ptr == nullptr || rows <= 0 || cols <= 0 || bs <= 1 || bs > 32 || rows % bs != 0 || cols % bs != 0 ||
        nnzb < 0 || rows > kI32 || cols > kI32 || nnzb * bs * bs > kI32 ||
        (nnzb > 0 && (bcol_idx == nullptr || bvals == nullptr)) || !dense_ok(X, ldx, batch, Y, ldy, rows, cols, layout))
        return DARB_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> lk(g_mu);
    cusparseSpMatDescr_t A = nullptr;
    const cusparseStatus_t s = cusparseCreateBsr(&A, rows / bs, cols / bs, nnzb, bs, bs,
                                                 const_cast<int32_t *>(brow_ptr), const_cast<int32_t *>(bcol_idx),
                                                 const_cast<float *>(bvals), CUSPARSE_INDEX_32I, CUSPARSE_INDEX_32I,
                                                 CUSPARSE_INDEX_BASE_ZERO, CUDA_R_32F, CUSPARSE_ORDER_ROW);
    darb_status_t st = from_cusparse(s);
    if (st == DARB_OK) st = spmm(A, rows, cols, X, ldx, batch, Y, ldy, layout, stream);
    if (A != nullptr) cusparseDestroySpMat(A);
    return st;
}

}  // extern "C"
