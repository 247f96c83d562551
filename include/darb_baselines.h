/*
 * darb_baselines.h -- C ABI of libdarb_baselines: the sparse formats DARB is
 * compared with, multiplied by cuSPARSE on the same GPU, so that their decode
 * and product cost can be measured against darb_spmm at equal density.
 *
 * The paper compares DARB's decoding with that of irregular pruning stored
 * as CSR (Sec. 2, "Irregular Pruning and Index Decoding": decoding one index
 * of a compressed row needs a search) and with 4x4 and 8x8 block pruning
 * (Sec. 2, "Structured Pruning", and Sec. 4.2), on its own hardware.  These
 * calls restate that comparison for a GB300: the same kept weights as CSR,
 * and a block-pruned matrix of the same density as BSR, each multiplied by
 * the vendor library.  They are measurement baselines, not part of the DARB
 * path (libdarb does not link them).
 *
 * Conventions as in darb.h: device pointers of the current device, Y is
 * overwritten, every call is asynchronous on `stream` and returns a
 * darb_status_t.  The dense operands take either layout, so that the vendor
 * library can be measured in the one it runs fastest:
 *   DARB_DENSE_ROWS  X is cols x batch with the batch contiguous (row k at
 *                    X + k * ldx), Y rows x batch (row r at Y + r * ldy): the
 *                    layout of darb_spmm;
 *   DARB_DENSE_COLS  each batch column contiguous: X element (k, b) at
 *                    X + b * ldx + k (ldx >= cols), Y element (r, b) at
 *                    Y + b * ldy + r (ldy >= rows).  cuSPARSE's workspace comes from
 * the device's stream-ordered memory pool on `stream` and goes back to it
 * before the call returns (in stream order).  One cuSPARSE handle per device
 * is created on first use and kept until the process exits.
 */
#ifndef DARB_BASELINES_H
#define DARB_BASELINES_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#include "darb.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { DARB_DENSE_ROWS = 0, DARB_DENSE_COLS = 1 } darb_dense_layout_t;

/*
 * Y = A X with A in CSR (the irregular format of Sec. 2), fp32 values.
 *   row_ptr  device int32[rows + 1], row_ptr[0] = 0, non-decreasing, row_ptr[rows] = nnz
 *   col_idx  device int32[nnz], columns of each row in [0, cols)
 *   vals     device fp32[nnz]
 * Errors: DARB_ERR_INVALID_ARG (null pointers, rows/cols/batch <= 0, nnz < 0,
 * a leading dimension below its layout's minimum, sizes that do not fit
 * int32, an unknown layout); DARB_ERR_UNSUPPORTED if cuSPARSE
 * refuses the shapes or layouts; DARB_ERR_OOM; DARB_ERR_CUDA (any other
 * CUDA or cuSPARSE failure).
 */
DARB_API darb_status_t darb_baseline_csr_spmm(const int32_t *row_ptr, const int32_t *col_idx, const float *vals,
                                              int64_t rows, int64_t cols, int64_t nnz, const float *X, int64_t ldx,
                                              int64_t batch, float *Y, int64_t ldy, darb_dense_layout_t layout,
                                              cudaStream_t stream);

/*
 * Y = A X with A in BSR: square bs x bs blocks (block pruning, Sec. 4.2),
 * fp32 values, each block row-major.
 *   brow_ptr device int32[rows / bs + 1] over block rows
 *   bcol_idx device int32[nnzb], block columns in [0, cols / bs)
 *   bvals    device fp32[nnzb * bs * bs]
 * rows and cols must be multiples of bs (1 < bs <= 32).
 * Errors as darb_baseline_csr_spmm.
 */
DARB_API darb_status_t darb_baseline_bsr_spmm(const int32_t *brow_ptr, const int32_t *bcol_idx, const float *bvals,
                                              int64_t rows, int64_t cols, int64_t bs, int64_t nnzb, const float *X,
                                              int64_t ldx, int64_t batch, float *Y, int64_t ldy,
                                              darb_dense_layout_t layout, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif
