/*
 * darb.h -- C ABI of libdarb: density-adaptive regular-block (DARB) pruned
 * matrices on one GB300 GPU (sm_103a).
 *
 * DARB (Ren et al., "DARB: A Density-Adaptive Regular-Block Pruning for Deep
 * Neural Networks", arXiv 1911.08020) splits every row of a weight matrix into
 * equal blocks whose size depends on the row (Sec. 3.2), keeps the one weight of
 * largest magnitude in each block (block-max weight masking, BMWM, Sec. 3.1),
 * and stores per block only that value and its position inside the block
 * (log2 m bits, Sec. 4.2).  Multiplying by such a matrix needs, per block, one
 * small selection among m activations (Sec. 3.2, Fig. 6(b)).
 *
 * This library encodes dense matrices into that format on the GPU and
 * multiplies with them, alone or fused into LSTM / GRU cell steps.
 *
 * Conventions shared by every call:
 *  - Every call returns a darb_status_t and never aborts the process.
 *  - Matrices are row-major with an explicit leading dimension in elements.
 *    Activations X are cols x batch with the batch contiguous (row k of X
 *    starts at X + k * ldx); outputs Y are rows x batch (row r at Y + r * ldy).
 *  - Pointers documented as "device" must be CUDA device (or managed) memory
 *    of the current device; "host" pointers are ordinary host memory.
 *  - The caller owns every buffer it passes; a handle owns the encoded matrix
 *    and any scratch it allocates, and releases both in darb_destroy.
 *  - Work is enqueued on the caller's stream.  Only darb_encode, darb_import,
 *    darb_export, darb_sync_status, darb_rnn_reserve and darb_destroy
 *    synchronise; the product, step and sequence calls are asynchronous.
 *    darb_spmm allocates nothing; the step calls use scratch owned by the
 *    handle (darb_rnn_reserve sizes it up front).
 *  - Only two opt-in calls take scratch from the device's stream-ordered
 *    memory pool: darb_spmm_ex with DARB_PATH_TENSOR_CORES and the sequence
 *    calls.  They return it to the pool on the same stream.  The first such
 *    call on a device raises the release threshold of the device's current
 *    pool to 1 GiB if it is lower, so that freed scratch stays mapped across
 *    synchronisations; darb_spmm never touches the pool.
 *  - There is no CPU fallback: without a usable CUDA device the GPU calls
 *    return DARB_ERR_CUDA.
 */
#ifndef DARB_H
#define DARB_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#if defined(__GNUC__)
#define DARB_API __attribute__((visibility("default")))
#else
#define DARB_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct darb_handle_s *darb_handle_t;

typedef enum {
    DARB_OK = 0,
    DARB_ERR_INVALID_ARG = 1,   /* null pointer, size <= 0, ld < width, m out of [1,256],
                                   shape mismatch, unknown or destroyed handle          */
    DARB_ERR_NONFINITE = 2,     /* a NaN weight was found while encoding                 */
    DARB_ERR_OOM = 3,           /* a device or host allocation failed                    */
    DARB_ERR_CUDA = 4,          /* a CUDA runtime call or kernel launch failed           */
    DARB_ERR_TIMEOUT = 5,       /* a bounded device-side wait gave up (darb_sync_status)  */
    DARB_ERR_UNSUPPORTED = 6    /* arguments valid but not supported by these kernels    */
} darb_status_t;

typedef enum { DARB_F32 = 0, DARB_BF16 = 1 } darb_dtype_t;

/* Largest block size the format stores (offsets take at most 8 bits). */
#define DARB_MAX_BLOCK 256

/*
 * Density-adaptive block-size rule (Sec. 3.2, the worked example with matrix
 * density 21.88%).  Host only; no CUDA call.
 *   row_nnz  host int64[rows]: retained weights per row after irregular pruning,
 *            0 <= row_nnz[r] <= cols.
 *   m_out    host int32[rows]: block size per row.
 * A row denser than the whole matrix has its density rounded UP to the next
 * power-of-two density 1/m, a sparser row DOWN; m = 1 / rounded density.
 * Readings where the paper is silent: a row exactly at the matrix density is
 * rounded up; an empty row gets m_max; the result is clamped to [m_min, m_max].
 * Errors: DARB_ERR_INVALID_ARG for null pointers, rows/cols <= 0, row_nnz out of
 * range, or not 1 <= m_min <= m_max <= DARB_MAX_BLOCK.
 */
DARB_API darb_status_t darb_assign_block_sizes(const int64_t *row_nnz, int64_t rows, int64_t cols,
                                      int32_t m_min, int32_t m_max, int32_t *m_out);

/*
 * Block sizes from the weights themselves (Sec. 3.2): the K = `keep` weights
 * of largest magnitude form the mask of irregular pruning (Sec. 2, "Irregular Pruning"), used
 * only to measure each row's density; darb_assign_block_sizes then turns the
 * row counts into block sizes.  Weights tied with the K-th largest magnitude
 * all count (the paper does not break such ties), so the counts may add up to
 * slightly more than K.  Magnitudes are compared on the stored values (bf16
 * or fp32); +0 and -0 tie; an infinity is the largest.
 *   W        device, rows x cols row-major, leading dimension ldw (elements),
 *            aligned to its element size
 *   keep     1 <= keep <= rows * cols (and rows * cols < 2^32)
 *   row_nnz_out  host int64[rows] receiving the counts, or NULL
 *   m_out    host int32[rows] receiving the block sizes
 * Runs on `stream` and synchronises it.  Device scratch (8 bytes per row) is
 * kept by the library between calls, one buffer per device; concurrent calls
 * take turns on it.
 * Errors: DARB_ERR_INVALID_ARG; DARB_ERR_NONFINITE if W holds a NaN;
 * DARB_ERR_UNSUPPORTED if rows * cols >= 2^32; DARB_ERR_OOM; DARB_ERR_CUDA.
 */
DARB_API darb_status_t darb_assign_from_weights(const void *W, darb_dtype_t wtype, int64_t rows, int64_t cols,
                                                int64_t ldw, int64_t keep, int32_t m_min, int32_t m_max,
                                                int64_t *row_nnz_out, int32_t *m_out, cudaStream_t stream);

/*
 * BMWM encode (Sec. 3.1 steps (1)-(3), with the per-row block size of Sec. 3.2).
 *   W      device, rows x cols, row-major, leading dimension ldw >= cols
 *          (elements); fp32 or bf16 as wtype says.  Any alignment.
 *   m      host int32[rows], 1 <= m[r] <= DARB_MAX_BLOCK (any value, not only
 *          powers of two).
 *   out    receives a new handle.
 * Row r is split into ceil(cols / m[r]) blocks, block j covering columns
 * [j*m[r], min((j+1)*m[r], cols)) (a shorter last block still keeps one
 * weight).  In each block the weight of largest magnitude is kept; among
 * equal magnitudes (including +0 / -0) the lowest column wins.  +-Inf are the
 * largest magnitudes.  The kept value is stored bit for bit in wtype.
 * Allocates the handle's device memory, runs on `stream` and synchronises it
 * before returning; W may be freed afterwards.
 * Errors: DARB_ERR_INVALID_ARG; DARB_ERR_NONFINITE if W holds a NaN (no handle
 * is returned); DARB_ERR_OOM; DARB_ERR_CUDA.
 */
DARB_API darb_status_t darb_encode(const void *W, darb_dtype_t wtype, int64_t rows, int64_t cols,
                          int64_t ldw, const int32_t *m, darb_handle_t *out, cudaStream_t stream);

/*
 * Re-run BMWM on a new W of the handle's shape and dtype, keeping its block
 * sizes, into the handle's existing memory (e.g. after a retraining step of
 * Sec. 4's prune-retrain loop).  Asynchronous on `stream`, allocates nothing.
 * A NaN in W is recorded on the device and reported by darb_sync_status.
 * The handle must not be in use by work on another stream meanwhile.
 */
DARB_API darb_status_t darb_reencode(darb_handle_t h, const void *W, int64_t ldw, cudaStream_t stream);

/*
 * darb_reencode from weights in HOST memory (Sec. 3.1's BMWM on a W that
 * lives on the host, as a serving or training loop hands it over).
 *   W      host, rows x ldw elements of the handle's dtype, row-major,
 *          ldw >= cols; only the first cols of each row are read.
 *   W_dev  device, rows x ldw elements (aligned to the element size), owned
 *          by the caller: W is copied there (rows of cols elements at pitch
 *          ldw), then re-encoded from it; it keeps the copy afterwards.
 * The copy and the encode are ordered on `stream`.  With pinned host memory
 * the call is asynchronous; with pageable memory the copy completes before
 * the call returns.  Allocates nothing.
 * Errors: as darb_reencode, and DARB_ERR_INVALID_ARG for a null W_dev;
 * DARB_ERR_CUDA if the copy cannot be issued.
 */
DARB_API darb_status_t darb_reencode_host(darb_handle_t h, const void *W, int64_t ldw, void *W_dev,
                                          cudaStream_t stream);

/* Synchronise `stream` and report what the handle's kernels recorded on the
 * device since the last call, then clear it: DARB_ERR_TIMEOUT if a bounded
 * device wait (for a bulk copy, or at a sequence call's grid barrier) gave up
 * -- results of that call are not valid, the device stays usable -- else
 * DARB_ERR_NONFINITE if a (re)encode met a NaN, else DARB_OK.                */
DARB_API darb_status_t darb_sync_status(darb_handle_t h, cudaStream_t stream);

/*
 * Y = W_darb X: for row r and batch column b,
 *   Y[r, b] = sum_j val[r, j] * X[j*m_r + off[r, j], b]
 * (block j of the row selects one activation row, Sec. 3.2 / Fig. 6(b)).
 *   X  device fp32, cols x batch, ldx >= batch, 4-byte aligned.
 *   Y  device fp32, rows x batch, ldy >= batch; overwritten.  Must not
 *      overlap X.
 * Every kept weight is multiplied only by the activation its block selects
 * (a NaN or infinity in an activation row that no kept weight selects does
 * not reach Y), in fp32, on the CUDA cores, for every dtype and batch.
 * Asynchronous on `stream`; allocates nothing; the handle is only read, so
 * calls on several streams may share it.  A bounded device wait that gave up
 * is reported by darb_sync_status.
 * Errors: DARB_ERR_INVALID_ARG (null, batch <= 0, ld < batch, X or Y not
 * 4-byte aligned, Y overlapping X); DARB_ERR_UNSUPPORTED (batch above 2^19);
 * DARB_ERR_CUDA.
 */
DARB_API darb_status_t darb_spmm(darb_handle_t h, const float *X, int64_t ldx, int64_t batch, float *Y,
                        int64_t ldy, cudaStream_t stream);

/*
 * darb_spmm with X and Y in HOST memory (Sec. 3.2's product as a caller
 * outside the GPU sees it: activations in, outputs back).
 *   X      host fp32, cols x batch, ldx >= batch.
 *   Y      host fp32, rows x batch, ldy >= batch; receives the product.
 *   X_dev  device fp32, cols x batch (rows of batch floats), owned by the
 *          caller: X is copied there first.
 *   Y_dev  device fp32, rows x batch (rows of batch floats), owned by the
 *          caller: the product is written there, then copied into Y.  Must
 *          not overlap X_dev.
 * Copy in, product (darb_spmm on X_dev, Y_dev) and copy out are ordered on
 * `stream`; with pinned host memory the call is asynchronous and Y holds the
 * product once `stream` has been synchronised.  Allocates nothing.
 * Errors: as darb_spmm (X_dev and Y_dev checked as its X and Y, X and Y for
 * null); DARB_ERR_CUDA if a copy cannot be issued.
 */
DARB_API darb_status_t darb_spmm_host(darb_handle_t h, const float *X, int64_t ldx, int64_t batch, float *Y,
                                      int64_t ldy, float *X_dev, float *Y_dev, cudaStream_t stream);

/* Which kernels compute a product (the paper has no counterpart: these are two
 * ways of evaluating the same sum on the GPU).                               */
typedef enum {
    DARB_PATH_AUTO = 0,          /* what darb_spmm does: the CUDA-core gather        */
    DARB_PATH_CUDA_CORES = 1,    /* gather-multiply-add on the CUDA cores (any weights) */
    DARB_PATH_TENSOR_CORES = 2   /* densified tiles on the tensor cores (bf16 weights) */
} darb_path_t;

/*
 * darb_spmm with the kernel family chosen by the caller.  DARB_PATH_AUTO and
 * DARB_PATH_CUDA_CORES are darb_spmm.  DARB_PATH_TENSOR_CORES is an opt-in
 * alternative that is not the paper's per-block selection: it multiplies every activation
 * of a stage by the densified tile, zeros included, with X split into two
 * bf16 parts (x = hi + lo): |Y - exact| <= 2^-16 * sum |val * x| plus fp32
 * rounding, a NaN or infinity in X may make rows NaN that do not select it,
 * and |x| must stay below the largest bf16.  It needs bf16 weights, and it
 * takes the split of X (4 bytes per element of X, batch rounded up to 8) from
 * the device's stream-ordered memory pool on `stream` for the duration of the
 * call (DARB_ERR_OOM if the pool cannot supply it); the CUDA-core path
 * allocates nothing.
 * Errors: as darb_spmm; DARB_ERR_INVALID_ARG for an unknown path;
 * DARB_ERR_UNSUPPORTED if DARB_PATH_TENSOR_CORES cannot take the call.
 */
DARB_API darb_status_t darb_spmm_ex(darb_handle_t h, const float *X, int64_t ldx, int64_t batch, float *Y,
                                    int64_t ldy, darb_path_t path, cudaStream_t stream);

/* The kernel family darb_spmm takes for this handle and batch (*path: always
 * DARB_PATH_CUDA_CORES), and how many kernels it launches per call (*kernels:
 * 1).  Host only.
 * Errors: DARB_ERR_INVALID_ARG (unknown handle, batch <= 0, null outputs). */
DARB_API darb_status_t darb_spmm_path(darb_handle_t h, int64_t batch, darb_path_t *path, int32_t *kernels);

/*
 * One LSTM cell step whose gate matrix is the handle (rows = 4H, cols = I + H),
 * multiplied with the stacked input [x_t; h_{t-1}].  Gate rows [0,H) = i,
 * [H,2H) = f, [2H,3H) = g, [3H,4H) = o (the paper names LSTMs, Sec. 4.1, but
 * writes no cell equations; this is the standard cell):
 *   c_t = sigmoid(f) * c_{t-1} + sigmoid(i) * tanh(g),  h_t = sigmoid(o) * tanh(c_t)
 *   x      device fp32, I x B (batch contiguous); may be NULL when I == 0
 *   h_prev, c_prev   device fp32, H x B
 *   bias   device fp32 [4H] added to the gate pre-activations, or NULL
 *   h_out, c_out     device fp32, H x B; must not overlap any input
 * Uses scratch owned by the handle (4H x B floats of gate sums and H counters),
 * allocated by the first step call that needs more than the handle holds (that
 * call synchronises); call darb_rnn_reserve first to size it up front.  Step
 * calls on one handle must be ordered on one stream.
 * Errors: DARB_ERR_INVALID_ARG (null, shape mismatch, B <= 0); DARB_ERR_OOM;
 * DARB_ERR_CUDA.
 */
DARB_API darb_status_t darb_lstm_step(darb_handle_t h, int64_t I, int64_t H, int64_t B, const float *x,
                             const float *h_prev, const float *c_prev, const float *bias,
                             float *h_out, float *c_out, cudaStream_t stream);

/*
 * One GRU cell step whose gate matrix is the handle (rows = 3H, cols = I + H).
 * Gate rows [0,H) = r, [H,2H) = z, [2H,3H) = n; columns [0,I) multiply x_t and
 * [I,I+H) multiply h_{t-1}, and the two parts are kept apart (the paper names
 * GRUs, Sec. 4.1, without equations; this is the standard cell):
 *   a = W[:, :I] x + b_ih,  bh = W[:, I:] h + b_hh
 *   r = sigmoid(a_r + bh_r), z = sigmoid(a_z + bh_z), n = tanh(a_n + r * bh_n)
 *   h_t = (1 - z) * n + z * h_{t-1}
 *   x device fp32 I x B (NULL allowed when I == 0); h_prev device fp32 H x B;
 *   b_ih, b_hh device fp32 [3H] or NULL; h_out device fp32 H x B, not
 *   overlapping any input.
 * Scratch, ordering and errors as for darb_lstm_step (scratch 2 x 3H x B floats).
 */
DARB_API darb_status_t darb_gru_step(darb_handle_t h, int64_t I, int64_t H, int64_t B, const float *x,
                            const float *h_prev, const float *b_ih, const float *b_hh,
                            float *h_out, cudaStream_t stream);

/*
 * T consecutive LSTM steps (the cell of darb_lstm_step) in one persistent
 * launch: the recurrence of an RNN layer over a whole input sequence (the
 * LSTM models of Sec. 4.1 run one step per token).  Each CTA keeps its share
 * of the gate matrix decoded in shared memory for all T steps and the steps
 * are separated by a grid-wide barrier, so W is read from memory once per
 * call instead of once per step.
 *   x_seq  device fp32, T x I x B (step t at x_seq + t*I*B); NULL allowed when I == 0
 *   h0, c0 device fp32, H x B: the state before the first step
 *   bias   device fp32 [4H] or NULL
 *   h_seq  device fp32, T x H x B: h_t of every step
 *   c_seq  device fp32, T x H x B: c_t of every step, or NULL
 *   c_last device fp32, H x B: c_T, or NULL
 * No output may overlap an input or another output.  T == 0 launches nothing
 * and copies c0 to c_last.  The results equal T calls of darb_lstm_step up to
 * the order of the fp32 additions inside each gate sum.
 * When x_t is at least a third of the stacked input (2I >= H), the sequence
 * has 64 to 2^19 columns (T * B) and the workspace below stays under 1 GiB,
 * the x parts of all T steps are computed first as one product
 * W [x_0 .. x_{T-1}; 0] of T * B columns (darb_spmm's kernels and numerics,
 * the CUDA-core gather); the recurrence then stages and
 * multiplies only h_{t-1}.
 * Resources: one cooperative launch of one CTA per SM (at most H CTAs); a
 * stream-ordered workspace of 256 bytes, plus H x B floats when c_last is
 * NULL and the cell state does not fit on chip, plus (I + H + 4H) x T*B
 * floats when the x parts are precomputed.  A barrier wait longer than 1 s
 * ends the launch and is reported by darb_sync_status as DARB_ERR_TIMEOUT.
 * For testing that path, the environment variable DARB_TEST_BARRIER_TIMEOUT=1
 * (read at every launch) shortens the limit to 1 ms and makes CTA 0 withhold
 * its first arrival, so the launch times out on purpose.
 * Errors: DARB_ERR_INVALID_ARG (shape mismatch, null, overlap, T < 0);
 * DARB_ERR_UNSUPPORTED when a CTA's share of the decoded matrix plus one
 * column tile of [x_t; h_{t-1}] does not fit in shared memory, or cols > 65535;
 * DARB_ERR_OOM; DARB_ERR_CUDA.
 */
DARB_API darb_status_t darb_lstm_sequence(darb_handle_t h, int64_t T, int64_t I, int64_t H, int64_t B,
                                          const float *x_seq, const float *h0, const float *c0,
                                          const float *bias, float *h_seq, float *c_seq, float *c_last,
                                          cudaStream_t stream);

/*
 * T consecutive GRU steps (the cell of darb_gru_step) in one persistent
 * launch, as darb_lstm_sequence.
 *   x_seq device fp32, T x I x B (NULL allowed when I == 0); h0 device fp32
 *   H x B; b_ih, b_hh device fp32 [3H] or NULL; h_seq device fp32, T x H x B,
 *   not overlapping any input.
 * Precomputed x parts, resources and errors as darb_lstm_sequence (workspace
 * with 3H rows of x parts).
 */
DARB_API darb_status_t darb_gru_sequence(darb_handle_t h, int64_t T, int64_t I, int64_t H, int64_t B,
                                         const float *x_seq, const float *h0, const float *b_ih,
                                         const float *b_hh, float *h_seq, cudaStream_t stream);

/*
 * darb_lstm_step without any allocation: the same step, same arguments and
 * same results, with its scratch (gate sums and arrival counters) in one
 * fixed array of 4 MiB inside this library instead of memory owned by the
 * handle.  It is for callers that cannot let a library call cudaMalloc at step
 * time -- a serving loop with a fixed memory budget, code that must not
 * synchronise the device mid-stream, or allocations that must all go through
 * the caller's own pool.  The paper has no counterpart; it is a property of
 * this library's interface only.
 *   - Limit: 4H*B floats (rounded up to 256 bytes) plus H*ceil(B/t) counters
 *     (t = 1, 2, 4 or 8 by batch) must fit in 4 MiB; larger calls return
 *     DARB_ERR_UNSUPPORTED and do nothing.
 *   - Every GPU that loads the library holds the 4 MiB until the process exits.
 *   - The first call on each device looks up the array's device address (one
 *     cudaGetSymbolAddress); make that first call before any stream capture.
 *   - All calls on a device share the one array, which keeps the last call's
 *     contents; each call clears the counters it needs on `stream`.  Calls that
 *     overlap on the GPU (other streams, or unordered launches) race on it.
 * Errors as darb_lstm_step, plus DARB_ERR_UNSUPPORTED for the size limit.
 */
DARB_API darb_status_t darb_lstm_step_noalloc(darb_handle_t h, int64_t I, int64_t H, int64_t B,
                                              const float *x, const float *h_prev, const float *c_prev,
                                              const float *bias, float *h_out, float *c_out,
                                              cudaStream_t stream);

/* Size the handle's RNN step scratch for batches up to max_batch now, so that
 * later step calls allocate nothing (e.g. before capturing them in a CUDA
 * graph).  Synchronises the device.  Errors: INVALID_ARG, OOM, CUDA.          */
DARB_API darb_status_t darb_rnn_reserve(darb_handle_t h, int64_t max_batch);

typedef struct {
    int64_t rows, cols;
    int64_t nnzb;            /* kept weights = blocks = sum_r ceil(cols / m_r)           */
    darb_dtype_t wtype;
    int32_t nbins;           /* distinct block sizes                                     */
    int32_t ngroups;         /* 32-row groups the kernels work on                        */
    int64_t value_bytes;     /* nnzb * sizeof(value): the values the paper stores       */
    int64_t offset_bytes;    /* stored offsets: 4 bits per block if m <= 16, else 8     */
    int64_t meta_bytes;      /* per-row block size and pointer (int32 + uint16)         */
    int64_t index_bits_min;  /* sum over blocks of ceil(log2 m): the paper's index bits */
    int64_t device_bytes;    /* device memory the handle holds (incl. padding, scratch) */
} darb_info_t;

/* Shape and storage accounting of a handle (Sec. 4.2 index-storage analysis). */
DARB_API darb_status_t darb_info(darb_handle_t h, darb_info_t *info);

/*
 * Copy the encoding out in canonical order: blocks in (row, j) order.
 *   val      host, nnzb values of the handle's dtype (fp32 or bf16 bits)
 *   off      host uint8[nnzb], position of the kept weight inside its block
 *   blk_ptr  host int64[rows + 1], first block of each row; blk_ptr[rows] = nnzb
 *   m        host int32[rows], block size of each row
 * Any of the four may be NULL to skip it.  Synchronises the device.
 */
DARB_API darb_status_t darb_export(darb_handle_t h, void *val, uint8_t *off, int64_t *blk_ptr, int32_t *m);

/* Build a handle from canonical host arrays (the inverse of darb_export).
 * off[p] must be < m[r] and j*m[r] + off[p] < cols.  Synchronises `stream`.  */
DARB_API darb_status_t darb_import(const void *val, const uint8_t *off, const int32_t *m,
                          darb_dtype_t wtype, int64_t rows, int64_t cols, darb_handle_t *out,
                          cudaStream_t stream);

/* Whether the library's kernels are launched with programmatic dependent
 * launch (PDL: a kernel may start its prologue, and read the handle's
 * immutable data, while the previous kernel on the stream drains; its reads
 * of X and writes of Y still wait for that kernel).  Process wide, on by
 * default; applies to launches made after the call (a CUDA graph keeps what
 * it captured).  For measuring the overlap; results are the same either way.
 * The paper has no counterpart.  Always DARB_OK.                             */
DARB_API darb_status_t darb_set_pdl(int enabled);

/* Release a handle and all device memory it owns; NULL is a no-op.  Waits for
 * the device to finish using it.                                              */
DARB_API darb_status_t darb_destroy(darb_handle_t h);

/* Static, human-readable name of a status code. */
DARB_API const char *darb_status_string(darb_status_t s);

#ifdef __cplusplus
}
#endif

#endif /* DARB_H */
