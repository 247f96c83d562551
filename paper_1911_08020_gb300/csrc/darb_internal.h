// darb_internal.h -- device layout of an encoded DARB matrix and the launchers
// that the C ABI (darb_api.cu) calls.  Internal to libdarb.
//
// Layout in HBM (one allocation per handle):
//
//  * Rows are binned by block size m (Sec. 3.2 gives every row its own m) and
//    each bin is cut into groups of 32 rows ("slots"); the last group of a bin
//    is zero-padded.  Groups are ordered by ascending m, i.e. by descending
//    blocks per row, so the heaviest groups are launched first.
//  * Values of a group are stored chunk-interleaved: chunk c holds blocks
//    [8c, 8c+8) of every slot, slot-major, 8 values per slot.  A warp whose
//    lane i works on slot i reads a chunk with one 16-byte (bf16) or two
//    16-byte (fp32) loads per lane, all 32 lanes contiguous.
//  * Offsets are packed per chunk and slot into a 4-byte record of eight
//    4-bit offsets when m <= 16, or an 8-byte record of eight 8-bit offsets
//    otherwise (the paper's log2 m bits per index, Sec. 4.2, rounded up to a
//    nibble or a byte so that they unpack with shifts in registers).
//  * rowmap[g*32 + i] is the matrix row held by slot i of group g (-1: pad);
//    rowloc[r] = g*32 + i is its inverse.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "darb.h"

namespace darb {

constexpr int kSlots = 32;   // rows per group
constexpr int kChunk = 8;    // blocks per chunk
constexpr int kEncTileElems = 12288;   // columns of W the encoder stages per tile, at most

// Blocks of a row with block size m that one encoder tile covers: whole
// blocks, a multiple of the chunk so that offset records never straddle tiles.
inline __host__ __device__ int enc_tile_blocks(int m) { return (kEncTileElems / m) / kChunk * kChunk; }

// The bf16 row encoder (block sizes powers of two from 8 to 256) takes tiles of
// kRowPassElems columns: kRowPassElems / m blocks, a multiple of the chunk.
constexpr int kRowPassElems = 2048;

struct Group {
    int32_t m;        // block size shared by the group's rows
    int32_t n;        // blocks per row, ceil(cols / m)
    int32_t nrows;    // slots in use (1..32)
    int32_t nib;      // 1: 4-bit offsets (m <= 16), 0: 8-bit offsets
    int64_t val_off;  // element index of chunk 0 / slot 0 in the value array
    int64_t off_off;  // uint32 word index of chunk 0 / slot 0 in the offset array
};

// One CTA's share of a product of batch_kernel: a row set (a run of up to 2^l
// consecutive 32-row groups of one block-size bin) and the chunks of the set's
// blocks that this CTA multiplies.  The ksub CTAs that share a set are
// consecutive ranks of one thread-block cluster (qsub = this CTA's index among
// them); they add their partial sums through distributed shared memory.
struct WorkItem {
    int32_t g0;      // first group of the set
    int16_t ng;      // groups in the set; 0: an idle rank that only joins the cluster's barriers
    int8_t qsub;     // this CTA's index among the CTAs that share the set
    int8_t ksub;     // CTAs that share the set (consecutive ranks of one cluster)
    int32_t c0, c1;  // chunks [c0, c1) of the set's blocks
};
constexpr int kWorkLevels = 4;   // row sets of up to 1, 2, 4, 8 groups

// A row set of the resident-activation product (xres.cuh): a run of
// ng <= kXresMaxGroups consecutive groups of one bin, in one 48-byte record (no dependent lookups).
// The groups of a bin have equal block counts, so group g0 + i starts i group
// strides after the first: values at val_off + i * nch * 256, offsets at
// off_off + i * nch * 32 * (nib ? 1 : 2) (nch = ceil(n / 8)); all groups are
// full except possibly the last.
struct __align__(16) SetGeo {
    int32_t g0;           // first group
    int32_t ng;           // groups (1..kXresMaxGroups)
    int32_t m, n;         // block size and blocks per row
    int32_t nib;          // 1: 4-bit offsets
    int32_t nrows_last;   // rows in use of the last group
    int64_t val_off;      // Group::val_off of the first group
    int64_t off_off;      // Group::off_off of the first group
    int64_t pad;
};
constexpr int kXresTables = 2;   // row-set tables of xres: 2 and 4 groups of the heaviest bin
// Groups of an xres row set, at most: its partial sums (128 rows x 32 columns)
// are one 16 KB buffer, which leaves the activation slice room enough for
// clusters of 6 on the widest layers
constexpr int kXresMaxGroups = 4;
constexpr int kWorkSplits = 4;   // clusters of 1, 2, 4, 8 CTAs

// Everything a kernel needs to read an encoded matrix.
struct Format {
    const Group *groups;
    const int32_t *rowmap;   // [ngroups * 32]
    const int32_t *rowloc;   // [rows]
    const int32_t *row_m;    // [rows]
    const void *vals;        // fp32 or bf16 bit patterns
    const uint32_t *offs;
    int32_t *status;         // sticky device status bits (NaN seen, wait timed out)
    // CTA work tables of batch_kernel: items[l][c] for row sets of up to 2^l
    // groups and clusters of 2^c CTAs (nitems[l][c] entries, a multiple of 2^c;
    // item_work[l][c] = the most group-chunks any one item multiplies)
    const WorkItem *items[kWorkLevels][kWorkSplits];
    int32_t nitems[kWorkLevels][kWorkSplits];
    int32_t item_work[kWorkLevels][kWorkSplits];
    int32_t nch_max;         // chunks of a row of the smallest block size
    // HOST memory (never read by a kernel): for the row sets of level l in the
    // order of items[l][0], set_prefix[l][s] = sum of the work (groups x
    // chunks per row) of sets [0, s); nitems[l][0] + 1 entries
    const int64_t *set_prefix[kWorkLevels];
    // row sets of xres (SetGeo): table i sizes the sets of every bin to about
    // the work of 2 << i groups of the heaviest bin (at most kXresMaxGroups); device
    // records, and on the HOST the prefix sums of their work (group-chunks)
    const SetGeo *xsets[kXresTables];
    int32_t nxsets[kXresTables];
    const int64_t *xset_prefix[kXresTables];
    const SetGeo *xsets_host[kXresTables];   // HOST copies of xsets
    int32_t ngroups;
    int32_t bf16;            // value dtype: 0 fp32, 1 bf16
    int32_t m_max;           // largest block size of any row
    int32_t m_min;           // smallest block size of any row (0: unknown)
    int64_t rows, cols;
};

// One encoder tile (a row, or a run of whole blocks of a long row), resolved
// on the host: where it sits in W and where its blocks go in the format, so
// that the encoder gets a tile from one 32-byte load instead of a chain of
// dependent lookups (tile -> row -> slot -> group).
struct __align__(16) EncTile {
    int32_t row;       // matrix row
    int32_t c0;        // first column, (first block) * m
    int32_t span;      // columns of W in the tile (the row's last tile may stop short)
    int16_t m;         // the row's block size
    int16_t nb;        // blocks in the tile, a multiple of the chunk except at the row's end
    int64_t val_base;  // value index of the tile's first block in the row's slot
    int64_t off_base;  // offs word index of the tile's first record (one word if m <= 16, else two)
};

// Writable view used by the encoder.
struct EncodeTarget {
    const EncTile *tiles;    // every encoder tile, row-major
    int32_t ntiles;
    int32_t max_tile;        // elements of the largest tile, max over tiles of nb * m (zero padding included)
    const EncTile *row_tiles;   // tiles of the bf16 row encoder (kRowPassElems columns), row-major
    int32_t n_row_tiles;        // 0 unless the weights are bf16 and every block size a power of two in [8, 256]
    void *vals;
    uint32_t *offs;
    int32_t bf16;
    int64_t rows, cols;
};

// Scratch for the fused RNN steps: gate sums and per-(unit, batch tile) arrival counters.
struct RnnScratch {
    float *gates;      // rows x B (LSTM) or 2 x rows x B (GRU: x part then h part)
    int32_t *counters; // units x batch tiles, zero between launches
};

cudaError_t launch_encode(const EncodeTarget &t, const void *W, int64_t ldw, int32_t *status,
                          cudaStream_t stream);

// Batch > 4 path (spmm_batch.cu).
cudaError_t launch_spmm_batch(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                              int64_t ldy, bool early, cudaStream_t stream);

// Tensor-core path (spmm_tc.cu): bf16 weights only; cudaErrorNotSupported
// when the call does not fit it.
cudaError_t launch_spmm_tc(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                           int64_t ldy, bool early, cudaStream_t stream);

// `early`: the handle's data is known to be complete, so a kernel may start
// reading it before the previous kernel on the stream has finished (PDL).
// `path`: a darb_path_t; DARB_PATH_AUTO and DARB_PATH_CUDA_CORES both take the
// CUDA-core gather.  cudaErrorNotSupported if DARB_PATH_TENSOR_CORES was asked
// for a call the tensor-core kernel cannot take.
// Y = (the first col_limit columns of W_darb) (the first col_limit rows of X),
// for X whose rows from col_limit on are zero: the product of launch_spmm,
// on xres without the columns from col_limit on where it can take the call.
cudaError_t launch_spmm_prefix(const Format &f, int64_t col_limit, const float *X, int64_t ldx, int64_t batch,
                               float *Y, int64_t ldy, bool early, cudaStream_t stream);

cudaError_t launch_spmm(const Format &f, const float *X, int64_t ldx, int64_t batch, float *Y,
                        int64_t ldy, bool early, int path, cudaStream_t stream);

// `early` as for launch_spmm (the handle's values may be read before the
// previous kernel on the stream finishes).
cudaError_t launch_lstm_step(const Format &f, int64_t I, int64_t H, int64_t B, const float *x,
                             const float *h_prev, const float *c_prev, const float *bias,
                             float *h_out, float *c_out, RnnScratch s, cudaStream_t stream,
                             bool early = false);

cudaError_t launch_gru_step(const Format &f, int64_t I, int64_t H, int64_t B, const float *x,
                            const float *h_prev, const float *b_ih, const float *b_hh,
                            float *h_out, RnnScratch s, cudaStream_t stream, bool early = false);

// T steps of an RNN layer in one persistent cooperative launch (sequence.cu).
// row_m: the host copy of the per-row block sizes.  cudaErrorNotSupported
// when a CTA's share of the matrix and one input tile do not fit on chip.
cudaError_t launch_lstm_sequence(const Format &f, const int32_t *row_m, int64_t T, int64_t I, int64_t H, int64_t B,
                                 const float *x, const float *h0, const float *c0, const float *bias, float *h_seq,
                                 float *c_seq, float *c_last, cudaStream_t stream);
cudaError_t launch_gru_sequence(const Format &f, const int32_t *row_m, int64_t T, int64_t I, int64_t H, int64_t B,
                                const float *x, const float *h0, const float *b_ih, const float *b_hh, float *h_seq,
                                cudaStream_t stream);

struct RnnArgs;
// Batch > 4 RNN steps (rnn_batch.cu); mode is kModeLstm or kModeGru.
cudaError_t launch_rnn_batch(const Format &f, const RnnArgs &ra, int mode, bool early, cudaStream_t stream);

// Batch-tile width the RNN step kernels use for a batch of B (sizes the counters).
int rnn_batch_tile(int64_t B);

// Streaming multiprocessors of the current device (cached).
int sm_count();

// Stream-ordered scratch (cudaMallocAsync).  The first call on a device raises
// the release threshold of the device's current memory pool to kPoolKeep (it
// never lowers it): scratch freed before a synchronisation then stays mapped
// for the next call instead of being unmapped at the synchronisation and mapped
// again, which costs more than the kernels the scratch serves.
constexpr uint64_t kPoolKeep = uint64_t(1) << 30;
cudaError_t stream_alloc(void **p, size_t bytes, cudaStream_t stream);

// Row densities of Sec. 3.2's first step (assign.cu): row_nnz[r] = number of
// weights of row r whose magnitude is >= the keep-th largest magnitude of W.
// work: 4608 bytes of device scratch; nan_flag: device int, set if W has a NaN.
cudaError_t launch_topk_row_nnz(const void *W, bool bf16, int64_t rows, int64_t cols, int64_t ldw, int64_t keep,
                                int64_t *row_nnz, void *work, int32_t *nan_flag, cudaStream_t stream);

// The argument checks of darb_lstm_step and the handle's read-only view, for
// an entry point that brings its own scratch.  Allocates nothing.
darb_status_t lstm_step_view(darb_handle_t h, int64_t I, int64_t H, int64_t B, const float *x,
                             const float *h_prev, const float *c_prev, const float *bias,
                             const float *h_out, const float *c_out, Format *f);

}  // namespace darb
