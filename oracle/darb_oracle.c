/*
 * darb_oracle.c -- plain, slow CPU oracle for DARB (arXiv 1911.08020).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the library calls this file: only the
 * test suite, the package smoke check and the benchmark's CPU-baseline leg load
 * it.  It shares no code, header, table or helper with the CUDA path.
 *
 * Every function is the plain definition of one step of the method, written as
 * loops in the paper's order, accumulating in double precision:
 *
 *   oracle_topk_row_nnz_*      Sec. 3.2's first step with Sec. 2's irregular
 *                              pruning: each row's count of the K weights of
 *                              largest magnitude (the row density)
 *   oracle_assign_block_sizes  Sec. 3.2 (density-adaptive rounding rule)
 *   oracle_block_pointers      Sec. 3.1 step (1): ceil(cols / m) blocks per row
 *   oracle_encode_f32/_bf16    Sec. 3.1 BMWM steps (1)-(3), per-row block size
 *                              of Sec. 3.2; lowest index wins a tie
 *   oracle_masked_dense        the dense matrix M (.) W that the encoding stands for
 *   oracle_darb_spmm           y = W_darb x via the per-block selection of
 *                              Sec. 3.2 (Fig. 6(b): block j of a row with block
 *                              size m picks activation j*m + offset)
 *   oracle_lstm_step           one LSTM cell step on the DARB gate matrix
 *   oracle_gru_step            one GRU cell step on the DARB gate matrix
 *
 * Status codes: 0 ok, 1 invalid argument, 2 non-finite (NaN) weight.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_OK 0
#define OR_INVALID 1
#define OR_NONFINITE 2

int oracle_set_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
    return omp_get_max_threads();
#else
    (void)n;
    return 1;
#endif
}

/* ------------------------------------------------------------------------ */
/* Sec. 3.2 starts from the mask of irregular pruning (Sec. 2, "Irregular Pruning": keep the K
 * weights of largest magnitude) and only counts it: row r's density is its
 * number of kept weights over cols.  Here: sort all magnitudes (widened
 * exactly to double) in decreasing order, take the K-th one as the threshold t,
 * and count per row the weights with |w| >= t.
 * Reading: the paper does not say which of several weights equal to the K-th
 * magnitude are kept; all of them count, so the counts may add up to more than
 * K.  A NaN weight is rejected.                                               */
static int cmp_desc(const void *a, const void *b) {
    const double x = *(const double *)a, y = *(const double *)b;
    return (x < y) - (x > y);
}

#define TOPK_BODY(LOAD)                                                               \
    if (!W || !row_nnz || rows <= 0 || cols <= 0 || ldw < cols || keep < 1 ||         \
        keep > rows * cols)                                                           \
        return OR_INVALID;                                                            \
    double *mag = (double *)malloc((size_t)(rows * cols) * sizeof(double));           \
    if (!mag) return OR_INVALID;                                                      \
    for (int64_t r = 0; r < rows; ++r)                                                \
        for (int64_t c = 0; c < cols; ++c) {                                          \
            const double v = LOAD(W[r * ldw + c]);                                    \
            if (isnan(v)) {                                                           \
                free(mag);                                                            \
                return OR_NONFINITE;                                                  \
            }                                                                         \
            mag[r * cols + c] = fabs(v);                                              \
        }                                                                             \
    qsort(mag, (size_t)(rows * cols), sizeof(double), cmp_desc);                      \
    const double t = mag[keep - 1];                                                   \
    free(mag);                                                                        \
    for (int64_t r = 0; r < rows; ++r) {                                              \
        int64_t n = 0;                                                                \
        for (int64_t c = 0; c < cols; ++c)                                            \
            if (fabs(LOAD(W[r * ldw + c])) >= t) ++n;                                 \
        row_nnz[r] = n;                                                               \
    }                                                                                 \
    return OR_OK;

static double bf16_bits_value(uint16_t bits);

int oracle_topk_row_nnz_f32(const float *W, int64_t rows, int64_t cols, int64_t ldw, int64_t keep,
                            int64_t *row_nnz) {
    TOPK_BODY((double))
}

int oracle_topk_row_nnz_bf16(const uint16_t *W, int64_t rows, int64_t cols, int64_t ldw, int64_t keep,
                             int64_t *row_nnz) {
    TOPK_BODY(bf16_bits_value)
}

/* ------------------------------------------------------------------------ */
/* Sec. 3.2: a row whose density is above the matrix density is rounded UP to
 * a power-of-two density 1/m, a row below it is rounded DOWN; the block size is
 * the reciprocal of the rounded density.  Densities are compared as integers:
 * nnz_r / cols  vs  total / (rows * cols)   <=>   nnz_r * rows  vs  total.
 * Readings (the paper states only the strict cases): a row exactly at the
 * matrix density is rounded up; an empty row takes m_max; the result is
 * clamped to [m_min, m_max].                                                  */
int oracle_assign_block_sizes(const int64_t *row_nnz, int64_t rows, int64_t cols,
                              int32_t m_min, int32_t m_max, int32_t *m_out) {
    if (!row_nnz || !m_out || rows <= 0 || cols <= 0 || m_min < 1 || m_max < m_min)
        return OR_INVALID;
    int64_t total = 0;
    for (int64_t r = 0; r < rows; ++r) {
        if (row_nnz[r] < 0 || row_nnz[r] > cols) return OR_INVALID;
        total += row_nnz[r];
    }
    for (int64_t r = 0; r < rows; ++r) {
        int64_t nnz = row_nnz[r];
        int64_t m;
        if (nnz == 0) {
            m = m_max;
        } else if (nnz * rows >= total) {
            /* round density up: the largest power of two m with 1/m >= nnz/cols */
            m = 1;
            while (2 * m * nnz <= cols) m *= 2;
        } else {
            /* round density down: the smallest power of two m with 1/m <= nnz/cols */
            m = 1;
            while (m * nnz < cols) m *= 2;
        }
        if (m < m_min) m = m_min;
        if (m > m_max) m = m_max;
        m_out[r] = (int32_t)m;
    }
    return OR_OK;
}

/* Sec. 3.1 step (1): a row of `cols` elements split into blocks of size m has
 * ceil(cols / m) blocks (a shorter last block still counts as a block).
 * blk_ptr[r] is the index of row r's first block; blk_ptr[rows] = total.      */
int oracle_block_pointers(const int32_t *m, int64_t rows, int64_t cols, int64_t *blk_ptr) {
    if (!m || !blk_ptr || rows <= 0 || cols <= 0) return OR_INVALID;
    blk_ptr[0] = 0;
    for (int64_t r = 0; r < rows; ++r) {
        if (m[r] < 1) return OR_INVALID;
        int64_t n = (cols + m[r] - 1) / m[r];
        blk_ptr[r + 1] = blk_ptr[r] + n;
    }
    return OR_OK;
}

static double bf16_value(uint16_t bits) {
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static double bf16_bits_value(uint16_t bits) { return bf16_value(bits); }

static double f32_value(float f) { return (double)f; }

/* BMWM, Sec. 3.1 steps (1)-(3), with the per-row block size of Sec. 3.2:
 * for every row r and block j covering columns [j*m, min((j+1)*m, cols)),
 * keep the element of largest magnitude; on equal magnitudes the lowest column
 * wins (first one met scanning left to right, strict '>' comparison).
 * val receives the kept element bit for bit, off its position inside the block. */
#define ENCODE_BODY(LOAD)                                                             \
    if (!W || !m || !val || !off || !blk_ptr || rows <= 0 || cols <= 0 || ldw < cols) \
        return OR_INVALID;                                                            \
    for (int64_t r = 0; r < rows; ++r)                                                \
        for (int64_t c = 0; c < cols; ++c)                                            \
            if (isnan(LOAD(W[r * ldw + c]))) return OR_NONFINITE;                     \
    if (oracle_block_pointers(m, rows, cols, blk_ptr) != OR_OK) return OR_INVALID;    \
    _Pragma("omp parallel for schedule(static)")                                      \
    for (int64_t r = 0; r < rows; ++r) {                                              \
        int64_t mr = m[r];                                                            \
        int64_t n = blk_ptr[r + 1] - blk_ptr[r];                                      \
        for (int64_t j = 0; j < n; ++j) {                                             \
            int64_t lo = j * mr;                                                      \
            int64_t hi = lo + mr < cols ? lo + mr : cols;                             \
            int64_t best = lo;                                                        \
            for (int64_t c = lo + 1; c < hi; ++c)                                     \
                if (fabs(LOAD(W[r * ldw + c])) > fabs(LOAD(W[r * ldw + best])))       \
                    best = c;                                                         \
            val[blk_ptr[r] + j] = W[r * ldw + best];                                  \
            off[blk_ptr[r] + j] = (uint8_t)(best - lo);                               \
        }                                                                             \
    }                                                                                 \
    return OR_OK;

int oracle_encode_f32(const float *W, int64_t rows, int64_t cols, int64_t ldw,
                      const int32_t *m, float *val, uint8_t *off, int64_t *blk_ptr) {
    for (int64_t r = 0; m && r < rows; ++r)
        if (m[r] < 1 || m[r] > 256) return OR_INVALID;
    ENCODE_BODY(f32_value)
}

int oracle_encode_bf16(const uint16_t *W, int64_t rows, int64_t cols, int64_t ldw,
                       const int32_t *m, uint16_t *val, uint8_t *off, int64_t *blk_ptr) {
    for (int64_t r = 0; m && r < rows; ++r)
        if (m[r] < 1 || m[r] > 256) return OR_INVALID;
    ENCODE_BODY(bf16_value)
}

/* The dense matrix the encoding stands for: zero everywhere except, in every
 * block, the kept weight at column j*m + off.  Wd is rows x cols, row-major. */
int oracle_masked_dense(const double *val, const uint8_t *off, const int64_t *blk_ptr,
                        const int32_t *m, int64_t rows, int64_t cols, double *Wd) {
    if (!val || !off || !blk_ptr || !m || !Wd || rows <= 0 || cols <= 0) return OR_INVALID;
    for (int64_t i = 0; i < rows * cols; ++i) Wd[i] = 0.0;
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t p = blk_ptr[r]; p < blk_ptr[r + 1]; ++p) {
            int64_t j = p - blk_ptr[r];
            int64_t c = j * m[r] + off[p];
            if (off[p] >= m[r] || c >= cols) return OR_INVALID;
            Wd[r * cols + c] = val[p];
        }
    return OR_OK;
}

/* y = W_darb X, X cols x batch (row k at X + k*ldx), Y rows x batch.
 * Block j of row r selects activation row j*m_r + off (Sec. 3.2, Fig. 6(b))
 * and multiplies it by the kept weight; the products are summed in double.
 * If absdot is given it receives sum |val * x| per output (the scale that the
 * tolerance of a finite-precision product is measured against).             */
int oracle_darb_spmm(const double *val, const uint8_t *off, const int64_t *blk_ptr,
                     const int32_t *m, int64_t rows, int64_t cols, const double *X,
                     int64_t ldx, int64_t batch, double *Y, int64_t ldy, double *absdot) {
    if (!val || !off || !blk_ptr || !m || !X || !Y || rows <= 0 || cols <= 0 || batch <= 0 ||
        ldx < batch || ldy < batch)
        return OR_INVALID;
    int bad = 0;
    _Pragma("omp parallel for schedule(static) reduction(|:bad)")
    for (int64_t r = 0; r < rows; ++r) {
        for (int64_t b = 0; b < batch; ++b) {
            double s = 0.0, a = 0.0;
            for (int64_t p = blk_ptr[r]; p < blk_ptr[r + 1]; ++p) {
                int64_t j = p - blk_ptr[r];
                int64_t k = j * m[r] + off[p];
                if (off[p] >= m[r] || k >= cols) { bad = 1; break; }
                s += val[p] * X[k * ldx + b];
                a += fabs(val[p] * X[k * ldx + b]);
            }
            Y[r * ldy + b] = s;
            if (absdot) absdot[r * ldy + b] = a;
        }
    }
    return bad ? OR_INVALID : OR_OK;
}

/* The same sum (Sec. 3.2, Fig. 6(b)) in single precision, for timing the
 * oracle as a CPU baseline only (never used as a reference value): kept values
 * widened to float, X float, one float accumulator per output, added in block
 * order; OpenMP over rows.                                                   */
int oracle_darb_spmm_f32_timed(const float *val, const uint8_t *off, const int64_t *blk_ptr,
                               const int32_t *m, int64_t rows, int64_t cols, const float *X,
                               int64_t ldx, int64_t batch, float *Y, int64_t ldy) {
    if (!val || !off || !blk_ptr || !m || !X || !Y || rows <= 0 || cols <= 0 || batch <= 0 ||
        ldx < batch || ldy < batch)
        return OR_INVALID;
    int bad = 0;
    _Pragma("omp parallel for schedule(static) reduction(|:bad)")
    for (int64_t r = 0; r < rows; ++r) {
        for (int64_t b = 0; b < batch; ++b) Y[r * ldy + b] = 0.0f;
        for (int64_t p = blk_ptr[r]; p < blk_ptr[r + 1]; ++p) {
            int64_t j = p - blk_ptr[r];
            int64_t k = j * m[r] + off[p];
            if (off[p] >= m[r] || k >= cols) { bad = 1; break; }
            for (int64_t b = 0; b < batch; ++b) Y[r * ldy + b] += val[p] * X[k * ldx + b];
        }
    }
    return bad ? OR_INVALID : OR_OK;
}

static double sigmoid(double v) { return 1.0 / (1.0 + exp(-v)); }

/* One LSTM step.  The gate matrix is 4H x (I+H), its input the stacked column
 * [x_t; h_{t-1}]; gate rows [0,H) = i, [H,2H) = f, [2H,3H) = g, [3H,4H) = o:
 *   c_t = sigmoid(f) * c_{t-1} + sigmoid(i) * tanh(g)
 *   h_t = sigmoid(o) * tanh(c_t)
 * x is I x B, h_prev / c_prev / h_out / c_out are H x B (batch contiguous);
 * bias (4H) may be NULL.  gate_abs (4H x B, optional) receives
 * sum |w * input| + |bias| of every gate pre-activation.                      */
int oracle_lstm_step(const double *val, const uint8_t *off, const int64_t *blk_ptr,
                     const int32_t *m, int64_t I, int64_t H, int64_t B, const double *x,
                     const double *h_prev, const double *c_prev, const double *bias,
                     double *h_out, double *c_out, double *gate_abs) {
    if (!x || !h_prev || !c_prev || !h_out || !c_out || I < 0 || H <= 0 || B <= 0)
        return OR_INVALID;
    int64_t rows = 4 * H, cols = I + H;
    double *u = malloc(sizeof(double) * cols * B);
    double *g = malloc(sizeof(double) * rows * B);
    double *ga = malloc(sizeof(double) * rows * B);
    if (!u || !g || !ga) { free(u); free(g); free(ga); return OR_INVALID; }
    for (int64_t k = 0; k < I; ++k)
        for (int64_t b = 0; b < B; ++b) u[k * B + b] = x[k * B + b];
    for (int64_t k = 0; k < H; ++k)
        for (int64_t b = 0; b < B; ++b) u[(I + k) * B + b] = h_prev[k * B + b];
    int st = oracle_darb_spmm(val, off, blk_ptr, m, rows, cols, u, B, B, g, B, ga);
    if (st == OR_OK) {
        for (int64_t r = 0; r < rows; ++r)
            for (int64_t b = 0; b < B; ++b) {
                double bb = bias ? bias[r] : 0.0;
                g[r * B + b] += bb;
                ga[r * B + b] += fabs(bb);
            }
        for (int64_t j = 0; j < H; ++j)
            for (int64_t b = 0; b < B; ++b) {
                double gi = g[(0 * H + j) * B + b], gf = g[(1 * H + j) * B + b];
                double gg = g[(2 * H + j) * B + b], go = g[(3 * H + j) * B + b];
                double c = sigmoid(gf) * c_prev[j * B + b] + sigmoid(gi) * tanh(gg);
                c_out[j * B + b] = c;
                h_out[j * B + b] = sigmoid(go) * tanh(c);
            }
        if (gate_abs) memcpy(gate_abs, ga, sizeof(double) * rows * B);
    }
    free(u); free(g); free(ga);
    return st;
}

/* One GRU step.  The gate matrix is 3H x (I+H); rows [0,H) = r, [H,2H) = z,
 * [2H,3H) = n.  Its columns [0,I) multiply x_t, columns [I,I+H) multiply
 * h_{t-1}, and the two parts are kept apart:
 *   a = W[:, :I] x + b_ih,   bh = W[:, I:] h + b_hh
 *   r = sigmoid(a_r + bh_r), z = sigmoid(a_z + bh_z)
 *   n = tanh(a_n + r * bh_n), h_t = (1 - z) * n + z * h_{t-1}
 * gate_abs (optional, 3H x B x 2): sum |w * input| + |bias| of a and of bh.   */
int oracle_gru_step(const double *val, const uint8_t *off, const int64_t *blk_ptr,
                    const int32_t *m, int64_t I, int64_t H, int64_t B, const double *x,
                    const double *h_prev, const double *b_ih, const double *b_hh,
                    double *h_out, double *gate_abs) {
    if (!val || !off || !blk_ptr || !m || !x || !h_prev || !h_out || I < 0 || H <= 0 || B <= 0)
        return OR_INVALID;
    int64_t rows = 3 * H, cols = I + H;
    double *a = calloc((size_t)(rows * B), sizeof(double));
    double *bh = calloc((size_t)(rows * B), sizeof(double));
    double *aa = calloc((size_t)(rows * B), sizeof(double));
    double *ba = calloc((size_t)(rows * B), sizeof(double));
    if (!a || !bh || !aa || !ba) { free(a); free(bh); free(aa); free(ba); return OR_INVALID; }
    int st = OR_OK;
    for (int64_t r = 0; r < rows && st == OR_OK; ++r)
        for (int64_t p = blk_ptr[r]; p < blk_ptr[r + 1]; ++p) {
            int64_t j = p - blk_ptr[r];
            int64_t k = j * m[r] + off[p];
            if (off[p] >= m[r] || k >= cols) { st = OR_INVALID; break; }
            for (int64_t b = 0; b < B; ++b) {
                if (k < I) {
                    a[r * B + b] += val[p] * x[k * B + b];
                    aa[r * B + b] += fabs(val[p] * x[k * B + b]);
                } else {
                    bh[r * B + b] += val[p] * h_prev[(k - I) * B + b];
                    ba[r * B + b] += fabs(val[p] * h_prev[(k - I) * B + b]);
                }
            }
        }
    if (st == OR_OK) {
        for (int64_t r = 0; r < rows; ++r)
            for (int64_t b = 0; b < B; ++b) {
                double bi = b_ih ? b_ih[r] : 0.0, bhh = b_hh ? b_hh[r] : 0.0;
                a[r * B + b] += bi;
                aa[r * B + b] += fabs(bi);
                bh[r * B + b] += bhh;
                ba[r * B + b] += fabs(bhh);
            }
        for (int64_t j = 0; j < H; ++j)
            for (int64_t b = 0; b < B; ++b) {
                double rr = sigmoid(a[(0 * H + j) * B + b] + bh[(0 * H + j) * B + b]);
                double zz = sigmoid(a[(1 * H + j) * B + b] + bh[(1 * H + j) * B + b]);
                double nn = tanh(a[(2 * H + j) * B + b] + rr * bh[(2 * H + j) * B + b]);
                h_out[j * B + b] = (1.0 - zz) * nn + zz * h_prev[j * B + b];
            }
        if (gate_abs)
            for (int64_t i = 0; i < rows * B; ++i) {
                gate_abs[2 * i] = aa[i];
                gate_abs[2 * i + 1] = ba[i];
            }
    }
    free(a); free(bh); free(aa); free(ba);
    return st;
}
