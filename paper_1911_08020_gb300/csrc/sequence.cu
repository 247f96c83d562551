// sequence.cu -- T steps of an LSTM or GRU cell on a DARB gate matrix in one
// persistent, cooperative launch (the RNNs of Sec. 4.1 run many steps per
// input; each step is the fused step of darb_lstm_step / darb_gru_step).
//
// Every CTA owns a contiguous range of hidden units and all gate rows of those
// units (LSTM rows u, H+u, 2H+u, 3H+u; GRU rows u, H+u, 2H+u), so the cell of
// a unit needs nothing from another CTA.  In the prologue a CTA decodes its
// rows once into shared memory as packed (value, absolute column) words -- a
// row's kept weights in column order -- and keeps them there for the whole
// sequence, so W_darb leaves HBM/L2 once instead of once per step.  Per step
// and per tile of batch columns it stages the stacked input [x_t; h_{t-1}] in
// shared memory and forms its gate sums: a warp per gate row, the 32 lanes
// split into 32/bt subgroups of bt batch columns, each subgroup taking every
// (32/bt)-th kept weight, then a shuffle reduction over the subgroups.  The
// cell is applied by the owning CTA, h_t goes to h_seq, c stays in a device
// buffer that only its owner touches.  Steps are separated by a grid-wide
// barrier (arrival counter in global memory, spun on with a 1 s limit; on
// expiry the kernel records a timeout, raises an abort flag that ends every
// other CTA's wait, and returns).  The launch is cooperative, so all CTAs are
// resident and the barrier cannot starve.  No CTA touches another CTA's shared
// memory, and no CTA leaves while a copy it issued may still be landing.
#include "darb_internal.h"
#include "launch.cuh"
#include "rnn_epilogue.cuh"
#include "tma.cuh"

#include <algorithm>
#include <cstdlib>
#include <vector>

namespace darb {
namespace seq {

constexpr int kThreads = 512;
constexpr int kSeqWarps = kThreads / 32;
constexpr int kMaxCtas = 256;
constexpr size_t kSmemCap = 226 * 1024;   // dynamic shared memory, below the 227 KB opt-in with room for the static part
constexpr int kMaxTile = 32;              // batch columns per tile, at most (one per lane)
constexpr size_t kCellOnChip = 16 * 1024; // LSTM cell state kept in shared memory up to this size

struct Ranges {
    int32_t start[kMaxCtas + 1];   // CTA q owns hidden units [start[q], start[q+1])
};

struct SeqArgs {
    int I, H, T;
    int lbt;                // log2 of the batch tile width bt (bt <= 32)
    int stage_mode;         // kStage*
    int piece;              // kept weights per work item, at most
    int c_on_chip;          // LSTM: cell state in shared memory
    // staged input rows: x_t at [0, I) (none when the x parts are precomputed),
    // h_{t-1} from row ipad, a zero row at ipad + hpad
    int ipad, hpad;
    // tensor-map staging (tma != 0): boxes of {bt columns, bxh rows} over x_t
    // (nbx of them) and {bt, bhh} over h_{t-1} (nbh), tile_bytes per tile in all
    int tma, nbx, bxh, nbh, bhh;
    uint32_t tile_bytes;
    int64_t B;
    const float *gx;        // x parts of the gate sums of every step, rows x ldgx (row r, step t, column b
                            // at r * ldgx + t * B + b), or nullptr: x_t is staged with h_{t-1} instead
    int64_t ldgx;
    const float *x;         // T x I x B
    const float *h0;        // H x B
    const float *c0;        // H x B (LSTM)
    const float *bias;      // LSTM [4H] or nullptr
    const float *b_ih;      // GRU [3H] or nullptr
    const float *b_hh;      // GRU [3H] or nullptr
    float *h_seq;           // T x H x B
    float *c_seq;           // T x H x B or nullptr (LSTM)
    float *c_state;         // H x B: the running cell state when it is not on chip (LSTM)
    float *c_last;          // H x B or nullptr (LSTM)
    // a copy of h_t with rows of ldp columns (B rounded up to the batch tile,
    // zeros past B) in two buffers by step parity, H x ldp each, or nullptr:
    // h_{t-1} is then staged from h_seq.  Boxes over it are whole 128-byte
    // aligned rows; boxes over B-column rows with a ragged tail are not
    float *h_pad;
    int64_t ldp;
    unsigned *bar;          // arrival counter, zero at launch
    int *abort_flag;        // zero at launch
    int32_t *status;
    unsigned long long barrier_ns;   // time limit of a grid-barrier wait (kWaitLimitNs unless a test shortens it)
    int skip_cta;           // test hook: this CTA does not arrive at the first barrier (-1: none)
};

// Byte offsets of the regions of a CTA's dynamic shared memory.
struct SmemPlan {
    uint32_t w_off, rowptr_off, mid_off, rowitem_off, item_off, bias_off, c_off, gx_off, in_off, part_off, total;
    int items_cap;
};

inline SmemPlan smem_plan(int64_t kept_cap, int rows_cap, int items_cap, int units_cap, bool bf16, bool gru,
                          int in_rows, int bt, int64_t B, bool c_on_chip, bool pre) {
    SmemPlan p{};
    p.items_cap = items_cap;
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o = (o + bytes + 15) / 16 * 16;
        return static_cast<uint32_t>(std::min<size_t>(at, UINT32_MAX));
    };
    p.w_off = take(size_t(kept_cap) * (bf16 ? 4 : 8));
    p.rowptr_off = take(size_t(rows_cap + 1) * 4);
    p.mid_off = take(size_t(rows_cap) * 4);
    p.rowitem_off = take(size_t(rows_cap + 1) * 4);
    p.item_off = take(size_t(items_cap) * 16);
    p.bias_off = take(size_t(rows_cap) * 2 * 4);
    p.c_off = take(c_on_chip ? size_t(units_cap) * size_t(B) * 4 : 0);
    p.gx_off = take(pre ? size_t(rows_cap) * bt * 4 : 0);
    p.in_off = take(size_t(in_rows) * bt * 4 + 128);   // rounded up to 128 bytes in the kernel
    p.part_off = take(size_t(gru ? 2 : 1) * items_cap * bt * 4);
    p.total = static_cast<uint32_t>(std::min<size_t>(o, UINT32_MAX));
    return p;
}

// Kept weight p of the CTA: its value and the index (row * bt) of the first
// element of the staged input row it multiplies.
template <bool BF16> struct Packed;
template <> struct Packed<true> {   // bf16 bits << 16 | index
    using T = uint32_t;
    static __device__ __forceinline__ T make(uint32_t bits, uint32_t col) { return (bits << 16) | col; }
    static __device__ __forceinline__ float val(T w) { return __uint_as_float(w & 0xFFFF0000u); }
    static __device__ __forceinline__ uint32_t col(T w) { return w & 0xFFFFu; }
};
template <> struct Packed<false> {  // fp32 bits, index
    using T = uint2;
    static __device__ __forceinline__ T make(uint32_t bits, uint32_t col) { return make_uint2(bits, col); }
    static __device__ __forceinline__ float val(T w) { return __uint_as_float(w.x); }
    static __device__ __forceinline__ uint32_t col(T w) { return w.y; }
};

// Grid-wide barrier with a time limit; false if this CTA gave up or another
// CTA did.  The CTA barrier orders every thread's h_t stores before thread 0's
// arrival, a release reduction on the counter (no return trip, no separate
// fence); thread 0 then polls with acquire loads.  An acquire that reads the
// final count synchronises with every arrival (each is a read-modify-write in
// the counter's release sequence), and the closing CTA barrier carries that
// to the CTA's other threads.
__device__ __forceinline__ bool grid_barrier(const SeqArgs &a, unsigned target, int *s_ok) {
    __syncthreads();
    if (threadIdx.x == 0) {
        if (!(int(blockIdx.x) == a.skip_cta && target == gridDim.x))
            asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(a.bar) : "memory");
        int ok = 1;
        const unsigned long long t0 = global_timer_ns();
        for (unsigned spin = 0;; ++spin) {
            unsigned v;
            asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(a.bar) : "memory");
            if (v >= target) break;
            if ((spin & 63) == 63) {
                if (*reinterpret_cast<volatile int *>(a.abort_flag)) {
                    ok = 0;
                    break;
                }
                if (global_timer_ns() - t0 > a.barrier_ns) {
                    ok = 0;
                    atomicExch(a.abort_flag, 1);
                    atomicOr(a.status, kStatusTimeout);
                    break;
                }
                __nanosleep(32);
            }
        }
        *s_ok = ok;
    }
    __syncthreads();
    return *s_ok != 0;
}

// On-chip layout of one row's kept weights: an x region, then an h region,
// each padded with zero weights (pointing at the zero row of the staged input)
// to a multiple of 4 so that a lane loads 4 weights at once.  Block jmid = I/m
// is the only block that can hold columns on both sides of I.
//   x parts precomputed: h region only, blocks jmid.. (an x weight of block
//     jmid becomes a zero weight);
//   GRU otherwise: blocks 0..jmid in the x region (block jmid there only if
//     its weight multiplies x), blocks jmid.. in the h region;
//   LSTM otherwise: one region of all blocks.
__host__ __device__ inline int round4(int v) { return (v + 3) & ~3; }
__host__ __device__ inline void row_regions(int n, int m, int I, bool pre, bool gru, int &xr, int &hr) {
    const int jmid = I / m;
    if (pre) {
        xr = 0;
        hr = round4(n - jmid);
    } else if (gru) {
        xr = round4(jmid + 1);
        hr = round4(n - jmid);
    } else {
        xr = round4(n);
        hr = 0;
    }
}

// Sum over kept weights [pa, pb) of the CTA (multiples of 4), subgroup `sub`
// taking every S-th group of 4 weights from pa + 4 sub, against one batch
// column of the staged input: s_inc = s_in + that column, and a weight's
// column field is the index of its staged row's first element, row * bt.
template <class P>
__device__ __forceinline__ float dot_range(const typename P::T *s_w, const float *s_inc, int pa, int pb, int sub,
                                           int S) {
    float acc0 = 0.0f, acc1 = 0.0f;
#pragma unroll 2
    for (int p = pa + 4 * sub; p < pb; p += 4 * S) {
        typename P::T w[4];
        if constexpr (sizeof(typename P::T) == 4) {
            const uint4 q = *reinterpret_cast<const uint4 *>(s_w + p);
            w[0] = q.x; w[1] = q.y; w[2] = q.z; w[3] = q.w;
        } else {
            const uint4 q0 = *reinterpret_cast<const uint4 *>(s_w + p);
            const uint4 q1 = *reinterpret_cast<const uint4 *>(s_w + p + 2);
            w[0] = make_uint2(q0.x, q0.y); w[1] = make_uint2(q0.z, q0.w);
            w[2] = make_uint2(q1.x, q1.y); w[3] = make_uint2(q1.z, q1.w);
        }
        const float v0 = s_inc[P::col(w[0])], v1 = s_inc[P::col(w[1])];
        const float v2 = s_inc[P::col(w[2])], v3 = s_inc[P::col(w[3])];
        acc0 = fmaf(P::val(w[0]), v0, acc0);
        acc1 = fmaf(P::val(w[1]), v1, acc1);
        acc0 = fmaf(P::val(w[2]), v2, acc0);
        acc1 = fmaf(P::val(w[3]), v3, acc1);
    }
    return acc0 + acc1;
}

// Input staging modes, chosen on the host from the shapes and alignments.
constexpr int kStageScalar = 0;   // one float per load
constexpr int kStageQuadCols = 1; // 4 batch columns per 16-byte load (B and bt multiples of 4, aligned)
constexpr int kStageQuadRows = 2; // B == 1: 4 input rows per 16-byte load (I, H multiples of 4, aligned)
constexpr int kStageUnroll = 8;   // loads a thread has in flight

// s_in[k][j] = [x_t; h_{t-1}][k][b0 + j] for j < nb, 0 for nb <= j < bt, for
// the K staged rows, of which the first I come from x_t (I = 0: h only).
// h_{t-1} was written by other CTAs of this launch, so every load goes to L2
// (ld.cg); the loads of a thread are issued together so that enough bytes are
// in flight to cover the L2 latency, and each CTA starts its sweep at its own
// offset so that the CTAs do not all ask for the same lines at once.
__device__ __forceinline__ void stage_input(const SeqArgs &a, int I, int K, const float *xt, const float *hp,
                                            int64_t b0, int nb, float *s_in) {
    const int lbt = a.lbt, bt = 1 << lbt;
    const int64_t B = a.B;
    const int tid = threadIdx.x;
    auto src = [&](int k) { return k < I ? xt + int64_t(k) * B : hp + int64_t(k - I) * B; };
    if (a.stage_mode == kStageQuadCols) {
        const int lq = lbt - 2, n = K << lq;   // quads
        const int rot = static_cast<int>(int64_t(blockIdx.x) * n / gridDim.x);
        for (int i0 = tid; i0 < n; i0 += kThreads * kStageUnroll) {
            float4 v[kStageUnroll];
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u) {
                int i = i0 + u * kThreads;
                v[u] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
                if (i < n) {
                    i = i + rot < n ? i + rot : i + rot - n;
                    const int k = i >> lq, j = (i & ((1 << lq) - 1)) * 4;
                    if (j < nb) v[u] = __ldcg(reinterpret_cast<const float4 *>(src(k) + b0 + j));
                }
            }
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u) {
                const int i = i0 + u * kThreads;
                if (i < n) reinterpret_cast<float4 *>(s_in)[i + rot < n ? i + rot : i + rot - n] = v[u];
            }
        }
    } else if (a.stage_mode == kStageQuadRows) {
        const int n = K >> 2;
        const int rot = static_cast<int>(int64_t(blockIdx.x) * n / gridDim.x);
        for (int i0 = tid; i0 < n; i0 += kThreads * kStageUnroll) {
            float4 v[kStageUnroll];
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u) {
                int i = i0 + u * kThreads;
                if (i < n) {
                    i = i + rot < n ? i + rot : i + rot - n;
                    v[u] = __ldcg(reinterpret_cast<const float4 *>(src(4 * i)));
                }
            }
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u) {
                const int i = i0 + u * kThreads;
                if (i < n) reinterpret_cast<float4 *>(s_in)[i + rot < n ? i + rot : i + rot - n] = v[u];
            }
        }
    } else {
        const int n = K << lbt;
        for (int i0 = tid; i0 < n; i0 += kThreads * kStageUnroll) {
            float v[kStageUnroll];
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u) {
                const int i = i0 + u * kThreads;
                const int k = i >> lbt, j = i & (bt - 1);
                v[u] = 0.0f;
                if (i < n && j < nb) v[u] = __ldcg(src(k) + b0 + j);
            }
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u)
                if (i0 + u * kThreads < n) s_in[i0 + u * kThreads] = v[u];
        }
    }
}

template <bool BF16, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
seq_kernel(Format f, SeqArgs a, Ranges rg, SmemPlan sp, const __grid_constant__ CUtensorMap mx,
           const __grid_constant__ CUtensorMap mh0, const __grid_constant__ CUtensorMap mhs) {
    constexpr int kGates = MODE == kModeLstm ? 4 : 3;
    constexpr bool kGru = MODE == kModeGru;
    using P = Packed<BF16>;
    using PT = typename P::T;
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ int s_ok, s_nitems, s_staged, s_next;
    __shared__ __align__(8) uint64_t s_full;   // the staged tile has landed
    PT *s_w = reinterpret_cast<PT *>(sm + sp.w_off);
    int *s_rowptr = reinterpret_cast<int *>(sm + sp.rowptr_off);
    int *s_mid = reinterpret_cast<int *>(sm + sp.mid_off);          // GRU: first kept weight of a row on h
    int *s_rowitem = reinterpret_cast<int *>(sm + sp.rowitem_off);  // items of local row lr: [s_rowitem[lr], s_rowitem[lr+1])
    int4 *s_item = reinterpret_cast<int4 *>(sm + sp.item_off);      // (first, end, local row, first on h)
    float *s_bias = reinterpret_cast<float *>(sm + sp.bias_off);    // [R] (GRU: [2R], b_ih then b_hh)
    float *s_c = reinterpret_cast<float *>(sm + sp.c_off);          // [units][B] when on chip
    float *s_gx = reinterpret_cast<float *>(sm + sp.gx_off);        // [R][bt]: x parts of this tile
    float *s_in = reinterpret_cast<float *>(                          // [kin + 1][bt], row kin zero
        (reinterpret_cast<uintptr_t>(sm + sp.in_off) + 127) & ~uintptr_t(127));
    float *s_part = reinterpret_cast<float *>(sm + sp.part_off);    // [parts][items][bt]
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int u0 = rg.start[blockIdx.x], nu = rg.start[blockIdx.x + 1] - u0;
    const int R = kGates * nu;   // local row q*nu + i is matrix row q*H + u0 + i
    const int I = a.I, H = a.H;
    const int lbt = a.lbt, bt = 1 << lbt, S = 32 >> lbt;
    const int sub = lane >> lbt, col = lane & (bt - 1);
    const int64_t B = a.B;
    // with the x parts precomputed only h_{t-1} is staged and only the kept
    // weights of blocks that reach column I are kept on chip (columns shifted by I)
    const bool pre = a.gx != nullptr;
    // GRU without precomputed x parts keeps the x and h sums of each item apart
    const bool split = kGru && !pre;
    const int kin = a.ipad + a.hpad;
    auto grow = [&](int lr) { return (lr / nu) * H + u0 + lr % nu; };

    // ---- prologue: row sizes, biases, cell state, the zero row of the staged input
    for (int lr = tid; lr < R; lr += kThreads) {
        const int r = grow(lr);
        const Group &g = f.groups[f.rowloc[r] / kSlots];
        int xr, hr;
        row_regions(g.n, g.m, I, pre, kGru, xr, hr);
        s_rowptr[lr + 1] = xr + hr;
        s_mid[lr] = xr;   // relative until the row pointers exist
        if constexpr (kGru) {
            s_bias[lr] = a.b_ih ? a.b_ih[r] : 0.0f;
            s_bias[R + lr] = a.b_hh ? a.b_hh[r] : 0.0f;
        } else {
            s_bias[lr] = a.bias ? a.bias[r] : 0.0f;
        }
    }
    if constexpr (!kGru)
        if (a.c_on_chip)
            for (int i = tid; i < nu * B; i += kThreads) s_c[i] = a.c0[int64_t(u0) * B + i];
    for (int j = tid; j < bt; j += kThreads) s_in[(kin << lbt) + j] = 0.0f;
    if (tid == 0) {
        mbar_init(&s_full, 1);
        fence_mbar_init();
    }
    __syncthreads();
    // row pointers and work items: every row cut into pieces of at most a.piece weights
    if (tid == 0) {
        int p = 0, ni = 0;
        for (int lr = 0; lr < R; ++lr) {
            const int n = s_rowptr[lr + 1];
            s_rowptr[lr] = p;
            s_mid[lr] += p;
            s_rowitem[lr] = ni;
            for (int q = 0; q < n; q += a.piece) s_item[ni++] = make_int4(p + q, p + min(n, q + a.piece), lr, 0);
            p += n;
        }
        s_rowptr[R] = p;
        s_rowitem[R] = ni;
        s_nitems = ni;
    }
    __syncthreads();
    // zero weights everywhere, then every kept weight as (value, staged row)
    for (int p = tid; p < s_rowptr[R]; p += kThreads) s_w[p] = P::make(0u, uint32_t(kin) << lbt);
    __syncthreads();
    for (int lr = warp; lr < R; lr += kSeqWarps) {
        const int loc = f.rowloc[grow(lr)];
        const Group g = f.groups[loc / kSlots];
        const int slot = loc % kSlots;
        const int base = s_rowptr[lr], mid = s_mid[lr];
        const int jmid = I / g.m;
        for (int j = (pre ? jmid : 0) + lane; j < g.n; j += 32) {
            const int64_t rec = int64_t(j / kChunk) * kSlots + slot;
            const int q = j % kChunk;
            uint32_t bits;
            if constexpr (BF16) bits = static_cast<const uint16_t *>(f.vals)[g.val_off + rec * kChunk + q];
            else bits = static_cast<const uint32_t *>(f.vals)[g.val_off + rec * kChunk + q];
            uint32_t o;
            if (g.nib) o = (f.offs[g.off_off + rec] >> (4 * q)) & 15u;
            else o = (f.offs[g.off_off + 2 * rec + (q >> 2)] >> (8 * (q & 3))) & 255u;
            uint32_t c = uint32_t(j) * uint32_t(g.m) + o;
            const bool on_h = c >= uint32_t(I);
            int at;
            if (pre || kGru) at = on_h ? mid + j - jmid : base + j;   // h region from block jmid on
            else at = base + j;
            if (on_h) {
                c = c - uint32_t(I) + uint32_t(a.ipad);   // staged row of h
            } else if (pre) {   // an x weight of block jmid: its product is in gx
                bits = 0;
                c = uint32_t(kin);
                at = mid;
            }
            s_w[at] = P::make(bits, c << lbt);   // (kin + 1) * bt floats fit in shared memory: < 2^16
        }
    }
    __syncthreads();
    const int NI = s_nitems;
    if (tid == 0) s_next = 0;
    for (int i = tid; i < NI; i += kThreads) {
        int4 it = s_item[i];
        it.w = split ? max(it.x, min(it.y, s_mid[it.z])) : it.y;
        s_item[i] = it;
    }
    __syncthreads();

    // ---- the steps
    int tile = 0;   // tiles staged so far: the parity of s_full
    float *c_run = kGru ? nullptr : (a.c_on_chip ? s_c : a.c_state + int64_t(u0) * B);
    for (int t = 0; t < a.T; ++t) {
        const float *xt = a.x + int64_t(t) * I * B;
        const float *hp = t == 0 ? a.h0 : a.h_seq + int64_t(t - 1) * H * B;
        float *ht = a.h_seq + int64_t(t) * H * B + int64_t(u0) * B;
        float *ct = a.c_seq ? a.c_seq + int64_t(t) * H * B + int64_t(u0) * B : nullptr;
        const float *cp = kGru ? nullptr : (t == 0 && !a.c_on_chip ? a.c0 + int64_t(u0) * B : c_run);
        for (int64_t b0 = 0; b0 < B; b0 += bt) {
            const int nb = static_cast<int>(B - b0 < bt ? B - b0 : bt);
            // stage [x_t; h_{t-1}] (or h_{t-1}) for columns [b0, b0 + nb), zeros past the batch
            if (a.tma && tid == 0) {
                // every thread of this CTA is done with the previous tile (the
                // barrier that ended it); order those reads before the copies
                fence_proxy_async_smem();
                fence_proxy_async_global();   // h_{t-1} was published by generic stores
                mbar_arrive_expect_tx(&s_full, a.tile_bytes);
                for (int bx = 0; bx < a.nbx + a.nbh; ++bx) {
                    const bool isx = bx < a.nbx;
                    const int y = isx ? bx * a.bxh : (bx - a.nbx) * a.bhh;
                    float *dst = s_in + (int64_t(isx ? y : a.ipad + y) << lbt);
                    const CUtensorMap *m = isx ? &mx : (t == 0 ? &mh0 : &mhs);
                    const int z = isx ? t : (t == 0 ? 0 : (a.h_pad ? (t - 1) & 1 : t - 1));
                    tensor3d_g2s(dst, m, static_cast<int>(b0), y, z, &s_full);
                }
                bool ok = mbar_wait(&s_full, tile & 1, false);
                if (!ok) {
                    atomicOr(a.status, kStatusTimeout);
                    atomicExch(a.abort_flag, 1);
                    // the copies may still land: give them a second bounded wait
                    // before this CTA leaves
                    mbar_wait(&s_full, tile & 1, false);
                }
                s_staged = ok;
            }
            if (pre)
                for (int i = tid; i < R << lbt; i += kThreads) {
                    const int lr = i >> lbt, j = i & (bt - 1);
                    s_gx[i] = j < nb ? __ldg(a.gx + int64_t(grow(lr)) * a.ldgx + int64_t(t) * B + b0 + j) : 0.0f;
                }
            if (!a.tma) stage_input(a, pre ? 0 : I, kin, xt, hp, b0, nb, s_in);
            __syncthreads();
            if (a.tma) {
                if (!s_staged) return;
                mbar_wait(&s_full, tile & 1, false);   // completed: makes the copied data visible to this thread
            }
            // partial gate sums of the work items, handed out to warps as they come free
            while (true) {
                int ii = 0;
                if (lane == 0) ii = atomicAdd(&s_next, 1);
                ii = __shfl_sync(0xFFFFFFFFu, ii, 0);
                if (ii >= NI) break;
                const int4 it = s_item[ii];
                float a0 = dot_range<P>(s_w, s_in + col, it.x, it.w, sub, S);
                float a1 = 0.0f;
                if (split) a1 = dot_range<P>(s_w, s_in + col, it.w, it.y, sub, S);
                for (int o = 16; o >= bt; o >>= 1) {
                    a0 += __shfl_xor_sync(0xFFFFFFFFu, a0, o);
                    if (split) a1 += __shfl_xor_sync(0xFFFFFFFFu, a1, o);
                }
                if (sub == 0) {
                    s_part[(ii << lbt) + col] = a0;
                    if (split) s_part[((NI + ii) << lbt) + col] = a1;
                }
            }
            __syncthreads();
            if (tid == 0) s_next = 0;   // for the next tile; every warp has left the loop
            // the cells of the owned units for these columns
            // partial sums of local row lr: part 0 (everything, or the x part of a
            // split GRU row), part 1 (the h part of a split GRU row)
            auto sum = [&](int lr, int part, int j) {
                float v = 0.0f;
                for (int ii = s_rowitem[lr]; ii < s_rowitem[lr + 1]; ++ii) v += s_part[((part * NI + ii) << lbt) + j];
                return v;
            };
            for (int i = tid; i < nu << lbt; i += kThreads) {
                const int ui = i >> lbt, j = i & (bt - 1);
                float *hq = a.h_pad ? a.h_pad + (int64_t(t & 1) * H + u0 + ui) * a.ldp + b0 + j : nullptr;
                if (j >= nb) {
                    if (hq) *hq = 0.0f;
                    continue;
                }
                const int64_t e = int64_t(ui) * B + b0 + j;
                auto xg = [&](int lr) { return pre ? s_gx[(lr << lbt) + j] : 0.0f; };
                if constexpr (MODE == kModeLstm) {
                    auto gate = [&](int lr) { return s_bias[lr] + sum(lr, 0, j) + xg(lr); };
                    const float pi = gate(ui), pf = gate(nu + ui), pg = gate(2 * nu + ui), po = gate(3 * nu + ui);
                    const float c = sigm(pf) * cp[e] + sigm(pi) * tanhf(pg);
                    c_run[e] = c;
                    if (ct) ct[e] = c;
                    const float hv = sigm(po) * tanhf(c);
                    ht[e] = hv;
                    if (hq) *hq = hv;
                } else {
                    // x part (b_ih + W_x x) and h part (b_hh + W_h h) of each gate
                    auto gx_ = [&](int lr) { return s_bias[lr] + (pre ? xg(lr) : sum(lr, 0, j)); };
                    auto gh_ = [&](int lr) { return s_bias[R + lr] + sum(lr, split ? 1 : 0, j); };
                    const float rr = sigm(gx_(ui) + gh_(ui));
                    const float zz = sigm(gx_(nu + ui) + gh_(nu + ui));
                    const float nn = tanhf(gx_(2 * nu + ui) + rr * gh_(2 * nu + ui));
                    const float hv = (1.0f - zz) * nn + zz * s_in[((a.ipad + u0 + ui) << lbt) + j];
                    ht[e] = hv;
                    if (hq) *hq = hv;
                }
            }
            __syncthreads();
            ++tile;
        }
        if (t + 1 < a.T && !grid_barrier(a, unsigned(t + 1) * gridDim.x, &s_ok)) return;
    }
    if constexpr (!kGru)
        if (a.c_on_chip && a.c_last)
            for (int i = tid; i < nu * B; i += kThreads) a.c_last[int64_t(u0) * B + i] = s_c[i];
}

}  // namespace seq

namespace {

// Test hook for the failure path of the grid barrier.  With the environment
// variable DARB_TEST_BARRIER_TIMEOUT=1 a launch's barrier waits give up after
// 1 ms and CTA 0 withholds its arrival at the first barrier: every CTA's wait
// runs out, the launch records DARB_ERR_TIMEOUT (read by darb_sync_status),
// raises the abort flag and ends.  Only the barrier is affected -- no copy is
// in flight while a CTA waits there -- and the results of that call are not
// valid.  Read on every launch so that a test can set and clear it.
void sequence_test_hook(unsigned long long *barrier_ns, int *skip_cta) {
    const char *v = std::getenv("DARB_TEST_BARRIER_TIMEOUT");
    if (v != nullptr && v[0] == '1' && v[1] == '\0') {
        *barrier_ns = 1000000ull;
        *skip_cta = 0;
    }
}

// Contiguous unit ranges over G CTAs with about equal kept weights each.
// Returns the largest weight count and unit count of any CTA.
void split_units(const std::vector<int64_t> &kept, int G, seq::Ranges &rg, int64_t &kept_cap, int &units_cap) {
    const int H = static_cast<int>(kept.size());
    int64_t total = 0;
    for (int64_t k : kept) total += k;
    kept_cap = 0;
    units_cap = 0;
    int u = 0;
    int64_t acc = 0;   // weights of units [0, u)
    for (int q = 0; q < G; ++q) {
        rg.start[q] = u;
        const int64_t target = q + 1 == G ? total : total * (q + 1) / G;
        const int last = H - (G - 1 - q);   // leave one unit for every later CTA
        int64_t mine = 0;
        while (u < last && (acc + mine < target || mine == 0)) mine += kept[static_cast<size_t>(u++)];
        acc += mine;
        kept_cap = std::max(kept_cap, mine);
        units_cap = std::max(units_cap, u - rg.start[q]);
    }
    rg.start[G] = H;
}

}  // namespace

// x_t of every step laid out as the columns of one product input:
// xall[k][t * B + b] = x[t][k][b] for k < I (a warp per (t, k), lanes over b).
__global__ void __launch_bounds__(256) gather_x_kernel(const float *x, int T, int I, int64_t B, float *xall,
                                                       int64_t ldx) {
    const int lane = threadIdx.x & 31;
    const int64_t nrows = int64_t(T) * I;
    for (int64_t row = int64_t(blockIdx.x) * 8 + (threadIdx.x >> 5); row < nrows; row += int64_t(gridDim.x) * 8) {
        const int64_t t = row / I, k = row % I;
        const float *src = x + row * B;
        float *dst = xall + k * ldx + t * B;
        for (int64_t b = lane; b < B; b += 32) dst[b] = __ldg(src + b);
    }
}

// Whether the x parts of all steps go through one darb_spmm-style product up
// front: when x_t is a large share of the stacked input the per-step staging
// and gate sums shrink by that share; the product has T*B columns.
inline bool precompute_x(int64_t T, int64_t I, int64_t H, int64_t B, size_t ws_bytes) {
    return I > 0 && 2 * I >= H && T * B >= 64 && T * B <= (int64_t(1) << 19) && ws_bytes <= (size_t(1) << 30);
}

template <bool BF16, int MODE>
static cudaError_t launch_seq_t(const Format &f, const int32_t *row_m, seq::SeqArgs a, float *c_last,
                                cudaStream_t stream) {
    using namespace seq;
    constexpr int kGates = MODE == kModeLstm ? 4 : 3;
    constexpr bool kGru = MODE == kModeGru;
    const int H = a.H, I = a.I;
    const int64_t B = a.B, T = a.T, rows = f.rows;
    if (f.cols > 65535) return cudaErrorNotSupported;   // columns are kept in 16 bits
    auto up = [](size_t v) { return (v + 255) / 256 * 256; };
    const int64_t ldx = (T * B + 3) / 4 * 4;   // 16-byte rows for the product's loads
    const size_t pre_bytes = up(size_t(I + H) * ldx * 4) + up(size_t(rows) * ldx * 4);
    const bool pre = precompute_x(T, I, H, B, pre_bytes);
    // kept weights on chip per row: all, or those of the blocks that reach column I
    auto row_kept = [&](int64_t r) {
        const int m = row_m[r];
        int xr, hr;
        row_regions(static_cast<int>((f.cols + m - 1) / m), m, I, pre, kGru, xr, hr);
        return int64_t(xr + hr);
    };
    std::vector<int64_t> kept(static_cast<size_t>(H));
    for (int u = 0; u < H; ++u) {
        int64_t k = 0;
        for (int q = 0; q < kGates; ++q) k += row_kept(int64_t(q) * H + u);
        kept[static_cast<size_t>(u)] = k;
    }
    auto aligned = [](const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
    const int xrows = pre ? 0 : I;   // staged rows that come from x_t
    const bool ptrs = (xrows == 0 || aligned(a.x)) && aligned(a.h0) && aligned(a.h_seq);
    // tensor-map staging needs 16-byte rows of every source (B a multiple of 4)
    const bool tma_ok = ptrs && B % 4 == 0 && tensor_map_encoder() != nullptr;
    const int G = std::max(1, std::min({sm_count(), H, kMaxCtas}));
    Ranges rg{};
    int64_t kept_cap = 0;
    int units_cap = 0;
    split_units(kept, G, rg, kept_cap, units_cap);
    if (kept_cap > (int64_t(1) << 20)) return cudaErrorNotSupported;
    const bool c_on_chip = !kGru && size_t(units_cap) * size_t(B) * 4 <= kCellOnChip;
    // staged rows per box: at most 256, and a multiple of 32 / bt so that every
    // box lands on a 128-byte boundary; as few padding rows as possible
    auto box_rows = [](int n, int align, int &nbox, int &rows) {
        nbox = (n + 255) / 256;
        rows = nbox ? ((n + nbox - 1) / nbox + align - 1) / align * align : 0;
        if (rows > 256) rows = 256 / align * align, nbox = (n + rows - 1) / rows;
    };
    int nbx = 0, bxh = 0, nbh = 0, bhh = 0;
    // widest batch tile (a power of two, <= 32) whose staging still fits, with
    // rows cut into work items of about kept_cap / (ipw * warps) weights (a
    // multiple of 4, at least 2 loads of 4 weights per subgroup): ipw = 4 items
    // per warp balances the warps best, fewer save the items' partial sums
    int bt = 1;
    while (bt < kMaxTile && bt < B) bt *= 2;
    SmemPlan sp{};
    int piece = 0;
    for (bool fits = false; !fits; bt /= 2) {
        if (bt == 0) return cudaErrorNotSupported;
        const int S = kMaxTile / bt;
        const bool tma = tma_ok && bt >= 4;
        if (tma) {
            box_rows(xrows, 32 / bt, nbx, bxh);
            box_rows(H, 32 / bt, nbh, bhh);
        }
        const int in_rows = tma ? nbx * bxh + nbh * bhh + 1 : xrows + H + 1;
        for (int ipw = 4; ipw >= 1 && !fits; ipw /= 2) {
            piece = round4(static_cast<int>(
                std::max<int64_t>(8 * S, (kept_cap + ipw * kSeqWarps - 1) / (ipw * kSeqWarps))));
            int items_cap = 0;
            for (int q = 0; q < G; ++q) {
                int items = 0;
                for (int g = 0; g < kGates; ++g)
                    for (int u = rg.start[q]; u < rg.start[q + 1]; ++u)
                        items += static_cast<int>((row_kept(int64_t(g) * H + u) + piece - 1) / piece);
                items_cap = std::max(items_cap, items);
            }
            sp = smem_plan(kept_cap, kGates * units_cap, items_cap, units_cap, BF16, kGru && !pre, in_rows, bt, B,
                           c_on_chip, pre);
            fits = sp.total <= kSmemCap;
        }
        if (fits) break;
    }
    a.piece = piece;
    a.c_on_chip = c_on_chip ? 1 : 0;
    a.c_last = c_last;
    a.lbt = 0;
    while ((1 << a.lbt) < bt) ++a.lbt;
    a.tma = tma_ok && bt >= 4 ? 1 : 0;
    if (a.tma) {
        a.nbx = nbx;
        a.bxh = bxh;
        a.nbh = nbh;
        a.bhh = bhh;
        a.ipad = nbx * bxh;
        a.hpad = nbh * bhh;
        a.tile_bytes = static_cast<uint32_t>((a.ipad + a.hpad) * bt * 4);
    } else {
        a.ipad = xrows;
        a.hpad = H;
    }
    a.stage_mode = kStageScalar;
    if (ptrs && B % 4 == 0 && bt % 4 == 0) a.stage_mode = kStageQuadCols;
    else if (ptrs && B == 1 && xrows % 4 == 0 && H % 4 == 0) a.stage_mode = kStageQuadRows;
    const cudaError_t attr = allow_smem(seq_kernel<BF16, MODE>, kSmemCap);
    if (attr != cudaSuccess) return attr;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeCooperative;
    at[0].val.cooperative = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(G));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = sp.total;
    cfg.stream = stream;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    // every wait is bounded by kWaitLimitNs; a test may shorten the barrier's
    // limit and hold back one CTA's first arrival (sequence_test_hook)
    a.barrier_ns = kWaitLimitNs;
    a.skip_cta = -1;
    sequence_test_hook(&a.barrier_ns, &a.skip_cta);
    // workspace: barrier word and abort flag; the cell state when it is neither
    // on chip nor in c_last; the x parts and the product input they come from;
    // the padded copy of h_t
    const size_t cbytes = kGru || c_on_chip || c_last ? 0 : up(size_t(H) * size_t(B) * 4);
    const int64_t ldp = (B + bt - 1) / bt * bt;
    const size_t pbytes = a.tma && ldp != B && T > 1 ? up(2 * size_t(H) * size_t(ldp) * 4) : 0;
    const size_t ws_bytes = 256 + cbytes + (pre ? pre_bytes : 0) + pbytes;
    char *ws = nullptr;
    cudaError_t e = stream_alloc(reinterpret_cast<void **>(&ws), ws_bytes, stream);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(ws, 0, 16, stream);
    a.bar = reinterpret_cast<unsigned *>(ws);
    a.abort_flag = reinterpret_cast<int *>(ws + 4);
    a.c_state = kGru || c_on_chip ? nullptr : (c_last ? c_last : reinterpret_cast<float *>(ws + 256));
    a.h_pad = pbytes ? reinterpret_cast<float *>(ws + ws_bytes - pbytes) : nullptr;
    a.ldp = ldp;
    if (pre && e == cudaSuccess) {
        float *xall = reinterpret_cast<float *>(ws + 256 + cbytes);
        float *gx = reinterpret_cast<float *>(ws + 256 + cbytes + up(size_t(I + H) * ldx * 4));
        e = cudaMemsetAsync(xall + size_t(I) * ldx, 0, size_t(H) * ldx * 4, stream);
        if (e == cudaSuccess) {
            const int64_t warps = T * I;
            const unsigned grid = static_cast<unsigned>(std::min<int64_t>((warps + 7) / 8, int64_t(sm_count()) * 16));
            gather_x_kernel<<<grid, 256, 0, stream>>>(a.x, a.T, I, B, xall, ldx);
            e = cudaGetLastError();
        }
        // only the x columns: xall's h rows are zero
        if (e == cudaSuccess) e = launch_spmm_prefix(f, I, xall, ldx, T * B, gx, ldx, false, stream);
        a.gx = gx;
        a.ldgx = ldx;
    }
    // tensor maps of the staged sources: 3-D (batch, rows, step) so that a box
    // running past the last row of a step reads zeros, never the next step;
    // h_{t-1} from the padded copy when the last batch tile is ragged
    CUtensorMap mx{}, mh0{}, mhs{};
    if (a.tma && e == cudaSuccess) {
        auto make = [&](CUtensorMap *m, const float *base, int64_t cols, int64_t rows, int64_t depth, int boxh) {
            const cuuint64_t dims[3] = {cuuint64_t(cols), cuuint64_t(rows), cuuint64_t(depth)};
            const cuuint64_t strides[2] = {cuuint64_t(cols) * 4, cuuint64_t(cols) * 4 * cuuint64_t(rows)};
            const cuuint32_t box[3] = {cuuint32_t(bt), cuuint32_t(boxh), 1};
            const cuuint32_t es[3] = {1, 1, 1};
            return tensor_map_encoder()(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float *>(base), dims,
                                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
        };
        bool ok = make(&mh0, a.h0, B, H, 1, bhh) &&
                  (a.h_pad ? make(&mhs, a.h_pad, a.ldp, H, 2, bhh) : make(&mhs, a.h_seq, B, H, T, bhh));
        if (ok && nbx) ok = make(&mx, a.x, B, I, T, bxh);
        if (!ok) {   // plain loads instead (the plan above has room for either)
            a.tma = 0;
            a.ipad = xrows;
            a.hpad = H;
            a.h_pad = nullptr;
        }
    }
    if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, seq_kernel<BF16, MODE>, f, a, rg, sp, mx, mh0, mhs);
    const cudaError_t ef = cudaFreeAsync(ws, stream);
    return e != cudaSuccess ? e : ef;
}

cudaError_t launch_lstm_sequence(const Format &f, const int32_t *row_m, int64_t T, int64_t I, int64_t H, int64_t B,
                                 const float *x, const float *h0, const float *c0, const float *bias, float *h_seq,
                                 float *c_seq, float *c_last, cudaStream_t stream) {
    seq::SeqArgs a{};
    a.I = static_cast<int>(I);
    a.H = static_cast<int>(H);
    a.T = static_cast<int>(T);
    a.B = B;
    a.x = x;
    a.h0 = h0;
    a.c0 = c0;
    a.bias = bias;
    a.h_seq = h_seq;
    a.c_seq = c_seq;
    a.status = f.status;
    return f.bf16 ? launch_seq_t<true, kModeLstm>(f, row_m, a, c_last, stream)
                  : launch_seq_t<false, kModeLstm>(f, row_m, a, c_last, stream);
}

cudaError_t launch_gru_sequence(const Format &f, const int32_t *row_m, int64_t T, int64_t I, int64_t H, int64_t B,
                                const float *x, const float *h0, const float *b_ih, const float *b_hh, float *h_seq,
                                cudaStream_t stream) {
    seq::SeqArgs a{};
    a.I = static_cast<int>(I);
    a.H = static_cast<int>(H);
    a.T = static_cast<int>(T);
    a.B = B;
    a.x = x;
    a.h0 = h0;
    a.b_ih = b_ih;
    a.b_hh = b_hh;
    a.h_seq = h_seq;
    a.status = f.status;
    return f.bf16 ? launch_seq_t<true, kModeGru>(f, row_m, a, nullptr, stream)
                  : launch_seq_t<false, kModeGru>(f, row_m, a, nullptr, stream);
}

}  // namespace darb
