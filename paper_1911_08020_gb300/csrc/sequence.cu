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
// resident and the barrier cannot starve.
#include "darb_internal.h"
#include "launch.cuh"
#include "rnn_epilogue.cuh"
#include "tma.cuh"

#include <algorithm>
#include <vector>

namespace darb {
namespace seq {

constexpr int kThreads = 256;
constexpr int kSeqWarps = kThreads / 32;
constexpr int kMaxCtas = 256;
constexpr size_t kSmemCap = 226 * 1024;   // dynamic shared memory, below the 227 KB opt-in with room for the static part
constexpr int kMaxTile = 32;   // batch columns per tile, at most (one per lane)

struct Ranges {
    int32_t start[kMaxCtas + 1];   // CTA q owns hidden units [start[q], start[q+1])
};

struct SeqArgs {
    int I, H, T;
    int lbt;                // log2 of the batch tile width bt (bt <= 32)
    int stage_mode;         // kStage*
    int64_t B;
    const float *x;         // T x I x B
    const float *h0;        // H x B
    const float *c0;        // H x B (LSTM)
    const float *bias;      // LSTM [4H] or nullptr
    const float *b_ih;      // GRU [3H] or nullptr
    const float *b_hh;      // GRU [3H] or nullptr
    float *h_seq;           // T x H x B
    float *c_seq;           // T x H x B or nullptr (LSTM)
    float *c_state;         // H x B: the running cell state (LSTM)
    unsigned *bar;          // arrival counter, zero at launch
    int *abort_flag;        // zero at launch
    int32_t *status;
};

// Byte offsets of the regions of a CTA's dynamic shared memory.
struct SmemPlan {
    uint32_t w_off, rowptr_off, mid_off, sorted_off, cnt_off, in_off, gate_off, total;
    int rows_cap;
};

inline SmemPlan smem_plan(int kept_cap, int rows_cap, bool bf16, bool gru, int in_rows, int bt) {
    SmemPlan p{};
    p.rows_cap = rows_cap;
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o = (o + bytes + 15) / 16 * 16;
        return static_cast<uint32_t>(at);
    };
    p.w_off = take(size_t(kept_cap) * (bf16 ? 4 : 8));
    p.rowptr_off = take(size_t(rows_cap + 1) * 4);
    p.mid_off = take(size_t(rows_cap) * 4);
    p.sorted_off = take(size_t(rows_cap) * 4);
    p.cnt_off = take(size_t(rows_cap) * 4);
    p.in_off = take(size_t(in_rows) * bt * 4);
    p.gate_off = take(size_t(gru ? 2 : 1) * rows_cap * bt * 4);
    p.total = static_cast<uint32_t>(std::min<size_t>(o, UINT32_MAX));
    return p;
}

// Kept weight p of the CTA: value and absolute column.
template <bool BF16> struct Packed;
template <> struct Packed<true> {   // bf16 bits << 16 | column
    using T = uint32_t;
    static __device__ __forceinline__ T make(uint32_t bits, uint32_t col) { return (bits << 16) | col; }
    static __device__ __forceinline__ float val(T w) { return __uint_as_float(w & 0xFFFF0000u); }
    static __device__ __forceinline__ uint32_t col(T w) { return w & 0xFFFFu; }
};
template <> struct Packed<false> {  // fp32 bits, column
    using T = uint2;
    static __device__ __forceinline__ T make(uint32_t bits, uint32_t col) { return make_uint2(bits, col); }
    static __device__ __forceinline__ float val(T w) { return __uint_as_float(w.x); }
    static __device__ __forceinline__ uint32_t col(T w) { return w.y; }
};

// Grid-wide barrier with a time limit (the arrive/spin/fence pattern of a
// cooperative grid sync); false if this CTA gave up or another CTA did.
__device__ __forceinline__ bool grid_barrier(const SeqArgs &a, unsigned target, int *s_ok) {
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();   // the CTA's h_t stores are visible before its arrival counts
        atomicAdd(a.bar, 1u);
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
                if (global_timer_ns() - t0 > kWaitLimitNs) {
                    ok = 0;
                    atomicExch(a.abort_flag, 1);
                    atomicOr(a.status, kStatusTimeout);
                    break;
                }
                __nanosleep(32);
            }
        }
        __threadfence();
        *s_ok = ok;
    }
    __syncthreads();
    return *s_ok != 0;
}

// Input staging modes, chosen on the host from the shapes and alignments.
constexpr int kStageScalar = 0;   // one float per load
constexpr int kStageQuadCols = 1; // 4 batch columns per 16-byte load (B and bt multiples of 4, aligned)
constexpr int kStageQuadRows = 2; // B == 1: 4 input rows per 16-byte load (I, H multiples of 4, aligned)
constexpr int kStageUnroll = 8;   // loads a thread has in flight

// s_in[k][j] = [x_t; h_{t-1}][k][b0 + j] for j < nb, 0 for nb <= j < bt.
// h_{t-1} was written by other CTAs of this launch, so every load goes to L2
// (ld.cg); the loads of a thread are issued together so that enough bytes are
// in flight to cover the L2 latency.
__device__ __forceinline__ void stage_input(const SeqArgs &a, const float *xt, const float *hp, int64_t b0, int nb,
                                            float *s_in) {
    const int I = a.I, K = a.I + a.H, lbt = a.lbt, bt = 1 << lbt;
    const int64_t B = a.B;
    const int tid = threadIdx.x;
    auto src = [&](int k) { return k < I ? xt + int64_t(k) * B : hp + int64_t(k - I) * B; };
    if (a.stage_mode == kStageQuadCols) {
        const int lq = lbt - 2, n = K << lq;   // quads
        for (int i0 = tid; i0 < n; i0 += kThreads * kStageUnroll) {
            float4 v[kStageUnroll];
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u) {
                const int i = i0 + u * kThreads;
                const int k = i >> lq, j = (i & ((1 << lq) - 1)) * 4;
                v[u] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
                if (i < n && j < nb) v[u] = __ldcg(reinterpret_cast<const float4 *>(src(k) + b0 + j));
            }
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u)
                if (i0 + u * kThreads < n) reinterpret_cast<float4 *>(s_in)[i0 + u * kThreads] = v[u];
        }
    } else if (a.stage_mode == kStageQuadRows) {
        const int n = K >> 2;
        for (int i0 = tid; i0 < n; i0 += kThreads * kStageUnroll) {
            float4 v[kStageUnroll];
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u) {
                const int i = i0 + u * kThreads;
                if (i < n) v[u] = __ldcg(reinterpret_cast<const float4 *>(src(4 * i)));
            }
#pragma unroll
            for (int u = 0; u < kStageUnroll; ++u)
                if (i0 + u * kThreads < n) reinterpret_cast<float4 *>(s_in)[i0 + u * kThreads] = v[u];
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
seq_kernel(Format f, SeqArgs a, Ranges rg, SmemPlan sp) {
    constexpr int kGates = MODE == kModeLstm ? 4 : 3;
    constexpr bool kGru = MODE == kModeGru;
    using P = Packed<BF16>;
    using PT = typename P::T;
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ int s_ok;
    PT *s_w = reinterpret_cast<PT *>(sm + sp.w_off);
    int *s_rowptr = reinterpret_cast<int *>(sm + sp.rowptr_off);
    int *s_mid = reinterpret_cast<int *>(sm + sp.mid_off);        // GRU: first kept weight on h
    int *s_sorted = reinterpret_cast<int *>(sm + sp.sorted_off);  // local rows, most weights first
    int *s_cnt = reinterpret_cast<int *>(sm + sp.cnt_off);
    float *s_in = reinterpret_cast<float *>(sm + sp.in_off);      // [I + H][bt]
    float *s_gate = reinterpret_cast<float *>(sm + sp.gate_off);  // [parts][R][bt]
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int u0 = rg.start[blockIdx.x], nu = rg.start[blockIdx.x + 1] - u0;
    const int R = kGates * nu;   // local row q*nu + i is matrix row q*H + u0 + i
    const int I = a.I, H = a.H;
    const int lbt = a.lbt, bt = 1 << lbt, S = 32 >> lbt;
    const int sub = lane >> lbt, col = lane & (bt - 1);
    const int64_t B = a.B;
    auto grow = [&](int lr) { return (lr / nu) * H + u0 + lr % nu; };

    // ---- prologue: weights per row, row pointers, rows by descending weight count
    for (int lr = tid; lr < R; lr += kThreads) s_cnt[lr] = f.groups[f.rowloc[grow(lr)] / kSlots].n;
    __syncthreads();
    if (tid == 0) {
        int p = 0;
        for (int lr = 0; lr < R; ++lr) {
            s_rowptr[lr] = p;
            p += s_cnt[lr];
        }
        s_rowptr[R] = p;
    }
    for (int lr = tid; lr < R; lr += kThreads) {
        int rank = 0;
        const int n = s_cnt[lr];
        for (int l = 0; l < R; ++l) rank += (s_cnt[l] > n || (s_cnt[l] == n && l < lr)) ? 1 : 0;
        s_sorted[rank] = lr;
    }
    __syncthreads();
    for (int lr = warp; lr < R; lr += kSeqWarps) {
        const int loc = f.rowloc[grow(lr)];
        const Group g = f.groups[loc / kSlots];
        const int slot = loc % kSlots;
        const int base = s_rowptr[lr];
        const int jmid = I / g.m;   // the only block that can hold columns on both sides of I
        for (int j = lane; j < g.n; j += 32) {
            const int64_t rec = int64_t(j / kChunk) * kSlots + slot;
            const int q = j % kChunk;
            uint32_t bits;
            if constexpr (BF16) bits = static_cast<const uint16_t *>(f.vals)[g.val_off + rec * kChunk + q];
            else bits = static_cast<const uint32_t *>(f.vals)[g.val_off + rec * kChunk + q];
            uint32_t o;
            if (g.nib) o = (f.offs[g.off_off + rec] >> (4 * q)) & 15u;
            else o = (f.offs[g.off_off + 2 * rec + (q >> 2)] >> (8 * (q & 3))) & 255u;
            const uint32_t c = uint32_t(j) * uint32_t(g.m) + o;
            s_w[base + j] = P::make(bits, c);
            if (j == jmid) s_mid[lr] = base + j + (c < uint32_t(I) ? 1 : 0);
        }
    }
    __syncthreads();

    // ---- the steps
    float *c_state = kGru ? nullptr : a.c_state + int64_t(u0) * B;
    for (int t = 0; t < a.T; ++t) {
        const float *xt = a.x + int64_t(t) * I * B;
        const float *hp = t == 0 ? a.h0 : a.h_seq + int64_t(t - 1) * H * B;
        float *ht = a.h_seq + int64_t(t) * H * B + int64_t(u0) * B;
        float *ct = a.c_seq ? a.c_seq + int64_t(t) * H * B + int64_t(u0) * B : nullptr;
        const float *cp = kGru ? nullptr : (t == 0 ? a.c0 + int64_t(u0) * B : c_state);
        for (int64_t b0 = 0; b0 < B; b0 += bt) {
            const int nb = static_cast<int>(B - b0 < bt ? B - b0 : bt);
            // stage [x_t; h_{t-1}] for columns [b0, b0 + nb), zeros past the batch
            stage_input(a, xt, hp, b0, nb, s_in);
            __syncthreads();
            // gate sums; rows go to warps in a snake over the sorted order
            for (int r0 = 0; r0 < R; r0 += kSeqWarps) {
                const int round = r0 / kSeqWarps;
                const int si = r0 + ((round & 1) ? kSeqWarps - 1 - warp : warp);
                if (si >= R) continue;
                const int lr = s_sorted[si];
                const int p0 = s_rowptr[lr], p1 = s_rowptr[lr + 1];
                const int pm = kGru ? s_mid[lr] : p1;
                float ax = 0.0f, ah = 0.0f;
                int p = p0 + sub;
                for (; p + 3 * S < pm; p += 4 * S) {
                    const PT w0 = s_w[p], w1 = s_w[p + S], w2 = s_w[p + 2 * S], w3 = s_w[p + 3 * S];
                    const float v0 = s_in[(P::col(w0) << lbt) + col], v1 = s_in[(P::col(w1) << lbt) + col];
                    const float v2 = s_in[(P::col(w2) << lbt) + col], v3 = s_in[(P::col(w3) << lbt) + col];
                    ax = fmaf(P::val(w0), v0, ax);
                    ax = fmaf(P::val(w1), v1, ax);
                    ax = fmaf(P::val(w2), v2, ax);
                    ax = fmaf(P::val(w3), v3, ax);
                }
                for (; p < pm; p += S) {
                    const PT w = s_w[p];
                    ax = fmaf(P::val(w), s_in[(P::col(w) << lbt) + col], ax);
                }
                if constexpr (kGru) {
                    // the h part starts at pm; each subgroup keeps its stride from there
                    p = pm + sub;
                    for (; p + 3 * S < p1; p += 4 * S) {
                        const PT w0 = s_w[p], w1 = s_w[p + S], w2 = s_w[p + 2 * S], w3 = s_w[p + 3 * S];
                        const float v0 = s_in[(P::col(w0) << lbt) + col], v1 = s_in[(P::col(w1) << lbt) + col];
                        const float v2 = s_in[(P::col(w2) << lbt) + col], v3 = s_in[(P::col(w3) << lbt) + col];
                        ah = fmaf(P::val(w0), v0, ah);
                        ah = fmaf(P::val(w1), v1, ah);
                        ah = fmaf(P::val(w2), v2, ah);
                        ah = fmaf(P::val(w3), v3, ah);
                    }
                    for (; p < p1; p += S) {
                        const PT w = s_w[p];
                        ah = fmaf(P::val(w), s_in[(P::col(w) << lbt) + col], ah);
                    }
                }
                for (int o = 16; o >= bt; o >>= 1) {
                    ax += __shfl_xor_sync(0xFFFFFFFFu, ax, o);
                    if constexpr (kGru) ah += __shfl_xor_sync(0xFFFFFFFFu, ah, o);
                }
                if (sub == 0) {
                    s_gate[(lr << lbt) + col] = ax;
                    if constexpr (kGru) s_gate[((R + lr) << lbt) + col] = ah;
                }
            }
            __syncthreads();
            // the cells of the owned units for these columns
            for (int i = tid; i < nu << lbt; i += kThreads) {
                const int ui = i >> lbt, j = i & (bt - 1), u = u0 + ui;
                if (j >= nb) continue;
                const int64_t e = int64_t(ui) * B + b0 + j;
                if constexpr (MODE == kModeLstm) {
                    float pre[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        pre[q] = s_gate[((q * nu + ui) << lbt) + j] + (a.bias ? a.bias[q * H + u] : 0.0f);
                    const float c = sigm(pre[1]) * cp[e] + sigm(pre[0]) * tanhf(pre[2]);
                    c_state[e] = c;
                    if (ct) ct[e] = c;
                    ht[e] = sigm(pre[3]) * tanhf(c);
                } else {
                    float ax[3], bh[3];
#pragma unroll
                    for (int q = 0; q < 3; ++q) {
                        ax[q] = s_gate[((q * nu + ui) << lbt) + j] + (a.b_ih ? a.b_ih[q * H + u] : 0.0f);
                        bh[q] = s_gate[((R + q * nu + ui) << lbt) + j] + (a.b_hh ? a.b_hh[q * H + u] : 0.0f);
                    }
                    const float rr = sigm(ax[0] + bh[0]);
                    const float zz = sigm(ax[1] + bh[1]);
                    const float nn = tanhf(ax[2] + rr * bh[2]);
                    ht[e] = (1.0f - zz) * nn + zz * s_in[((I + u) << lbt) + j];
                }
            }
            __syncthreads();
        }
        if (t + 1 < a.T && !grid_barrier(a, unsigned(t + 1) * gridDim.x, &s_ok)) return;
    }
}

}  // namespace seq

namespace {

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

template <bool BF16, int MODE>
static cudaError_t launch_seq_t(const Format &f, const int32_t *row_m, seq::SeqArgs a, float *c_last,
                                cudaStream_t stream) {
    using namespace seq;
    constexpr int kGates = MODE == kModeLstm ? 4 : 3;
    constexpr bool kGru = MODE == kModeGru;
    const int H = a.H, I = a.I;
    if (f.cols > 65535) return cudaErrorNotSupported;   // columns are kept in 16 bits
    std::vector<int64_t> kept(static_cast<size_t>(H));
    for (int u = 0; u < H; ++u) {
        int64_t k = 0;
        for (int q = 0; q < kGates; ++q) {
            const int64_t m = row_m[static_cast<size_t>(q) * H + u];
            k += (f.cols + m - 1) / m;
        }
        kept[static_cast<size_t>(u)] = k;
    }
    const int G = std::max(1, std::min({sm_count(), H, kMaxCtas}));
    Ranges rg{};
    int64_t kept_cap = 0;
    int units_cap = 0;
    split_units(kept, G, rg, kept_cap, units_cap);
    if (kept_cap > (int64_t(1) << 20)) return cudaErrorNotSupported;
    // widest batch tile (a power of two, <= 32) whose staging still fits
    int bt = 1;
    while (bt < kMaxTile && bt < a.B) bt *= 2;
    SmemPlan sp{};
    for (;; bt /= 2) {
        sp = smem_plan(static_cast<int>(kept_cap), kGates * units_cap, BF16, kGru, I + H, bt);
        if (sp.total <= kSmemCap) break;
        if (bt == 1) return cudaErrorNotSupported;
    }
    a.lbt = 0;
    while ((1 << a.lbt) < bt) ++a.lbt;
    auto aligned = [](const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
    const bool ptrs = (I == 0 || aligned(a.x)) && aligned(a.h0) && aligned(a.h_seq);
    a.stage_mode = kStageScalar;
    if (ptrs && a.B % 4 == 0 && bt % 4 == 0) a.stage_mode = kStageQuadCols;
    else if (ptrs && a.B == 1 && I % 4 == 0 && H % 4 == 0) a.stage_mode = kStageQuadRows;
    static const cudaError_t attr = cudaFuncSetAttribute(seq_kernel<BF16, MODE>,
                                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                         static_cast<int>(kSmemCap));
    if (attr != cudaSuccess) return attr;
    // workspace: barrier word, abort flag, and the cell state unless c_last holds it
    const size_t cbytes = kGru || c_last ? 0 : size_t(H) * size_t(a.B) * 4;
    void *ws = nullptr;
    cudaError_t e = cudaMallocAsync(&ws, 256 + cbytes, stream);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(ws, 0, 16, stream);
    a.bar = static_cast<unsigned *>(ws);
    a.abort_flag = reinterpret_cast<int *>(static_cast<char *>(ws) + 4);
    a.c_state = kGru ? nullptr : (c_last ? c_last : reinterpret_cast<float *>(static_cast<char *>(ws) + 256));
    if (e == cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(G));
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = sp.total;
        cfg.stream = stream;
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeCooperative;
        at[0].val.cooperative = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, seq_kernel<BF16, MODE>, f, a, rg, sp);
    }
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
