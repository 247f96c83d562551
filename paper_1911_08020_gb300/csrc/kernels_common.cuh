// kernels_common.cuh -- device pieces shared by the product and RNN-step kernels:
// chunk loads of kept values, offset unpacking, and the "row per lane" gather-FMA
// loop over a range of chunks.
//
// The product is Y[r, b] = sum_j val[r, j] * X[j*m_r + off[r, j], b]
// (Sec. 3.2, Fig. 6(b): block j of a row selects one of its m activations).
// A warp's lane i works on slot i of a 32-row group, so at any instant the 32
// lanes gather from the same window [j*m, j*m + m) of X: for m <= 32 that is
// at most one or two 128-byte lines, and lanes that pick the same activation
// share the load.
#pragma once

#include "darb_internal.h"

namespace darb {

constexpr int kWarps = 8;   // warps per CTA for the row-per-lane kernels

// acc += v * x for a float4 accumulator with two packed fp32 FMAs (PTX
// fma.rn.f32x2, sm_100 and later): each element is one IEEE fma, as fmaf,
// in half the instructions.
__device__ __forceinline__ void fma4(float4 &acc, float v, const float4 &x) {
    asm("{\n"
        " .reg .b64 vv, xl, xh, al, ah;\n"
        " mov.b64 vv, {%8, %8};\n"
        " mov.b64 xl, {%4, %5};\n"
        " mov.b64 xh, {%6, %7};\n"
        " mov.b64 al, {%0, %1};\n"
        " mov.b64 ah, {%2, %3};\n"
        " fma.rn.f32x2 al, vv, xl, al;\n"
        " fma.rn.f32x2 ah, vv, xh, ah;\n"
        " mov.b64 {%0, %1}, al;\n"
        " mov.b64 {%2, %3}, ah;\n"
        "}"
        : "+f"(acc.x), "+f"(acc.y), "+f"(acc.z), "+f"(acc.w)
        : "f"(x.x), "f"(x.y), "f"(x.z), "f"(x.w), "f"(v));
}

// The 8 kept values of (chunk c, slot i), widened to fp32 (bf16 -> fp32 is exact).
template <bool BF16>
__device__ __forceinline__ void load_chunk(const void *vals, int64_t idx, float (&v)[kChunk]) {
    if constexpr (BF16) {
        const uint4 q = __ldg(reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(vals) + idx));
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            v[2 * e] = __uint_as_float(w[e] << 16);
            v[2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
        }
    } else {
        const float4 *p = reinterpret_cast<const float4 *>(static_cast<const float *>(vals) + idx);
        const float4 a = __ldg(p), b = __ldg(p + 1);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
}

// Offset record of (chunk c, slot i): one word of nibbles or two words of bytes.
template <bool NIB>
__device__ __forceinline__ uint2 load_offsets(const uint32_t *offs, int64_t rec) {
    if constexpr (NIB) {
        return make_uint2(__ldg(offs + rec), 0u);
    } else {
        return __ldg(reinterpret_cast<const uint2 *>(offs) + rec);
    }
}

template <bool NIB>
__device__ __forceinline__ int unpack_offset(uint2 w, int e) {
    if constexpr (NIB) {
        return (w.x >> (4 * e)) & 15u;
    } else {
        return ((e < 4 ? w.x : w.y) >> (8 * (e & 3))) & 255u;
    }
}

// Activation source: a single X, or the stacked RNN input [x; h].
struct XPlain {
    const float *X;
    int64_t ldx;
    __device__ __forceinline__ const float *row(int k) const { return X + static_cast<int64_t>(k) * ldx; }
    __device__ __forceinline__ bool first_part(int) const { return true; }
};

struct XStacked {
    const float *x;   // I x ld
    const float *h;   // H x ld
    int I;
    int64_t ld;
    __device__ __forceinline__ const float *row(int k) const {
        return k < I ? x + static_cast<int64_t>(k) * ld : h + static_cast<int64_t>(k - I) * ld;
    }
    __device__ __forceinline__ bool first_part(int k) const { return k < I; }
};

// Accumulate chunks [c_begin, c_end) of slot `slot` of group `g` into acc (and,
// when SPLIT, the products whose activation lies in the second part of a
// stacked input into acc2), for batch columns b0 .. b0+nb-1 (nb <= BT).
template <bool BF16, bool NIB, int BT, bool SPLIT, class XS>
__device__ __forceinline__ void rowlane_accumulate(const Format &f, const Group &g, int slot,
                                                   int c_begin, int c_end, const XS &xs,
                                                   int64_t b0, int nb, float (&acc)[BT],
                                                   float (&acc2)[BT]) {
    const int m = g.m, n = g.n;
    for (int c = c_begin; c < c_end; ++c) {
        float v[kChunk];
        load_chunk<BF16>(f.vals, g.val_off + (static_cast<int64_t>(c) * kSlots + slot) * kChunk, v);
        const uint2 ow = load_offsets<NIB>(f.offs + g.off_off, static_cast<int64_t>(c) * kSlots + slot);
        const bool full = (c + 1) * kChunk <= n;
#pragma unroll
        for (int e = 0; e < kChunk; ++e) {
            const int j = c * kChunk + e;
            if (full || j < n) {
                const int k = j * m + unpack_offset<NIB>(ow, e);
                const float *xr = xs.row(k) + b0;
                const bool p1 = !SPLIT || xs.first_part(k);
#pragma unroll
                for (int t = 0; t < BT; ++t) {
                    if (t < nb) {
                        const float xv = __ldg(xr + t);
                        if (p1) acc[t] = fmaf(v[e], xv, acc[t]);
                        else acc2[t] = fmaf(v[e], xv, acc2[t]);
                    }
                }
            }
        }
    }
}

__device__ __forceinline__ float sigmoidf_(float v) { return 1.0f / (1.0f + expf(-v)); }

}  // namespace darb
