// tcgen05.cuh -- inline-PTX helpers for the 5th-generation tensor cores of
// sm_103a: tensor-memory (TMEM) allocation, shared-memory matrix descriptors,
// the instruction descriptor of kind::f16 (bf16 operands), tcgen05.mma /
// commit, and loads of the accumulator back to registers.
//
// Conventions used by the kernels here (cta_group::1, M = 128):
//  * the accumulator D is 128 TMEM lanes (one per row of A) by N 32-bit
//    columns; warp w of a CTA may read lanes [32*(w%4), 32*(w%4)+32);
//  * A and B are read from shared memory through 64-bit descriptors naming a
//    swizzled canonical layout: with 128-byte swizzle, 8-row x 128-byte atoms
//    whose 16-byte chunk c of row r sits at chunk c ^ (r % 8); with 64-byte
//    swizzle, 8-row x 64-byte atoms, chunk c of row r at c ^ ((r / 2) % 4).
//    Atoms are aligned to their size; a K step inside an atom advances the
//    start address only.
//  * tf32 operands are not used: with an MN-major B they produced zeros on
//    this part, and the activations X are MN-major (batch contiguous).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "tma.cuh"

namespace darb {

// Allocate `ncols` TMEM columns (a power of two, 32..512) for this CTA; the
// base address is written to *dst.  Executed by one whole warp.
__device__ __forceinline__ void tmem_alloc(uint32_t *dst, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(dst)),
                 "r"(ncols)
                 : "memory");
}

__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

// Executed by the same warp that allocated.
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// Order tcgen05 operations around a thread synchronisation (barrier, mbarrier).
__device__ __forceinline__ void tc_fence_before_sync() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after_sync() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory layouts the descriptors can name.
constexpr uint32_t kLayoutSw128 = 2;   // 128-byte swizzle: 8-row x 128-byte atoms
constexpr uint32_t kLayoutSw64 = 4;    // 64-byte swizzle: 8-row x 64-byte atoms

// Shared-memory matrix descriptor.  lbo/sbo in bytes: K-major operands use
// sbo = the stride between 8-row groups (lbo unused); MN-major operands use
// lbo = the stride between swizzle-wide column groups and sbo = the stride
// between 8-deep K groups.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo, uint32_t layout) {
    uint64_t d = 0;
    d |= uint64_t((saddr & 0x3FFFFu) >> 4);              // start address, bits 0-13
    d |= uint64_t((lbo >> 4) & 0x3FFFu) << 16;           // leading byte offset, bits 16-29
    d |= uint64_t((sbo >> 4) & 0x3FFFu) << 32;           // stride byte offset, bits 32-45
    d |= uint64_t(1) << 46;                              // descriptor version for tcgen05
    d |= uint64_t(layout) << 61;                         // swizzle mode, bits 61-63
    return d;
}

// Instruction descriptor of tcgen05.mma kind::f16 with bf16 A and B and an
// fp32 accumulator; A K-major (MN-major if a_mn), B MN-major if b_mn; M x N.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool a_mn, bool b_mn) {
    return (1u << 4)                            // D format: f32
           | (1u << 7)                          // A format: bf16
           | (1u << 10)                         // B format: bf16
           | (uint32_t(a_mn) << 15)             // A major-ness
           | (uint32_t(b_mn) << 16)             // B major-ness
           | (uint32_t(N >> 3) << 17)           // N / 8
           | (uint32_t(M >> 4) << 24);          // M / 16
}

// D[tmem] (+)= A[desc] * B[desc] (K = 16); accumulate when acc != 0.  One thread issues.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t acc) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(acc)
        : "memory");
}

// Arrive (once) on `bar` when every tcgen05.mma this thread issued so far is complete.
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     smem_addr(bar))
                 : "memory");
}

// 32 consecutive accumulator columns of this thread's lane (32x32b shape, 32 repeats).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
          "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
          "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void prefetch_tensormap(const void *map) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(map) : "memory");
}

}  // namespace darb
