// tma.cuh -- inline-PTX helpers for sm_103a: mbarriers, bulk (TMA) copies into
// shared memory, programmatic dependent launch, and bounded waits.
//
// Every wait here is bounded: after kWaitLimitNs of wall time it gives up and
// returns false, so a kernel can record an error and leave instead of hanging.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace darb {

constexpr unsigned long long kWaitLimitNs = 1000000000ull;   // 1 s

// Device status word bits (sticky until read by darb_sync_status).
constexpr int kStatusNaN = 1;
constexpr int kStatusTimeout = 2;

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long global_timer_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

// Make mbarrier initialisation visible to the async (TMA) proxy.
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}

// Plain arrival (release) on an mbarrier.
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

// Add expected transaction bytes to the current phase without arriving.
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.expect_tx.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes) : "memory");
}

// Wait for the phase with the given parity to complete; false after the time
// limit.  Each try_wait suspends the thread in hardware while the phase is
// pending (up to the hint), so polling costs few issue slots and the wait
// ends as soon as the phase completes.  With `backoff` the thread also sleeps
// between attempts (32 ns doubling to 512 ns); only for waits that are long
// and not on a critical path: a thread that sleeps past the completion holds
// up every thread that waits for it (a warp's shuffle, a CTA barrier).
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, bool backoff = false) {
    const uint32_t a = smem_addr(bar);
    unsigned long long t0 = 0;
    unsigned sleep_ns = 32;
    while (true) {
        uint32_t done;
        asm volatile(
            "{\n .reg .pred p;\n"
            " mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
            " selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(done) : "r"(a), "r"(parity), "r"(10000u) : "memory");
        if (done) return true;
        const unsigned long long now = global_timer_ns();
        if (t0 == 0) t0 = now;
        else if (now - t0 > kWaitLimitNs) return false;
        if (backoff) {
            __nanosleep(sleep_ns);
            if (sleep_ns < 512) sleep_ns <<= 1;
        }
    }
}

// 1-D bulk copy global -> this CTA's shared memory, completing on `bar`.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(smem_addr(dst)), "l"(src), "r"(bytes), "r"(smem_addr(bar)) : "memory");
}

// 2-D tensor-map copy (box at coordinates x = innermost, y) -> shared memory.
// x * element size must be a multiple of 16 bytes.
__device__ __forceinline__ void tensor2d_g2s(void *dst, const void *tmap, int x, int y, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];"
        ::"r"(smem_addr(dst)), "l"(tmap), "r"(x), "r"(y), "r"(smem_addr(bar)) : "memory");
}

// 3-D tensor-map copy (box at coordinates x = innermost, y, z) -> this CTA's
// shared memory, completing on `bar`.  x * element size must be a multiple of
// 16 bytes; dst 128-byte aligned.
__device__ __forceinline__ void tensor3d_g2s(void *dst, const void *tmap, int x, int y, int z, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];"
        ::"r"(smem_addr(dst)), "l"(tmap), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar)) : "memory");
}

// Order this thread's earlier generic-proxy view of global memory (e.g. data
// other CTAs published through a release/acquire handshake) before its later
// async-proxy (TMA) reads.
__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Arrive on the mbarrier at the same shared-memory offset as `bar` in CTA
// `rank` of this cluster, with the default semantics (release at CTA scope):
// it orders this CTA's earlier accesses to its own shared memory (made by
// other threads too, after a CTA barrier) before the arrival -- enough to
// hand shared-memory data to another CTA, which reads it through distributed
// shared memory -- without waiting for this CTA's global stores to drain, as
// a release at cluster scope would.
__device__ __forceinline__ void mbar_arrive_remote(uint64_t *bar, uint32_t rank) {
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_addr(bar)), "r"(rank));
    asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(remote) : "memory");
}

// mbar_wait with acquire at cluster scope, for phases completed by arrivals of
// other CTAs of the cluster (mbar_arrive_remote); false after the time limit.
// With `backoff` the thread sleeps between attempts (as mbar_wait), so that a
// warp that waits long leaves the issue slots to the others.
__device__ __forceinline__ bool mbar_wait_acq_cluster(uint64_t *bar, uint32_t parity, bool backoff = false) {
    const uint32_t a = smem_addr(bar);
    unsigned long long t0 = 0;
    unsigned sleep_ns = 32;
    while (true) {
        uint32_t done;
        asm volatile(
            "{\n .reg .pred p;\n"
            " mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n"
            " selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(done) : "r"(a), "r"(parity), "r"(10000u) : "memory");
        if (done) return true;
        const unsigned long long now = global_timer_ns();
        if (t0 == 0) t0 = now;
        else if (now - t0 > kWaitLimitNs) return false;
        if (backoff) {
            __nanosleep(sleep_ns);
            if (sleep_ns < 512) sleep_ns <<= 1;
        }
    }
}

// Named barrier `id` (1..15) over `threads` threads of the CTA (a multiple of
// 32; the warps that take part all call it with the same id and count).
__device__ __forceinline__ void named_sync(uint32_t id, uint32_t threads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Programmatic dependent launch: let the next kernel on the stream start its
// prologue, and wait until the previous kernel's writes are visible.
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ void pdl_wait_previous() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

}  // namespace darb
