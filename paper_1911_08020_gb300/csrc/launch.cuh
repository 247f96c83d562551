// launch.cuh -- cudaLaunchKernelEx wrapper: thread-block clusters and
// programmatic dependent launch (PDL) on the caller's stream; the driver's
// tensor-map encoder.
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <atomic>
#include <map>
#include <mutex>
#include <tuple>
#include <utility>

namespace darb {

// Whether kernels are launched with programmatic dependent launch (process
// wide; darb_set_pdl).  On by default.
inline std::atomic<int> &pdl_setting() {
    static std::atomic<int> on{1};
    return on;
}
inline bool pdl_enabled() { return pdl_setting().load(std::memory_order_relaxed) != 0; }

// The calling thread's current device (0 if it cannot be read).
inline int current_device() {
    int d = 0;
    if (cudaGetDevice(&d) != cudaSuccess) {
        cudaGetLastError();
        d = 0;
    }
    return d;
}

namespace detail {
inline std::mutex &cache_mutex() {
    static std::mutex mu;
    return mu;
}
// (key, sub-key, device) -> value
inline std::map<std::tuple<const void *, long long, int>, long long> &cache_map() {
    static std::map<std::tuple<const void *, long long, int>, long long> m;
    return m;
}
}  // namespace detail

// A figure computed once per (key, sub-key, device) and kept for the process:
// kernel attributes and occupancy belong to a device, so a process that
// drives several devices computes them on each.  `compute` runs outside the
// lock (it may call the runtime); two threads may both compute a missing entry.
template <class F>
long long per_device(const void *key, long long sub, F compute) {
    const auto k = std::make_tuple(key, sub, current_device());
    {
        std::lock_guard<std::mutex> lk(detail::cache_mutex());
        const auto it = detail::cache_map().find(k);
        if (it != detail::cache_map().end()) return it->second;
    }
    const long long v = compute();
    std::lock_guard<std::mutex> lk(detail::cache_mutex());
    detail::cache_map()[k] = v;
    return v;
}

template <typename... KArgs, typename... Args>
cudaError_t launch_ex(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                      cudaStream_t stream, unsigned cluster, bool pdl, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    unsigned n = 0;
    if (cluster > 1) {
        attr[n].id = cudaLaunchAttributeClusterDimension;
        attr[n].val.clusterDim.x = cluster;
        attr[n].val.clusterDim.y = 1;
        attr[n].val.clusterDim.z = 1;
        ++n;
    }
    if (pdl && pdl_enabled()) {
        attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Raise a kernel's dynamic shared memory limit to at least `bytes` on the
// current device (once per kernel, device and larger size).
template <typename... KArgs>
cudaError_t allow_smem(void (*kernel)(KArgs...), size_t bytes) {
    if (bytes <= 48 * 1024) return cudaSuccess;
    const void *fn = reinterpret_cast<const void *>(kernel);
    const auto k = std::make_tuple(fn, -1ll, current_device());
    std::lock_guard<std::mutex> lk(detail::cache_mutex());
    auto &m = detail::cache_map();
    const auto it = m.find(k);
    if (it != m.end() && it->second >= static_cast<long long>(bytes)) return cudaSuccess;
    const cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
    if (e != cudaSuccess) {
        cudaGetLastError();
        return e;
    }
    m[k] = static_cast<long long>(bytes);
    return cudaSuccess;
}

// cuTensorMapEncodeTiled from the driver (through the runtime, so that the
// library does not link libcuda); nullptr if unavailable.
inline PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            cudaGetLastError();
            return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
        }
        return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }();
    return fn;
}

}  // namespace darb
