// noalloc.cu -- an LSTM step that allocates no device memory.
//
// darb_lstm_step keeps its gate sums and per-unit arrival counters in scratch
// that the handle owns and allocates with cudaMalloc the first time a step
// needs more than it holds.  Some callers cannot let a library allocate at
// that point: a serving loop running under a fixed memory budget, where any
// cudaMalloc outside start-up can fail or stall every stream on the device;
// code that must not synchronise the device mid-stream (cudaMalloc and
// cudaFree can); and callers whose allocations all go through their own pool.
// darb_lstm_step_noalloc runs the same kernel with that scratch in one fixed
// array compiled into this library instead, so nothing is allocated at call
// time (or ever, apart from the array itself, which every GPU that loads the
// library holds until the process exits).
#include "darb.h"
#include "trace.h"
#include "darb_internal.h"

#include <mutex>

namespace {

// Scratch shared by every darb_lstm_step_noalloc call on a device: gate sums
// (4H x B floats) followed by arrival counters (H x batch tiles ints).
constexpr size_t kNoAllocScratchBytes = size_t(4) << 20;
static __device__ __align__(256) unsigned char g_step_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_scratch_addr[kMaxDevices] = {};

// Device address of g_step_scratch on the current device.  The name itself is
// only a host-side stand-in; the first call on each device looks the address
// up once and keeps it.
darb_status_t scratch_address(void **out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return DARB_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) return DARB_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_scratch_addr[dev] == nullptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_step_scratch) != cudaSuccess || p == nullptr) {
            cudaGetLastError();
            return DARB_ERR_CUDA;
        }
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return DARB_OK;
}

}  // namespace

extern "C" darb_status_t darb_lstm_step_noalloc(darb_handle_t h, int64_t I, int64_t H, int64_t B,
                                                const float *x, const float *h_prev,
                                                const float *c_prev, const float *bias,
                                                float *h_out, float *c_out, cudaStream_t stream) {
    DARB_TRACE("darb_lstm_step_noalloc");
    darb::Format f;
    darb_status_t st = darb::lstm_step_view(h, I, H, B, x, h_prev, c_prev, bias, h_out, c_out, &f);
    if (st != DARB_OK) return st;
    const size_t gate_bytes = size_t(f.rows) * size_t(B) * sizeof(float);
    const size_t gate_span = (gate_bytes + 255) / 256 * 256;
    const int bt = darb::rnn_batch_tile(B);
    const size_t counter_bytes = size_t(H) * size_t((B + bt - 1) / bt) * sizeof(int32_t);
    if (gate_span + counter_bytes > kNoAllocScratchBytes) return DARB_ERR_UNSUPPORTED;
    void *base = nullptr;
    st = scratch_address(&base);
    if (st != DARB_OK) return st;
    darb::RnnScratch sc;
    sc.gates = static_cast<float *>(base);
    sc.counters = reinterpret_cast<int32_t *>(static_cast<unsigned char *>(base) + gate_span);
    // the array keeps whatever the last call left: counters must start at zero
    if (cudaMemsetAsync(sc.counters, 0, counter_bytes, stream) != cudaSuccess) {
        cudaGetLastError();
        return DARB_ERR_CUDA;
    }
    return darb::launch_lstm_step(f, I, H, B, x, h_prev, c_prev, bias, h_out, c_out, sc, stream) == cudaSuccess
               ? DARB_OK
               : DARB_ERR_CUDA;
}
