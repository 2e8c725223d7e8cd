// static_scratch.cu -- rps_score_step_noalloc: row statistics with library-owned
// scratch, for callers that cannot allocate device memory.
//
// The scratch is one file-scope device array of RPS_STATIC_SCRATCH_BYTES. Host
// code cannot use the array's name as a device address (in host code it names a
// host-side stand-in), so the first call on each device looks its device address
// up with cudaGetSymbolAddress while that device is current and caches it.
#include <cstring>
#include <mutex>

#include "rps_internal.cuh"

namespace {

static __device__ __align__(256) unsigned char g_static_scratch[RPS_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mutex;
void *g_scratch_ptr[kMaxDevices] = {};

// Device address of this device's scratch array; set up once per device.
rps_status scratch_for_current_device(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RPS_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) return RPS_ERR_CUDA;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return RPS_OK;
}

}  // namespace

extern "C" rps_status rps_score_step_noalloc(const rps_logits *logits, const rps_row_list *rows,
                                             const rps_params *prm, const rps_row_stats *out,
                                             rps_stream_t stream) {
    // the argument rules of rps_score_step, checked before anything is enqueued
    int32_t k = 0;
    const rps_status arg = rps::check_row_stats_args(logits, rows, prm, out, &k);
    if (arg != RPS_OK) return arg;
    const size_t need =
        rps_workspace_bytes(static_cast<int64_t>(rows->n_seg) * rows->cap, logits->vocab, logits->dtype, k);
    if (need == 0) return RPS_ERR_INVALID_ARG;
    if (need > RPS_STATIC_SCRATCH_BYTES) return RPS_ERR_UNSUPPORTED;  // beyond the fixed scratch

    void *scratch = nullptr;
    const rps_status st = scratch_for_current_device(&scratch);
    if (st != RPS_OK) return st;
    // The array keeps whatever the previous call left; the per-row completion
    // tickets and the health word must start at zero, so the part of the array
    // this call uses is cleared on the call's stream (a memset, no allocation).
    if (cudaMemsetAsync(scratch, 0, need, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) return RPS_ERR_CUDA;
    return rps_score_step(logits, rows, prm, out, scratch, RPS_STATIC_SCRATCH_BYTES, stream);
}
