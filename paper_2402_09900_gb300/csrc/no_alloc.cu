// no_alloc.cu -- a forward diagonal scan that needs no caller-provided
// workspace and allocates nothing.
//
// Some callers cannot hand the library a workspace: code that runs where
// device allocation is unavailable or forbidden (inside a custom allocator or
// an allocation callback, under a memory-accounting framework that must not
// see untracked buffers, or in a host runtime that pins its whole device
// budget up front).  For them memoroid_scan_diag_fwd_static uses a scratch
// array that lives in this library's own device memory: a file-scope
// __device__ array of MEMOROID_STATIC_WORKSPACE_BYTES, created when the module
// is loaded on a device and kept until the process exits.
//
// Rules of use:
//   * The first call on a device looks up the array's device address
//     (cudaGetSymbolAddress) with that device current; make that first call
//     outside any stream capture.
//   * Every call shares the one array and leaves its contents behind; the
//     scan clears the part that must start at zero itself.  Calls that
//     overlap on the GPU (different streams, or different host threads
//     without ordering) race on the array and give wrong results.
//   * Shapes whose workspace would exceed the array are rejected with
//     MEMOROID_ERR_WORKSPACE; nothing is allocated, on any path.
//   * A bounded device-side wait that runs out records MEMOROID_ERR_TIMEOUT in
//     the array's header like in any workspace; callers never see the array's
//     address, so memoroid_get_static_device_error reads it for them.
//   * The address is cached per device: after cudaDeviceReset the process
//     must not call these entry points on that device again.
#include <cuda_runtime.h>

#include <mutex>

#include "internal.cuh"

namespace memoroid {
namespace {

constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_static_ws[MEMOROID_STATIC_WORKSPACE_BYTES];

std::mutex g_mutex;
void* g_ws_ptr[kMaxDevices] = {};

// Device address of the array on the current device (looked up once per device).
cudaError_t static_workspace(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mutex);
    if (g_ws_ptr[dev] == nullptr) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_ws);
        if (e != cudaSuccess) return e;
        g_ws_ptr[dev] = p;
    }
    *out = g_ws_ptr[dev];
    return cudaSuccess;
}

}  // namespace
}  // namespace memoroid

extern "C" memoroid_status_t memoroid_scan_diag_fwd_static(const void* lambda, int lambda_per_step,
                                                           const void* u, const uint8_t* start,
                                                           const void* h0, void* h, void* h_last,
                                                           int64_t B, int64_t L, int64_t D,
                                                           void* stream) {
    if (B < 0 || L < 0 || D < 0 || (D % 2) != 0) return MEMOROID_ERR_INVALID_ARG;
    const size_t need = memoroid_scan_diag_workspace_bytes(B, L, D);
    if (need > static_cast<size_t>(MEMOROID_STATIC_WORKSPACE_BYTES)) return MEMOROID_ERR_WORKSPACE;
    void* ws = nullptr;
    if (memoroid::static_workspace(&ws) != cudaSuccess) return MEMOROID_ERR_CUDA;
    return memoroid_scan_diag_fwd(lambda, lambda_per_step, u, start, h0, h, h_last, B, L, D, ws,
                                  static_cast<size_t>(MEMOROID_STATIC_WORKSPACE_BYTES), stream);
}

extern "C" memoroid_status_t memoroid_get_static_device_error(void* stream) {
    void* ws = nullptr;
    if (memoroid::static_workspace(&ws) != cudaSuccess) return MEMOROID_ERR_CUDA;
    return memoroid_get_device_error(ws, stream);
}
