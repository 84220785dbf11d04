// gradlev_noalloc.cu -- a forward-scan entry point that needs no caller workspace.
//
// Some callers cannot allocate device memory at call time and cannot hand the
// library a workspace either: for example code that plugs into a host framework
// through a fixed "inputs, outputs, stream" signature, or a serving loop whose
// device memory budget is fixed once at start-up and owned by someone else.
// gradlev_forward_scan_noalloc serves them.  It runs the same forward scan as
// gradlev_forward_scan, with the kernel's scratch (work ticket, look-back flags
// and per-segment aggregates) placed in a fixed-size array that lives in this
// library's device image, so the call itself allocates nothing.
//
// The array costs GRADLEV_NOALLOC_SCRATCH_BYTES on every GPU that loads the
// library, for the life of the process.  All calls on a device share it and it
// keeps the previous call's contents; the scan clears the part that must start
// at zero (ticket, flags, error word) at the start of every call, on the
// caller's stream.  Calls that could overlap on the GPU (different streams, or
// different host threads on the same device without ordering) race on the
// array and must not be issued.
//
// A bounded device-side wait that expires leaves its error bit in the array's
// status word, as it would in a caller workspace; gradlev_forward_scan_noalloc_status
// reads it back.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/gradlev.h"

namespace gl {
size_t forward_workspace_bytes(const gradlev_desc* desc);
}

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[GRADLEV_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

// Device address of the array on the current device.  Host code cannot use the
// symbol itself (on the host it names a stand-in, not device memory), so the
// address is looked up once per device, with that device current, and cached.
// The cache outlives a cudaDeviceReset, after which the address is stale: the
// entry point is not for processes that reset a device they have called it on.
void* scratch_on_current_device() {
    static void* addr[kMaxDevices] = {};
    static std::mutex mu;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    std::lock_guard<std::mutex> g(mu);
    if (!addr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
        addr[dev] = p;
    }
    return addr[dev];
}

}  // namespace

extern "C" int gradlev_forward_scan_noalloc(const gradlev_desc* desc, const gradlev_tensor* x,
                                            const gradlev_tensor* g_hat, const float* W0,
                                            float eta, int act, const gradlev_tensor* y,
                                            const gradlev_tensor* act_out,
                                            gradlev_stream_t stream) {
    // the forward scan's own need (gradlev_workspace_bytes is the larger of
    // both directions, which would reject forward shapes that fit)
    const size_t need = gl::forward_workspace_bytes(desc);
    if (need == 0) return GRADLEV_ERR_INVALID_ARG;
    if (need > (size_t)GRADLEV_NOALLOC_SCRATCH_BYTES) return GRADLEV_ERR_WORKSPACE;
    void* scratch = scratch_on_current_device();
    if (!scratch) return GRADLEV_ERR_CUDA;
    return gradlev_forward_scan(desc, x, g_hat, W0, eta, act, y, act_out, scratch,
                                (size_t)GRADLEV_NOALLOC_SCRATCH_BYTES, stream);
}

extern "C" int gradlev_forward_scan_noalloc_status(gradlev_stream_t stream) {
    // Word 1 of the scratch is the status word the kernels set when a bounded
    // wait expires (the same layout as a caller workspace).
    unsigned int word = 0;
    if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    if (cudaMemcpyFromSymbol(&word, g_noalloc_scratch, sizeof(word), sizeof(unsigned int),
                             cudaMemcpyDeviceToHost) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    return word == 0 ? GRADLEV_OK : GRADLEV_ERR_TIMEOUT;
}
