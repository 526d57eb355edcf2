// lrar_noalloc.cu -- lrar_backward_noalloc: the backward pass for callers that
// cannot allocate device memory.
//
// lrar_backward needs a caller-provided workspace for the per-CTA partial sums
// of dq.  Some callers have no way to provide one at call time: plugin
// callbacks of inference or training runtimes that are forbidden to allocate
// while they run, services that must stay inside a fixed device-memory budget,
// and C hosts that only ever receive device pointers from another component
// and have no device allocator of their own.  This entry point serves them:
// its scratch is a fixed array compiled into the library, so the call itself
// allocates nothing (no cudaMalloc, no cudaFree, no allocating library call).
//
// Costs and rules:
//   * every GPU that loads the library holds kScratchBytes (4 MiB) for the
//     scratch until the process exits, whether or not the call is used;
//   * problems whose workspace would exceed kScratchBytes are rejected with
//     LRAR_ERR_UNSUPPORTED (lrar_backward_workspace_size() <= 4 MiB, i.e. a
//     dq width -- r, or d for full keys -- of at most 1024);
//   * all calls on a device share the one array.  Nothing in it needs to start
//     at zero (each CTA overwrites its own row of partial sums before the
//     reduction reads it), but calls that may run at the same time on the GPU
//     (on different streams, or issued by different host threads without
//     ordering) race on it and must be serialised by the caller;
//   * the first call on each device that gets past the argument checks looks
//     up the array's device address (cudaGetSymbolAddress) with that device
//     current and keeps it for the life of the process; make that first call
//     before any stream capture.  A reset of the device or of its primary
//     context (cudaDeviceReset) unloads the library's device code and leaves
//     the kept address stale, so the call must not be used on a device after
//     such a reset.
#include <mutex>

#include "lrar.h"
#include "lrar_device.cuh"
#include "lrar_launch.h"

#define LRAR_API extern "C" __attribute__((visibility("default")))

namespace {

constexpr size_t kScratchBytes = size_t(4) << 20;
constexpr int kMaxDevices = 64;

// The scratch itself.  In host code `g_scratch` names a host-side stand-in,
// not device memory, so host code must never pass it to a kernel directly;
// scratch_address() returns the real device address.
static __device__ __align__(256) float g_scratch[kScratchBytes / sizeof(float)];

std::mutex g_mu;
void *g_address[kMaxDevices];  // device address of g_scratch on each device, once looked up

// Device address of the scratch on the current device (looked up on first use).
int scratch_address(void **out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return lrar::record_error(LRAR_ERR_CUDA, "lrar_backward_noalloc: cudaGetDevice failed");
    if (dev < 0 || dev >= kMaxDevices)
        return lrar::record_error(LRAR_ERR_UNSUPPORTED, "lrar_backward_noalloc: device index out of range");
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_address[dev] == nullptr) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_scratch);
        if (e != cudaSuccess || p == nullptr)
            return lrar::record_error(LRAR_ERR_CUDA, "lrar_backward_noalloc: cudaGetSymbolAddress failed");
        g_address[dev] = p;
    }
    *out = g_address[dev];
    return LRAR_OK;
}

}  // namespace

LRAR_API int lrar_backward_noalloc(int variant, int in_dtype, int grad_dtype, const void *values, const void *keys,
                                   const float *query, int n_src, int64_t T, int d, int r, float eps, const void *dh,
                                   const void *h, int h_dtype, const float *lse, void *dvalues, void *dkeys,
                                   float *dq, int accumulate, int *status, void *stream) {
    // lrar_backward's own checks first, so that a bad argument gets its code and
    // message without touching the device
    int rc = lrar::check_backward(variant, in_dtype, grad_dtype, values, keys, query, n_src, T, d, r, eps, dh, h,
                                  h_dtype, lse, dvalues, dkeys, dq, accumulate, status);
    if (rc != LRAR_OK) return rc;
    if (T == 0)  // nothing to reduce: lrar_backward only sets dq (no workspace involved)
        return lrar_backward(variant, in_dtype, grad_dtype, values, keys, query, n_src, T, d, r, eps, dh, h, h_dtype,
                             lse, dvalues, dkeys, dq, accumulate, nullptr, 0, status, stream);
    const size_t need = lrar_backward_workspace_size(variant, n_src, T, d, r);
    if (need > kScratchBytes)
        return lrar::record_error(LRAR_ERR_UNSUPPORTED,
                                  "lrar_backward_noalloc: needs more scratch than its fixed 4 MiB (dq width > 1024); "
                                  "use lrar_backward with a workspace");
    void *scratch = nullptr;
    if ((rc = scratch_address(&scratch)) != LRAR_OK) return rc;
    return lrar_backward(variant, in_dtype, grad_dtype, values, keys, query, n_src, T, d, r, eps, dh, h, h_dtype, lse,
                         dvalues, dkeys, dq, accumulate, scratch, kScratchBytes, status, stream);
}
