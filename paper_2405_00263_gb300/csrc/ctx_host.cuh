// Host-side identity of the calling thread's current CUDA context, reached
// through the runtime's driver entry-point query (the library does not link
// libcuda).  Per-context state (a kernel's shared-memory attribute, a device
// symbol's address) is keyed on this id rather than on the device ordinal:
// after cudaDeviceReset, or under a non-primary context on the same device,
// a device ordinal names a different context whose module state starts anew.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace clover {

using CtxGetCurrentFn = CUresult (*)(CUcontext *);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long *);

template <typename Fn>
inline Fn driver_fn(const char *name) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion(name, &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
        return nullptr;
    return reinterpret_cast<Fn>(p);
}

// Unique id of the current context, plus one (cuCtxGetId: ids are never
// reused within a process).  A thread with no current context first gets the
// current device's primary context, as the runtime's next call would bind it
// anyway (cudaSetDevice does this without allocating).  Returns 0 when no
// context can be made current.
inline unsigned long long current_context_id() {
    static const CtxGetCurrentFn get_current = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent");
    static const CtxGetIdFn get_id = driver_fn<CtxGetIdFn>("cuCtxGetId");
    if (!get_current || !get_id) return 0;
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) {
        // no context bound to this thread yet: bind the device's primary one
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || cudaSetDevice(dev) != cudaSuccess) return 0;
        if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
    }
    unsigned long long id = 0;
    if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id + 1;   // 0 stays "unknown"
}

}  // namespace clover
