// Device and pinned-host allocations of the library, counted, with a
// host-side failure hook for tests (emtk_debug_fail_alloc).  Every
// cudaMalloc / cudaFree / cudaHostAlloc / cudaFreeHost of the library goes
// through these functions, so that a test can make any one allocation fail,
// as an exhausted device would, and then check that the entry point reported
// EMTK_ERR_OOM, that the context still works, and that nothing leaked (the
// live counts are back where they were).  Nothing here touches a kernel: the
// failure is made on the host, before the CUDA call.
#include <atomic>

#include "emtk_internal.h"

namespace emtk {
namespace {

// < 0: no failure armed; n >= 0: n more allocations succeed, the next fails
std::atomic<int64_t> g_fail_after{-1};
std::atomic<int64_t> g_live_device{0};
std::atomic<int64_t> g_live_host{0};

bool injected_failure() {
    int64_t c = g_fail_after.load();
    while (c >= 0) {
        if (g_fail_after.compare_exchange_weak(c, c - 1)) return c == 0;
    }
    return false;
}

}  // namespace

cudaError_t dev_alloc(void **p, size_t bytes) {
    *p = nullptr;
    if (injected_failure()) return cudaErrorMemoryAllocation;
    const cudaError_t e = cudaMalloc(p, bytes);
    if (e == cudaSuccess)
        g_live_device++;
    else
        *p = nullptr;
    return e;
}

cudaError_t dev_free(void *p) {
    if (p == nullptr) return cudaSuccess;
    const cudaError_t e = cudaFree(p);
    if (e == cudaSuccess) g_live_device--;
    return e;
}

cudaError_t host_alloc(void **p, size_t bytes) {
    *p = nullptr;
    if (injected_failure()) return cudaErrorMemoryAllocation;
    const cudaError_t e = cudaHostAlloc(p, bytes, cudaHostAllocDefault);
    if (e == cudaSuccess)
        g_live_host++;
    else
        *p = nullptr;
    return e;
}

cudaError_t host_free(void *p) {
    if (p == nullptr) return cudaSuccess;
    const cudaError_t e = cudaFreeHost(p);
    if (e == cudaSuccess) g_live_host--;
    return e;
}

}  // namespace emtk

extern "C" {

void emtk_debug_fail_alloc(int64_t after) { emtk::g_fail_after.store(after < 0 ? -1 : after); }

void emtk_debug_alloc_counts(int64_t *device, int64_t *host) {
    if (device) *device = emtk::g_live_device.load();
    if (host) *host = emtk::g_live_host.load();
}

}  // extern "C"
