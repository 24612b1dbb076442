// Patch cut that allocates nothing (emtk_extract_patches_static).
//
// Who needs it: callers that cannot call cudaMalloc.  Examples are a process
// whose device memory is already owned by another allocator, such as a
// framework's caching pool or a budget fixed at start-up, so that a new
// allocation fails or is not allowed, and code that must not pay for the
// device-wide synchronisation that cudaMalloc / cudaFree can cause.  Such a
// caller cannot create an emtk context either, because creating one
// allocates the weights and the workspace, so this entry point needs no
// context at all.
//
// The only scratch the patch cut needs is the time-interval image of the
// plane.  Here it lives in a file-scope device array of fixed size.  Every
// GPU that loads the library holds the array until the process exits.  Each
// call writes every interval it later reads, so nothing has to be cleared
// between calls.  All calls share the one array: calls that overlap on the
// GPU (on two streams, or two host threads) race and must be serialised by
// the caller.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "emtk_internal.h"

namespace emtk {
namespace {

constexpr size_t kStaticScratchBytes = EMTK_STATIC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_interval_scratch[kStaticScratchBytes];

// The array's device address belongs to the device's context: a context that
// is destroyed and created again (cudaDeviceReset, a framework resetting the
// device) may load the library's module at another address.  So the address
// is kept together with the unique id of the context it was looked up in,
// and looked up again when the current context is another one.
struct ScratchSlot {
    unsigned long long ctx_id;
    void *addr;
};
std::mutex g_scratch_mutex;
ScratchSlot g_scratch_slot[kMaxDevices];
PFN_cuCtxGetCurrent_v4000 g_ctx_get_current = nullptr;
PFN_cuCtxGetId_v12000 g_ctx_get_id = nullptr;

// Resolves the two driver calls once (through the runtime, so the library
// needs no link against the driver library).
bool resolve_driver_calls() {
    if (g_ctx_get_current && g_ctx_get_id) return true;
    void *a = nullptr, *b = nullptr;
    cudaDriverEntryPointQueryResult qa, qb;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &a, 4000, cudaEnableDefault, &qa) != cudaSuccess ||
        cudaGetDriverEntryPointByVersion("cuCtxGetId", &b, 12000, cudaEnableDefault, &qb) != cudaSuccess ||
        qa != cudaDriverEntryPointSuccess || qb != cudaDriverEntryPointSuccess || !a || !b)
        return false;
    g_ctx_get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(a);
    g_ctx_get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(b);
    return true;
}

// The array's device address in the current context of `device` (the
// caller's current device).  Looked up with cudaGetSymbolAddress the first
// time a context is seen; in host code the name g_interval_scratch is only a
// host-side stand-in, never a device address.
cudaError_t scratch_address(int device, void **out) {
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!resolve_driver_calls()) return cudaErrorNotSupported;
    CUcontext ctx = nullptr;
    if (g_ctx_get_current(&ctx) != CUDA_SUCCESS) return cudaErrorInitializationError;
    if (ctx == nullptr) {  // no context bound to this thread yet: bind the device's primary one
        const cudaError_t e = cudaSetDevice(device);
        if (e != cudaSuccess) return e;
        if (g_ctx_get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return cudaErrorInitializationError;
    }
    unsigned long long id = 0;
    if (g_ctx_get_id(ctx, &id) != CUDA_SUCCESS) return cudaErrorInitializationError;
    ScratchSlot &slot = g_scratch_slot[device];
    if (slot.addr == nullptr || slot.ctx_id != id) {
        void *p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_interval_scratch);
        if (e != cudaSuccess) return e;
        slot.addr = p;
        slot.ctx_id = id;
    }
    *out = slot.addr;
    return cudaSuccess;
}

}  // namespace
}  // namespace emtk

extern "C" emtk_status emtk_extract_patches_static(const float *d_adc, int32_t nwires, int32_t nticks, int64_t ld,
                                                   const emtk_hit *d_hits, int32_t nhits, void *d_patches,
                                                   emtk_patch_format fmt, emtk_stream stream) {
    using namespace emtk;
    if (fmt != EMTK_PATCH_F32 && fmt != EMTK_PATCH_BF16 && fmt != EMTK_PATCH_F16) return EMTK_ERR_ARG;
    if (nwires < 0 || nticks < 0 || nhits < 0 || ld < nticks) return EMTK_ERR_ARG;
    if (nhits == 0) return EMTK_OK;
    if (d_adc == nullptr || d_hits == nullptr || d_patches == nullptr) return EMTK_ERR_ARG;
    if ((reinterpret_cast<uintptr_t>(d_adc) & 15u) != 0 || (ld % 4) != 0) return EMTK_ERR_ALIGN;
    if ((reinterpret_cast<uintptr_t>(d_hits) & 7u) != 0) return EMTK_ERR_ALIGN;
    if ((reinterpret_cast<uintptr_t>(d_patches) & 15u) != 0) return EMTK_ERR_ALIGN;

    const int32_t nint = nticks / kDs;
    const int32_t pitch = (nint + 7) / 8 * 8;
    const uint64_t elem = fmt == EMTK_PATCH_F32 ? 4u : 2u;
    if ((uint64_t)nwires * (uint64_t)pitch * elem > kStaticScratchBytes) return EMTK_ERR_ARG;  // plane too large

    int device = 0;
    if (cudaGetDevice(&device) != cudaSuccess) return EMTK_ERR_CUDA;
    if (device < 0 || device >= kMaxDevices) return EMTK_ERR_UNSUPPORTED;
    void *img = nullptr;
    if (scratch_address(device, &img) != cudaSuccess) return EMTK_ERR_CUDA;

    ReqTable t;  // on the host stack: a kernel parameter, not an allocation
    t.n = 1;
    t.pad = 0;
    ReqDesc &d = t.r[0];
    d.adc = d_adc;
    d.hits = d_hits;
    d.scores = nullptr;
    d.ld = ld;
    d.hit_begin = 0;
    d.d_off = 0;
    d.nwires = nwires;
    d.nticks = nticks;
    d.nhits = nhits;
    d.nint = nint;
    d.pitch = pitch;
    d.halo = 0;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (launch_interval_images(t, img, fmt, s) != cudaSuccess) return EMTK_ERR_CUDA;
    if (launch_gather(t, img, fmt, 0, nhits, d_patches, nullptr, 0, s) != cudaSuccess) return EMTK_ERR_CUDA;
    return EMTK_OK;
}
