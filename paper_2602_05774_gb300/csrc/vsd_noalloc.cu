// vsd_noalloc.cu -- vsd_estep_mstep_noalloc: the fused E-step + M-step for
// callers that cannot hand the library any device scratch memory.
//
// Some callers have no way to allocate device memory at the point where they
// call this library: a plugin reached through a C interface that is given
// only its input and output pointers, a process whose device memory is wholly
// reserved by another allocator, or a latency-critical loop in which a
// cudaMalloc/cudaFree would synchronise the device.  For them the scratch that
// vsd_estep_mstep normally takes from the caller lives in a fixed array in
// device memory owned by this library.  Every GPU that loads the library keeps
// that array (VSD_NOALLOC_SCRATCH_BYTES) until the process exits.
#include <mutex>

#include <cuda.h>
#include <cuda_runtime.h>

#include "vsd.h"

// The scratch, one copy per device.  Host code must not use this name as a
// device address; it uses the address cudaGetSymbolAddress returns instead.
static __device__ __align__(256) unsigned char g_noalloc_scratch[VSD_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 256;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices];          // device address of g_noalloc_scratch, per device
unsigned long long g_scratch_ctx[kMaxDevices];  // id of the context it was looked up in

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

// The unique id of the calling thread's current context (0 if it cannot be
// read), through the runtime's driver entry points.
unsigned long long current_context_id() {
    static std::once_flag once;
    static CtxGetCurrentFn get_current = nullptr;
    static CtxGetIdFn get_id = nullptr;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess && q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<CtxGetCurrentFn>(p);
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<CtxGetIdFn>(p);
    });
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx) return 0;
    if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of the scratch on the current device.  The first call on a
// device looks it up (with that device current) and caches it; the lookup is
// repeated when the device's context has changed since (after a
// cudaDeviceReset the array lives at a new address in a new context).
vsd_status scratch_on_current_device(void** out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return VSD_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return VSD_ERR_UNSUPPORTED;
    // makes the context current (cudaGetSymbolAddress would too) before its id is read
    if (cudaFree(nullptr) != cudaSuccess) return VSD_ERR_CUDA;
    const unsigned long long ctx = current_context_id();
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_scratch_ptr[dev] == nullptr || ctx == 0 || ctx != g_scratch_ctx[dev]) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || p == nullptr) return VSD_ERR_CUDA;
        g_scratch_ptr[dev] = p;
        g_scratch_ctx[dev] = ctx;
    }
    *out = g_scratch_ptr[dev];
    return VSD_OK;
}

}  // namespace

extern "C" vsd_status vsd_estep_mstep_noalloc(const void* draft, const void* target,
                                              vsd_dtype dtype, vsd_layout layout, float T,
                                              const float* u_draft, const float* u_accept,
                                              const float* u_correct, const float* ref_logkappa,
                                              const vsd_params* params, vsd_linear_outputs* out,
                                              void* stream) {
    const size_t need = vsd_workspace_bytes(layout);
    if (need == 0) return VSD_ERR_INVALID_ARG;
    if (need > (size_t)VSD_NOALLOC_SCRATCH_BYTES) return VSD_ERR_TOO_LARGE;
    void* scratch = nullptr;
    const vsd_status st = scratch_on_current_device(&scratch);
    if (st != VSD_OK) return st;
    // The fused call clears the counters it needs at the start of every call,
    // so what an earlier call left in the scratch does not matter.
    return vsd_estep_mstep(draft, target, dtype, layout, T, u_draft, u_accept, u_correct,
                           ref_logkappa, params, out, scratch, (size_t)VSD_NOALLOC_SCRATCH_BYTES,
                           stream);
}

extern "C" vsd_status vsd_noalloc_device_status(void* stream, int32_t* status_bits) {
    if (!status_bits) return VSD_ERR_INVALID_ARG;
    void* scratch = nullptr;
    const vsd_status st = scratch_on_current_device(&scratch);
    if (st != VSD_OK) return st;
    // the status word is the first word of the scratch, as of any workspace
    return vsd_device_status(scratch, stream, status_bits);
}
