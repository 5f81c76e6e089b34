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

#include <cuda_runtime.h>

#include "vsd.h"

// The scratch, one copy per device.  Host code must not use this name as a
// device address; it uses the address cudaGetSymbolAddress returns instead.
static __device__ __align__(256) unsigned char g_noalloc_scratch[VSD_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 256;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices];  // device address of g_noalloc_scratch, per device

// Device address of the scratch on the current device.  The first call on a
// device looks it up (with that device current) and caches it.
vsd_status scratch_on_current_device(void** out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return VSD_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return VSD_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_scratch_ptr[dev] == nullptr) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || p == nullptr) return VSD_ERR_CUDA;
        g_scratch_ptr[dev] = p;
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
