// static_scratch.cu -- wino_step for callers that cannot allocate device memory.
//
// Some callers have no way to hand this library a workspace: an inference
// server plugin that is given only its input and output buffers, a process
// whose memory pool owns all device memory, or a decode loop that must not
// call cudaMalloc / cudaFree once it is running (both synchronise the
// device).  For them, wino_step_static_scratch runs the same kernels as
// wino_step with the workspace taken from a fixed array in device memory that
// belongs to this library (WINO_STATIC_SCRATCH_BYTES, reserved on every GPU
// that loads the library, until the process exits).  Nothing is allocated
// per call.
#include <mutex>

#include "internal.h"

namespace wino {
namespace {

// The scratch every call of wino_step_static_scratch on a device shares.
static __device__ __align__(256) unsigned char g_static_scratch[WINO_STATIC_SCRATCH_BYTES];

// In host code g_static_scratch only names the array; its device address is looked up with the device
// current, on every call (a cheap table lookup once the module is loaded), so that a module reloaded
// after cudaDeviceReset is never reached through a stale address.  The first call that sees an address
// (per device) also clears the status words at the start of the array on the caller's stream, which the
// kernels expect to find zeroed before their first use.
int scratch_address(cudaStream_t stream, void **out)
{
    static std::mutex mu;
    static void *seen[64];
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
        return WINO_ERR_CUDA;
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p)
        return WINO_ERR_CUDA;
    std::lock_guard<std::mutex> g(mu);
    if (seen[dev] != p) {
        if (cudaMemsetAsync(p, 0, 256, stream) != cudaSuccess)
            return WINO_ERR_CUDA;
        seen[dev] = p;
    }
    *out = p;
    return WINO_OK;
}

}  // namespace
}  // namespace wino

extern "C" int wino_step_static_scratch(const uint16_t *H, const uint16_t *W, int64_t d, int64_t V, int32_t *tokens,
                                        const wino_params *p, int32_t *counts, int8_t *flags, void *stream)
{
    if (!p)
        return WINO_ERR_ARG;
    size_t need = 0;
    const int rc = wino_workspace_size_step(p, d, V, &need);
    if (rc != WINO_OK)
        return rc;
    if (need > WINO_STATIC_SCRATCH_BYTES)
        return WINO_ERR_WORKSPACE;  // the problem needs more scratch than the fixed array holds
    void *scratch = nullptr;
    const int rs = wino::scratch_address(static_cast<cudaStream_t>(stream), &scratch);
    if (rs != WINO_OK)
        return rs;
    return wino_step(H, W, d, V, tokens, p, counts, flags, scratch, WINO_STATIC_SCRATCH_BYTES, stream);
}
