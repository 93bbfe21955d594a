// noalloc.cu -- dge_score_noalloc: dge_score with scratch the library owns.
//
// For callers that may not allocate device memory at all (a serving runtime
// that owns the device-memory plan, or code that must not risk the device-wide
// synchronisation of cudaMalloc / cudaFree), the scoring scratch lives in one
// file-scope device array instead of a caller workspace.  Nothing here
// allocates: the array is part of the library's device image.
#include <stdio.h>

#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace {

constexpr size_t kScratchBytes = DGE_NOALLOC_SCRATCH_BYTES;

// The scratch itself.  In host code this name is only a handle for the
// runtime's symbol lookup, never an address to hand to a kernel.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_scratch_addr[kMaxDevices];  // device address of g_noalloc_scratch, per device

// Device address of the scratch on the current device, looked up once per device (the
// header asks callers not to use the entry point across a device reset).  With lookup
// false, only an address already looked up is returned.
int scratch_on_current_device(void **out, bool lookup = true)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        char msg[160];
        snprintf(msg, sizeof msg, "dge_score_noalloc: cudaGetDevice: %s", cudaGetErrorName(e));
        dge::record_error_text(msg);
        return DGE_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices)
        return DGE_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch_addr[dev]) {
        if (!lookup)
            return DGE_ERR_INVALID_ARG;
        void *ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
        if (e != cudaSuccess || !ptr) {
            char msg[160];
            snprintf(msg, sizeof msg, "dge_score_noalloc: cudaGetSymbolAddress: %s",
                     cudaGetErrorName(e));
            dge::record_error_text(msg);
            return DGE_ERR_CUDA;
        }
        g_scratch_addr[dev] = ptr;
    }
    *out = g_scratch_addr[dev];
    return DGE_OK;
}

}  // namespace

extern "C" int dge_score_noalloc(const dge_problem *p, const dge_buffers *bufs, void *stream)
{
    size_t need = 0;
    int rc = dge_workspace_size(p, &need);
    if (rc != DGE_OK)
        return rc;
    if (need > kScratchBytes) {
        char msg[200];
        snprintf(msg, sizeof msg,
                 "dge_score_noalloc: problem needs %zu bytes of scratch, the built-in buffer "
                 "holds %zu",
                 need, kScratchBytes);
        dge::record_error_text(msg);
        return DGE_ERR_WORKSPACE_TOO_SMALL;
    }
    void *scratch = nullptr;
    if ((rc = scratch_on_current_device(&scratch)) != DGE_OK)
        return rc;
    return dge_score(p, bufs, scratch, kScratchBytes, stream);
}

// The status word at the start of the scratch (the first 4 bytes of a workspace are the
// status word for every scoring call), read, cleared and returned like a caller's.
extern "C" int dge_noalloc_status(void *stream)
{
    void *scratch = nullptr;
    const int rc = scratch_on_current_device(&scratch, false);
    if (rc != DGE_OK)
        return rc;
    return dge_get_device_status(scratch, stream);
}
