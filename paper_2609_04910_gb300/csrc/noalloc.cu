// gauss_sum_noalloc: the forward Gauss sum with its scratch memory in a
// fixed, statically sized device array instead of a per-call allocation.
//
// Some callers cannot allocate device memory at the point where they need
// the sum: code running inside a framework that owns every allocation (a
// custom allocator or memory pool the library must not bypass), code that
// has reserved all remaining device memory up front, or code on a path
// where an allocation call would synchronise or fail.  For them this entry
// point reuses the normal kernels with a workspace that the library already
// holds: a file-scope __device__ array of GS_NOALLOC_SCRATCH_BYTES bytes,
// which every GPU that loads the library keeps until the process exits.
//
// Rules of use:
//  * The caller passes inputs and outputs exactly as for gauss_sum (device
//    pointers, default options: centring on, automatic key splits).
//  * Calls whose workspace would exceed the static array are rejected with
//    GS_ERR_UNSUPPORTED before any GPU work is issued.
//  * The first call on a device looks up the device address of the array
//    (cudaGetSymbolAddress, with that device current) and keeps it for the
//    life of the process; make that first call before any stream capture
//    begins.  The kept address assumes the device's primary context is never
//    reset: after cudaDeviceReset it is stale (as is the device status word's
//    address that api.cu keeps), so a process that resets a device must not
//    call the library on it again.
//  * All calls on a device share the one array and leave their data in it.
//    Calls whose GPU work overlaps (different streams without ordering, or
//    several host threads) race on it and give wrong results; order them.
//  * Nothing in the array has to start at zero: each call writes every
//    scratch value it reads (the one accumulator that needs zeroing is
//    cleared by the call itself).
//  * Neither this entry point nor the kernels it runs call cudaMalloc,
//    cudaMallocAsync, cudaFree or any allocating library routine.
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "gauss_sum.h"
#include "internal.h"

namespace {

// 1-KiB aligned (the workspace layout aligns its parts to 1 KiB).
static __device__ __align__(1024) unsigned char g_noalloc_scratch[GS_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of the static scratch array on the current device.
cudaError_t scratch_for_current_device(void** ptr) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *ptr = g_scratch_ptr[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" gs_status gauss_sum_noalloc(const void* q, const void* k, const void* v, double tau,
                                       int64_t M, int64_t N, int64_t D, int64_t C,
                                       gs_dtype dtype, float* out, void* stream) {
    size_t need = 0;
    gs_status st = gs::forward_workspace_bytes(q, k, v, tau, M, N, D, C, dtype, out, &need);
    if (st != GS_OK) return st;
    if (need > static_cast<size_t>(GS_NOALLOC_SCRATCH_BYTES)) {
        char msg[200];
        std::snprintf(msg, sizeof(msg),
                      "gauss_sum_noalloc: this call needs %zu bytes of scratch, the static "
                      "scratch array holds %zu bytes",
                      need, static_cast<size_t>(GS_NOALLOC_SCRATCH_BYTES));
        return gs::set_last_error(GS_ERR_UNSUPPORTED, msg);
    }
    void* scratch = nullptr;
    cudaError_t e = scratch_for_current_device(&scratch);
    if (e != cudaSuccess) {
        char msg[200];
        std::snprintf(msg, sizeof(msg), "gauss_sum_noalloc: cudaGetSymbolAddress failed: %s",
                      cudaGetErrorString(e));
        return gs::set_last_error(GS_ERR_CUDA, msg);
    }
    gs_options opt;
    gauss_sum_default_options(&opt);
    opt.workspace = scratch;
    opt.workspace_bytes = static_cast<size_t>(GS_NOALLOC_SCRATCH_BYTES);
    return gauss_sum_ex(q, k, v, tau, M, N, D, C, dtype, out, stream, &opt);
}
