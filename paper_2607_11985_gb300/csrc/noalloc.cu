// noalloc.cu -- vqc_backward_noalloc: the adjoint backward for callers that
// cannot allocate device memory.
//
// vqc_backward needs a caller-provided workspace (a 256-byte control block
// plus one dw partial per CTA).  Some callers cannot obtain one: a plugin whose
// host application owns all device memory, a real-time loop that must not pay
// cudaMalloc's latency or its implicit device synchronisation, or code that runs
// under a fixed, pre-planned device-memory budget.  This entry point takes the
// same inputs and outputs but keeps its scratch in a fixed-size array in device
// memory that is part of the loaded library (VQC_NOALLOC_SCRATCH_BYTES per GPU,
// held until the process exits).  It calls no cudaMalloc, cudaFree or
// allocating library routine.
//
// All calls on a device share that one array, and it keeps the previous call's
// contents: each call clears the control block (the CTA-completion counter)
// before its launch.  Calls whose kernels overlap on the GPU race on the array,
// so callers must order them (e.g. on one stream).
//
// The device address of the array is looked up once per device, on the first
// call made while that device is current (cudaGetSymbolAddress); make that first
// call before any CUDA stream capture begins.  The cached address belongs to the
// device's primary context (the one the CUDA runtime uses): the entry point
// assumes callers stay in it and do not reset the device (cudaDeviceReset)
// while the library is loaded; after a reset the cached address is stale.
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "engine.h"

namespace vqc {
// Implemented in capi.cu: the backward launch with an explicit scratch buffer.
vqc_status backward_with_scratch(const vqc_plan* plan, int32_t batch, const void* x,
                                 const void* w, const void* psi0, const void* psi_final,
                                 const void* grad_expz, void* grad_x, void* grad_w, void* scratch,
                                 size_t scratch_bytes, void* stream, bool clear_control);
vqc_status set_error(vqc_status s, const std::string& msg);
}  // namespace vqc

// File-scope scratch: one copy per GPU that loads this library.
static __device__ __align__(256) unsigned char vqc_noalloc_scratch[VQC_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (host code cannot
// use the symbol itself: on the host it is only a stand-in, not a device
// address).
vqc_status scratch_address(void** out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return vqc::set_error(VQC_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices)
        return vqc::set_error(VQC_ERR_UNSUPPORTED, "device ordinal beyond the scratch table");
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, vqc_noalloc_scratch);
        if (e != cudaSuccess || !p)
            return vqc::set_error(VQC_ERR_CUDA, std::string("cudaGetSymbolAddress(scratch): ") +
                                                    cudaGetErrorString(e));
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return VQC_OK;
}

}  // namespace

extern "C" vqc_status vqc_backward_noalloc(const vqc_plan* plan, int32_t batch, const void* x,
                                           const void* w, const void* psi0, const void* psi_final,
                                           const void* grad_expz, void* grad_x, void* grad_w,
                                           void* stream) {
    try {
        void* scratch = nullptr;
        vqc_status st = scratch_address(&scratch);
        if (st != VQC_OK) return st;
        return vqc::backward_with_scratch(plan, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                          grad_w, scratch, VQC_NOALLOC_SCRATCH_BYTES, stream, true);
    } catch (...) {
        return vqc::set_error(VQC_ERR_INVALID_ARG, "internal error in vqc_backward_noalloc");
    }
}
