// kernels_dd_fused.cu -- instantiations of the FUSED backward (it sweeps
// forward itself and writes E; vqc_forward_backward) with double-float
// arithmetic (complex128 storage), full-warp and sub-warp sample groups.
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_dd_fused(int K, bool full) {
    if (full) {
        switch (K) {
        case 1: return reinterpret_cast<const void*>(&sweep_kernel<dd, 1, 1, true, true>);
        case 2: return reinterpret_cast<const void*>(&sweep_kernel<dd, 2, 1, true, true>);
        case 3: return reinterpret_cast<const void*>(&sweep_kernel<dd, 3, 1, true, true>);
        default: return nullptr;
        }
    }
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<dd, 1, 1, false, true>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<dd, 2, 1, false, true>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<dd, 3, 1, false, true>);
    default: return nullptr;
    }
}

}  // namespace vqc
