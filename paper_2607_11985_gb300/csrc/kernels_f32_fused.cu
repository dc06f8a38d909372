// kernels_f32_fused.cu -- instantiations of the sweep kernel for float, mode 1
// with FUSED: the backward that sweeps forward itself and writes E
// (vqc_forward_backward), for full-warp and sub-warp sample groups.
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f32_fused(int K, bool full) {
    if (full) {
        switch (K) {
        case 1: return reinterpret_cast<const void*>(&sweep_kernel<float, 1, 1, true, true>);
        case 2: return reinterpret_cast<const void*>(&sweep_kernel<float, 2, 1, true, true>);
        case 3: return reinterpret_cast<const void*>(&sweep_kernel<float, 3, 1, true, true>);
        case 4: return reinterpret_cast<const void*>(&sweep_kernel<float, 4, 1, true, true>);
        default: return nullptr;
        }
    }
    if (!full) {
        switch (K) {
        case 1: return reinterpret_cast<const void*>(&sweep_kernel<float, 1, 1, false, true>);
        case 2: return reinterpret_cast<const void*>(&sweep_kernel<float, 2, 1, false, true>);
        case 3: return reinterpret_cast<const void*>(&sweep_kernel<float, 3, 1, false, true>);
        case 4: return reinterpret_cast<const void*>(&sweep_kernel<float, 4, 1, false, true>);
        default: return nullptr;
        }
    }
    return nullptr;
}

}  // namespace vqc
