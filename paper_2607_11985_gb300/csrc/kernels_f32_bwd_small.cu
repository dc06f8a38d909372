// kernels_f32_bwd_small.cu -- instantiations of the sweep kernel for float, mode 1, sample
// groups of fewer than 32 threads (small circuits or large blocks).
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f32_bwd_small(int K) {
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<float, 1, 1, false, false>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<float, 2, 1, false, false>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<float, 3, 1, false, false>);
    case 4: return reinterpret_cast<const void*>(&sweep_kernel<float, 4, 1, false, false>);
    default: return nullptr;
    }
}

}  // namespace vqc
