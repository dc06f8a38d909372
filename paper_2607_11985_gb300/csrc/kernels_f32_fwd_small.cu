// kernels_f32_fwd_small.cu -- instantiations of the sweep kernel for float, mode 0, sample
// groups of fewer than 32 threads (small circuits or large blocks).
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f32_fwd_small(int K) {
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<float, 1, 0, false, false>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<float, 2, 0, false, false>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<float, 3, 0, false, false>);
    case 4: return reinterpret_cast<const void*>(&sweep_kernel<float, 4, 0, false, false>);
    case 5: return reinterpret_cast<const void*>(&sweep_kernel<float, 5, 0, false, false>);
    default: return nullptr;
    }
}

}  // namespace vqc
