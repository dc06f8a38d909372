// kernels_f32_bwd.cu -- instantiations of the sweep kernel for float, mode 1, sample
// groups of at least one warp (full-warp reductions).
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f32_bwd(int K) {
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<float, 1, 1, true, false>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<float, 2, 1, true, false>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<float, 3, 1, true, false>);
    case 4: return reinterpret_cast<const void*>(&sweep_kernel<float, 4, 1, true, false>);
    default: return nullptr;
    }
}

}  // namespace vqc
