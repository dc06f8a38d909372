// kernels_f32_fwd.cu -- instantiations of the sweep kernel for float, mode 0, sample
// groups of at least one warp (full-warp reductions).
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f32_fwd(int K) {
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<float, 1, 0, true, false>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<float, 2, 0, true, false>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<float, 3, 0, true, false>);
    case 4: return reinterpret_cast<const void*>(&sweep_kernel<float, 4, 0, true, false>);
    case 5: return reinterpret_cast<const void*>(&sweep_kernel<float, 5, 0, true, false>);
    default: return nullptr;
    }
}

}  // namespace vqc
