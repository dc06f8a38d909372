// kernels_f64_bwd.cu -- instantiations of the sweep kernel for double, mode 1, sample
// groups of at least one warp (full-warp reductions).
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f64_bwd(int K) {
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<double, 1, 1, true, false>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<double, 2, 1, true, false>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<double, 3, 1, true, false>);
    default: return nullptr;
    }
}

}  // namespace vqc
