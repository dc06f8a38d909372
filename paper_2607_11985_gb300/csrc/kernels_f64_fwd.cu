// kernels_f64_fwd.cu -- instantiations of the sweep kernel for double, mode 0, sample
// groups of at least one warp (full-warp reductions).
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f64_fwd(int K) {
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<double, 1, 0, true, false>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<double, 2, 0, true, false>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<double, 3, 0, true, false>);
    case 4: return reinterpret_cast<const void*>(&sweep_kernel<double, 4, 0, true, false>);
    default: return nullptr;
    }
}

}  // namespace vqc
