// kernels_f64_fwd_small.cu -- instantiations of the sweep kernel for double, mode 0, sample
// groups of fewer than 32 threads (small circuits or large blocks).
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f64_fwd_small(int K) {
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<double, 1, 0, false, false>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<double, 2, 0, false, false>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<double, 3, 0, false, false>);
    case 4: return reinterpret_cast<const void*>(&sweep_kernel<double, 4, 0, false, false>);
    default: return nullptr;
    }
}

}  // namespace vqc
