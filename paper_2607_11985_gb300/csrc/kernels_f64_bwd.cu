// kernels_f64_bwd.cu -- instantiations of the sweep kernel for double, mode 1.
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f64_bwd(int K) {
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<double, 1, 1>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<double, 2, 1>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<double, 3, 1>);
    default: return nullptr;
    }
}

}  // namespace vqc
