// kernels_dd_bwd.cu -- instantiations of the sweep kernel with double-float
// arithmetic (complex128 storage), mode 1: full-warp and sub-warp sample groups.
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_dd_bwd(int K, bool full) {
    if (full) {
        switch (K) {
        case 1: return reinterpret_cast<const void*>(&sweep_kernel<dd, 1, 1, true, false>);
        case 2: return reinterpret_cast<const void*>(&sweep_kernel<dd, 2, 1, true, false>);
        case 3: return reinterpret_cast<const void*>(&sweep_kernel<dd, 3, 1, true, false>);
        default: return nullptr;
        }
    }
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<dd, 1, 1, false, false>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<dd, 2, 1, false, false>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<dd, 3, 1, false, false>);
    default: return nullptr;
    }
}

}  // namespace vqc
