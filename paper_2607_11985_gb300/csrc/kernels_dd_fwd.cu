// kernels_dd_fwd.cu -- instantiations of the sweep kernel with double-float
// arithmetic (complex128 storage), mode 0: full-warp and sub-warp sample groups.
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_dd_fwd(int K, bool full) {
    if (full) {
        switch (K) {
        case 1: return reinterpret_cast<const void*>(&sweep_kernel<dd, 1, 0, true, false>);
        case 2: return reinterpret_cast<const void*>(&sweep_kernel<dd, 2, 0, true, false>);
        case 3: return reinterpret_cast<const void*>(&sweep_kernel<dd, 3, 0, true, false>);
        case 4: return reinterpret_cast<const void*>(&sweep_kernel<dd, 4, 0, true, false>);
        default: return nullptr;
        }
    }
    switch (K) {
    case 1: return reinterpret_cast<const void*>(&sweep_kernel<dd, 1, 0, false, false>);
    case 2: return reinterpret_cast<const void*>(&sweep_kernel<dd, 2, 0, false, false>);
    case 3: return reinterpret_cast<const void*>(&sweep_kernel<dd, 3, 0, false, false>);
    case 4: return reinterpret_cast<const void*>(&sweep_kernel<dd, 4, 0, false, false>);
    default: return nullptr;
    }
}

}  // namespace vqc
