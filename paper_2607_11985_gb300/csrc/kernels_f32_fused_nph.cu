// kernels_f32_fused_nph.cu -- instantiations of the float forward+backward
// (fused) sweep kernel for plans without diagonal two-qubit phase ops (CRZ,
// RZZ): the switch has no phase cases, which frees registers (see apply_op).
#include "kernels.h"
#include "sweep.cuh"

namespace vqc {

const void* sweep_ptr_f32_fused_nph(int K, bool full) {
#define VQC_NPH(K_) \
    case K_: return full ? reinterpret_cast<const void*>(&sweep_kernel<float, K_, 1, true, true, false>) \
                         : reinterpret_cast<const void*>(&sweep_kernel<float, K_, 1, false, true, false>);
    switch (K) {
        VQC_NPH(1) VQC_NPH(2) VQC_NPH(3) VQC_NPH(4)
    default: return nullptr;
    }
#undef VQC_NPH
}

}  // namespace vqc
