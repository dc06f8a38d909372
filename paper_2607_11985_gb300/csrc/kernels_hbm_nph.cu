// kernels_hbm_nph.cu -- the float forward pass kernel for plans without diagonal
// two-qubit phase ops (CRZ, RZZ): no phase cases in the switch (see apply_op).
// The backward pass kernel keeps them: without them its register allocation
// measured slower.
#include "kernels.h"
#include "pass.cuh"

namespace vqc {

const void* pass_ptr_f32_fwd_nph(int K, bool full) {
    if (K != 5) return nullptr;
    return full ? reinterpret_cast<const void*>(&pass_kernel<float, 5, 0, true, false>)
                : reinterpret_cast<const void*>(&pass_kernel<float, 5, 0, false, false>);
}

}  // namespace vqc
