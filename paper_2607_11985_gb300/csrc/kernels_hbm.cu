// kernels_hbm.cu -- instantiations of the HBM-tiled pass kernels and the
// fixed-order partial reductions.
#include "kernels.h"
#include "pass.cuh"

namespace vqc {

const void* pass_ptr(bool dbl, int mode, int K, bool full) {
    if (!dbl) {
        if (mode == 0 && K == 5) return full ? reinterpret_cast<const void*>(&pass_kernel<float, 5, 0, true>)
                                             : reinterpret_cast<const void*>(&pass_kernel<float, 5, 0, false>);
        if (mode == 1 && K == 4) return full ? reinterpret_cast<const void*>(&pass_kernel<float, 4, 1, true>)
                                             : reinterpret_cast<const void*>(&pass_kernel<float, 4, 1, false>);
    } else {
        if (mode == 0 && K == 4) return full ? reinterpret_cast<const void*>(&pass_kernel<double, 4, 0, true>)
                                             : reinterpret_cast<const void*>(&pass_kernel<double, 4, 0, false>);
        if (mode == 1 && K == 3) return full ? reinterpret_cast<const void*>(&pass_kernel<double, 3, 1, true>)
                                             : reinterpret_cast<const void*>(&pass_kernel<double, 3, 1, false>);
    }
    return nullptr;
}

const void* reduce_expz_ptr(bool dbl) {
    return dbl ? reinterpret_cast<const void*>(&reduce_expz<double>)
               : reinterpret_cast<const void*>(&reduce_expz<float>);
}
const void* reduce_dx_ptr(bool dbl) {
    return dbl ? reinterpret_cast<const void*>(&reduce_dx<double>)
               : reinterpret_cast<const void*>(&reduce_dx<float>);
}
const void* reduce_cols_ptr(bool dbl) {
    return dbl ? reinterpret_cast<const void*>(&reduce_cols<double>)
               : reinterpret_cast<const void*>(&reduce_cols<float>);
}
const void* abs2_ptr(bool dbl) {
    return dbl ? reinterpret_cast<const void*>(&abs2_kernel<double>)
               : reinterpret_cast<const void*>(&abs2_kernel<float>);
}
const void* ps_tables_ptr(bool dbl) {
    return dbl ? reinterpret_cast<const void*>(&ps_tables<double>)
               : reinterpret_cast<const void*>(&ps_tables<float>);
}
const void* reduce_terms_ptr(bool dbl) {
    return dbl ? reinterpret_cast<const void*>(&reduce_terms<double>)
               : reinterpret_cast<const void*>(&reduce_terms<float>);
}
const void* reduce_dw_ptr(bool dbl) {
    return dbl ? reinterpret_cast<const void*>(&reduce_dw<double>)
               : reinterpret_cast<const void*>(&reduce_dw<float>);
}

}  // namespace vqc
