// kernels_dd_hbm.cu -- double-float (complex128 storage) instantiations of the
// HBM-tiled pass kernels (K = 4 forward, 3 backward, as complex128), of the
// per-sample tables and gradient-term reduction and of the cluster-path forward
// (K = 4).
#include "cluster.cuh"
#include "kernels.h"
#include "pass.cuh"

namespace vqc {

const void* pass_ptr_dd(int mode, int K, bool full) {
    if (mode == 0 && K == 4) return full ? reinterpret_cast<const void*>(&pass_kernel<dd, 4, 0, true>)
                                         : reinterpret_cast<const void*>(&pass_kernel<dd, 4, 0, false>);
    if (mode == 1 && K == 3) return full ? reinterpret_cast<const void*>(&pass_kernel<dd, 3, 1, true>)
                                         : reinterpret_cast<const void*>(&pass_kernel<dd, 3, 1, false>);
    return nullptr;
}

const void* cluster_ptr_dd() { return reinterpret_cast<const void*>(&cluster_fwd_kernel<dd, 4>); }
const void* reduce_terms_ptr_dd() { return reinterpret_cast<const void*>(&reduce_terms<dd>); }
const void* ps_tables_ptr_dd() { return reinterpret_cast<const void*>(&ps_tables<dd>); }

}  // namespace vqc
