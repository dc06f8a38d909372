// kernels_cluster_bwd.cu -- instantiations of the cluster-path backward kernel
// (complex64: K = 4, complex128: K = 3, double-float: K = 3).
#include "kernels.h"
#include "cluster.cuh"

namespace vqc {

const void* cluster_bwd_ptr(bool dbl, bool dfloat) {
    if (dfloat) return reinterpret_cast<const void*>(&cluster_bwd_kernel<dd, 3>);
    return dbl ? reinterpret_cast<const void*>(&cluster_bwd_kernel<double, 3>)
               : reinterpret_cast<const void*>(&cluster_bwd_kernel<float, 4>);
}

}  // namespace vqc
