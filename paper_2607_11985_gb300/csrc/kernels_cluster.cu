// kernels_cluster.cu -- instantiations of the cluster-path forward kernel
// (complex64: K = 5, complex128: K = 4).
#include "kernels.h"
#include "cluster.cuh"

namespace vqc {

const void* cluster_ptr(bool dbl) {
    return dbl ? reinterpret_cast<const void*>(&cluster_fwd_kernel<double, 4>)
               : reinterpret_cast<const void*>(&cluster_fwd_kernel<float, 5>);
}

}  // namespace vqc
