// kernels.h -- entry points into the kernel translation units (one per real
// type and mode, compiled in parallel).  Each returns the address of the
// sweep kernel instantiated for register-block size K, or nullptr.
#pragma once

namespace vqc {

const void* sweep_ptr_f32_fwd(int K);          // sample groups of >= 32 threads
const void* sweep_ptr_f32_bwd(int K);
const void* sweep_ptr_f64_fwd(int K);
const void* sweep_ptr_f64_bwd(int K);
const void* sweep_ptr_f32_fwd_small(int K);    // sample groups of < 32 threads
const void* sweep_ptr_f32_bwd_small(int K);
const void* sweep_ptr_f64_fwd_small(int K);
const void* sweep_ptr_f64_bwd_small(int K);
const void* sweep_ptr_f32_fused(int K, bool full);   // backward that also writes E
// plans without CRZ / RZZ phase ops: instantiations without the phase cases
const void* sweep_ptr_f32_fwd_nph(int K, bool full);
const void* sweep_ptr_f32_bwd_nph(int K, bool full);
const void* sweep_ptr_f32_fused_nph(int K, bool full);
const void* pass_ptr_f32_fwd_nph(int K, bool full);
const void* sweep_ptr_f64_fused(int K, bool full);
// double-float arithmetic on complex128 storage (VQC_C128_DF plans)
const void* sweep_ptr_dd_fwd(int K, bool full);
const void* sweep_ptr_dd_bwd(int K, bool full);
const void* sweep_ptr_dd_fused(int K, bool full);
const void* pass_ptr_dd(int mode, int K, bool full);
const void* cluster_ptr_dd();
const void* reduce_terms_ptr_dd();
const void* ps_tables_ptr_dd();

// HBM-tiled pass kernels (K fixed per type and mode) and partial reductions.
const void* pass_ptr(bool dbl, int mode, int K, bool full);   // full: tile groups >= 32 threads
const void* reduce_expz_ptr(bool dbl);
const void* reduce_dx_ptr(bool dbl);
const void* reduce_dw_ptr(bool dbl);
const void* reduce_terms_ptr(bool dbl);   // per-sample gradient terms from per-tile rho sums
const void* ps_tables_ptr(bool dbl);      // per-sample table entries of every sample (HBM passes)
const void* reduce_cols_ptr(bool dbl);
const void* abs2_ptr(bool dbl);   // |psi|^2, elementwise
const void* cluster_ptr(bool dbl);   // cluster-path forward (K = 5 / 4 for complex64 / 128)
const void* cluster_bwd_ptr(bool dbl, bool dfloat);   // cluster-path backward (K = 4 / 3)

// Largest block (threads) each instantiation is compiled for.
inline int sweep_max_threads(bool is_double, int mode, int K) {
    (void)is_double;
    (void)mode;
    (void)K;
    return 512;   // sweep kernels: __launch_bounds__(512) (<= 128 registers)
}

}  // namespace vqc
