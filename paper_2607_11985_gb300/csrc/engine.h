// engine.h -- host-side plan object shared by the compiler (compiler.cpp) and
// the C ABI / launch code (capi.cu).  Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>
#include <string>
#include <vector>

#include "plan.h"
#include "../../include/vqc.h"

static_assert(sizeof(vqc_gate) == 48, "vqc_gate layout");

namespace vqc {

// A fused op of the lowered circuit (time-valid order).
struct HOp {
    uint8_t type;      // OpType
    int q0, q1;        // M1: q0 target; CX: q0 control, q1 target; CZ/PH2: q0, q1
    int entry;         // table entry id for M1 / PH2, else -1
    uint8_t gen;       // OPF_GEN_* for PH2
};

// One register-block stage schedule for a (mode, K, tile) choice.
struct Schedule {
    int mode = 0;          // 0 forward, 1 backward
    int K = 0;             // register-block qubits
    int m = 0;             // qubits per shared-memory tile (== n on the resident path)
    int path = VQC_PATH_RESIDENT;
    int thread_bits = 0;   // m - K
    int group_lanes_log2 = 0;   // log2(threads per sample group) when < 2^G
    int cta_bits = 0;           // cluster path: log2(threads per CTA); 2^(m-K-cta_bits) CTAs
    std::vector<DOp> ops;
    std::vector<DStage> stages;
    std::vector<DPass> passes;            // HBM path: one record per pass
    std::vector<int32_t> pass_entries;    // HBM path: table entries per pass (ps, then sh)
    std::vector<int32_t> pass_accs;       // HBM path: accumulator ids per pass
    // Per stage, kMaxK + kMaxThreadBits physical-index masks: the image under
    // the stage's absorbed permutation of each local bit, then of each thread
    // bit (exported for tests; the kernels use the swizzled store map).
    std::vector<uint32_t> store_masks;
    size_t dev_ops = 0, dev_stages = 0;   // byte offsets inside the device buffer
    size_t dev_passes = 0, dev_pass_entries = 0, dev_pass_accs = 0;
    size_t dev_region_begin = 0, dev_region_end = 0;   // [ops .. pass_accs] in the blob
};

struct HostPlan {
    int n = 0, num_x = 0, num_w = 0, dtype = 0, num_gates_in = 0;
    int G_swz = 4;                         // swizzle chunk bits (4: c64, 3: c128)
    bool dfloat = false;                   // VQC_C128_DF: complex128 storage, double-float kernels
    bool has_ph2 = false;                  // the op list holds diagonal two-qubit phases (CRZ / RZZ)
    std::vector<HOp> ops;
    std::vector<DEntry> entries;
    std::vector<DConst> consts;
    std::vector<double> cmat;              // 8 doubles per constant 2x2 matrix
    std::vector<double> cang;              // constant angles
    std::vector<int32_t> term_src, term_idx;   // per term: SRC_X / SRC_W, column
    std::vector<DAcc> accs;
    std::vector<int32_t> xocc_ptr, xocc, wocc_ptr, wocc;   // terms of each x column / w index
    int n_ps = 0, n_sh = 0;                // per-sample / shared table sizes
    int n_runs = 0;
    std::vector<Schedule> scheds;
    double fwd_flops = 0, bwd_flops = 0, recompute_flops = 0;

    // device copy
    int device = -1;
    void* dbuf = nullptr;
    size_t dbytes = 0;
    size_t dev_entries = 0, dev_ps_list = 0, dev_sh_list = 0, dev_consts = 0, dev_cmat = 0, dev_cang = 0;
    size_t dev_xocc_ptr = 0, dev_xocc = 0, dev_wocc_ptr = 0, dev_wocc = 0, dev_accs = 0;
    unsigned* dev_error = nullptr;        // device error word (kernel self-checks)
    size_t dev_tab_begin = 0, dev_tab_end = 0;   // [entries .. wocc] in the blob
};

// Largest n whose state(s) fit one CTA's shared memory on the resident path.
inline int resident_max_qubits(int mode, int dtype) {
    if (dtype == VQC_C64) return mode == 0 ? 14 : 13;
    return mode == 0 ? 13 : 12;
}
// Tile qubits of an HBM pass: 64 KiB of tile state per CTA (two states for the backward).
inline int hbm_tile_qubits(int mode, int dtype, int G) {
    (void)G;
    if (dtype == VQC_C64) return mode == 0 ? 13 : 12;
    return mode == 0 ? 12 : 11;
}
inline int hbm_k(int mode, int dtype) {
    if (dtype == VQC_C64) return mode == 0 ? 5 : 4;
    return mode == 0 ? 4 : 3;
}

// Maximum K per (mode, dtype) for register-resident blocks.
inline int max_k(int mode, int dtype) {
    if (dtype == VQC_C64) return mode == 0 ? 5 : 4;
    return mode == 0 ? 4 : 3;
}

// compiler.cpp
vqc_status compile_host(const vqc_gate* gates, int32_t G, int32_t n, int32_t nx, int32_t nw,
                        int dtype, HostPlan& out, std::string& err);
const Schedule* find_schedule(const HostPlan& p, int mode, int K);
const Schedule* find_hbm_schedule(const HostPlan& p, int mode);
const Schedule* find_cluster_schedule(const HostPlan& p, int mode);
std::vector<uint8_t> export_plan(const HostPlan& p);

}  // namespace vqc

// The opaque handle of the C ABI: a compiled host plan (and its device copy).
struct vqc_plan {
    vqc::HostPlan hp;
};
