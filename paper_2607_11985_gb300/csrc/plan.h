// plan.h -- the compiled plan: host representation and the POD records the
// kernels read from device memory.
//
// A plan is the "gate sequence with cached static unitaries" of the paper's
// compile phase (Alg. 1, compile phase), lowered further for the GPU:
//
//   * single-qubit gates that meet consecutively on a qubit are fused into a
//     run; consecutive constant factors of a run are pre-multiplied on the host
//     in fp64 (Alg. 1: "precompute and cache" constant matrices);
//   * two-qubit gates become CX (conditional swap), CZ (sign) or a diagonal
//     two-qubit phase (CRZ, RZZ); SWAP is lowered to three CX;
//   * the op list is cut into stages.  In a stage every thread of a sample's
//     thread group holds a register block of 2^K amplitudes spanned by the
//     stage's K "active" qubits; every non-diagonal op of the stage acts on
//     active qubits only, diagonal ops and CX controls may use any qubit.
//     Between stages the state goes through shared memory.
//
// Amplitude addressing in shared memory (per sample, tile-local index u):
//   slot(u) = sw(u) ^ h_sample,   sw(u) = u ^ (fold_G(u >> G) & (2^G - 1))
// with G = 4 for complex64 and 3 for complex128 (2^G amplitudes = 128 bytes).
// sw is linear over GF(2), so the slot of amplitude r of a thread's block is
// XOR(swizzled thread base, XOR of sigma[j] over set bits j of r).
#pragma once

#include <cstdint>

namespace vqc {

constexpr int kMaxK = 5;             // register-block qubits per thread (<= 32 amplitudes)
constexpr int kMaxThreadBits = 16;   // thread-index bits of one sample group / tile
constexpr uint8_t kRefPhys = 8;      // qubit ref >= 8: physical qubit (ref - 8), not active

// ---- ops (8 bytes) -------------------------------------------------------
enum OpType : uint8_t {
    OP_M1 = 1,    // general 2x2 on active local position a; table entry `slot`
    OP_CX = 2,    // control ref a (local or physical), target local b
    OP_CZ = 3,    // sign on bit a & bit b (refs)
    OP_PH2 = 4    // diagonal phase ph[bit a + 2 bit b] from table entry `slot`
};
enum OpFlags : uint8_t {
    OPF_PER_SAMPLE = 1,   // table entry lives in the per-sample table
    OPF_GEN_CRZ = 2,      // generator |1><1|_a (x) Z_b   (CRZ)
    OPF_GEN_RZZ = 4,      // generator Z_a (x) Z_b        (RZZ)
    OPF_HAS_ACC = 8       // op accumulates a gradient slot (aux) in the backward
};

// Dispatch code of a compiled op (DOp::code): the kernels take one jump-table
// branch per op, each case specialised for fixed local positions.
enum DispatchCode : uint8_t {
    DC_M1 = 0,       // + t: 2x2 on local position t (0..4)
    DC_CX_LL = 5,    // + 4c + (t < c ? t : t - 1): local control c, local target t
    DC_CX_PL = 25,   // + t: control outside the block (ref a), local target t
    DC_CZ_LL = 30,   // + cz_pair_index(lo, hi): both qubits local
    DC_CZ_PL = 40,   // + l: local qubit l (ref a), other qubit outside the block (ref b)
    DC_CZ_PP = 45,   // both qubits outside the block
    DC_PH2_LL = 46,  // + cz_pair_index(lo, hi): diagonal two-qubit phase, both qubits local
    DC_PH2_PL = 56,  // + l: diagonal phase, one qubit local (position l), the other outside
    DC_PH2_PP = 61,  // diagonal phase, both qubits outside the block
    DC_NUM = 62
};
// Index of the local pair (lo < hi < 5) in (0,1),(0,2),(0,3),(0,4),(1,2),...,(3,4).
constexpr int cz_pair_index(int lo, int hi) {
    return lo == 0 ? hi - 1 : lo == 1 ? 2 + hi : lo == 2 ? 4 + hi : 5 + hi;
}

struct DOp {
    uint8_t code;    // DispatchCode
    uint8_t a, b;    // qubit refs (< kRefPhys: local position; else kRefPhys + qubit)
    uint8_t flags;
    uint16_t slot;   // table entry index inside its table (per-sample or shared)
    uint16_t aux;    // accumulator slot for the backward (run or phase op id)
};
static_assert(sizeof(DOp) == 8, "DOp layout");

// ---- stages ----------------------------------------------------------------
// A stage loads each block through its load map (sigma, tau), applies its ops
// and stores the block through its store map (sigma_st, tau_st).  On the
// resident path the compiler folds CX gates into the store map instead of
// emitting them as ops: a CX is a permutation of basis states, linear over
// GF(2) in the amplitude index, so storing amplitude k of the block at the slot
// of pi(k) applies it at no arithmetic cost (pi = the stage's absorbed CX gates
// in time order; every op of the stage that follows one of them in time acts on
// other qubits, so it commutes with pi).  Without absorbed gates the two maps
// are equal.
struct DStage {
    int32_t op_begin, op_end;
    int32_t sigma[kMaxK];             // load: swizzled slot offset of local bit j
    int32_t tau[kMaxThreadBits];      // load: swizzled slot offset of thread bit i
    uint32_t tmask[kMaxThreadBits];   // physical-index bit of thread bit i
    int32_t sigma_st[kMaxK];          // store: slot offset of pi(local bit j)
    int32_t tau_st[kMaxThreadBits];   // store: slot offset of pi(thread bit i)
    uint8_t active[kMaxK];            // physical qubit of local bit j
    uint8_t nthreadbits;
    uint8_t nperm;                    // CX gates absorbed into the store map
    uint8_t cl_local;                 // cluster path: bit 0 loads, bit 1 stores stay in the
                                      // thread's own CTA (its rank = top thread bits)
};
static_assert(sizeof(DStage) == 248, "DStage layout");

// ---- table entries and their constituents ----------------------------------
enum ConstKind : uint8_t {
    CK_CONST = 1,    // pre-multiplied constant 2x2 (cmat[idx0])
    CK_RX = 2, CK_RY = 3, CK_RZ = 4,   // exp(-i t P / 2), angle from src0
    CK_GPHASE = 5,   // scalar e^{i (t0 + t1) / 2} (global phase of U3)
    CK_CRZ = 6,      // phases (1, e^{-it/2}, 1, e^{it/2}) on s = b0 + 2 b1
    CK_RZZ = 7       // phases (e^{-it/2}, e^{it/2}, e^{it/2}, e^{-it/2})
};
enum SrcKind : uint8_t { SRC_NONE = 0, SRC_CONST = 1, SRC_X = 2, SRC_W = 3 };

struct DConst {
    uint8_t kind, src0, src1, pad;
    int32_t idx0, idx1;   // x column / w index / const-angle index (or cmat index for CK_CONST)
    int32_t term;         // gradient term index, -1 if none
};
static_assert(sizeof(DConst) == 16, "DConst layout");

struct DEntry {
    uint16_t cfirst, ccount;   // constituents, in time order
    uint16_t slot;             // index inside its table
    uint8_t per_sample;        // 1: depends on x[b]
    uint8_t phase;             // 0: 2x2 matrix, 1: four diagonal phases
    uint16_t acc;              // accumulator slot (backward)
    uint16_t pad;
};
static_assert(sizeof(DEntry) == 12, "DEntry layout");

// One pass of the HBM-tiled path: its stages act on tiles of m qubits; the
// other n - m qubits index the tiles of a sample.
struct DPass {
    int32_t stage_begin, stage_end;
    int32_t m, nout;
    uint8_t tile_q[24];   // tile-local bit i -> qubit
    uint8_t out_q[24];    // tile index bit j -> qubit
    int32_t ps_begin, ps_count;    // per-sample table entries of the pass (into pass_entries)
    int32_t sh_begin, sh_count;    // shared table entries of the pass
    int32_t acc_begin, acc_count;  // accumulators of the pass (into pass_accs)
};
static_assert(sizeof(DPass) == 88, "DPass layout");

// Accumulator slot -> what it holds (backward).
struct DAcc {
    int32_t entry;   // table entry id
    int32_t kind;    // 0: 2x2 rho of a run, 1: scalar of a phase op
};

}  // namespace vqc
