/*
 * vqc.h -- C ABI of the GB300 batched statevector engine for static
 * parametrised quantum circuits.
 *
 * The operation (paper, Alg. 1 "Compile-Once Lowering and Batched Execution",
 * and Sec. 3 "Compile-Once Lowering and Execution"):
 *   compile once:  a static gate list (no measurement, no classical control,
 *                  only angles vary; Sec. 3 "Static Circuit Scope") is lowered
 *                  to a plan; constant gates are pre-multiplied into cached
 *                  matrices, parametrised gates stay symbolic (Alg. 1, compile
 *                  phase).
 *   execute:       for a batch of B samples, psi_b = U_G ... U_1 psi0_b with
 *                  psi0_b = |0...0> unless given, and
 *                  E[b, j] = sum_k (-1)^{k_j} |psi_b[k]|^2     (Alg. 1, execute
 *                  phase and return statement).
 *   differentiate: for L = sum_{b,j} gE[b, j] * E[b, j], dL/dx[b, .] for the
 *                  per-sample angles and dL/dw[.] for the shared angles
 *                  (Sec. 3 "Gate Application and Differentiation": gradients
 *                  with respect to trainable parameters).  The engine uses the
 *                  adjoint method (two states, O(B 2^n) memory) where the paper
 *                  used autograd (O(B G 2^n) memory, Sec. 3 "Complexity and
 *                  Tradeoffs").
 *
 * Conventions.  Qubit q is bit q of the amplitude index (little endian).  A
 * gate list is in time order.  States are interleaved (re, im) pairs: float2
 * for VQC_C64, double2 for VQC_C128 and VQC_C128_DF; arrays are row-major
 * and sample-major.  Real arrays (x, w, E, gradients) are float for VQC_C64
 * and double for VQC_C128 and VQC_C128_DF.  Gate matrices: RX/RY/RZ(t) = exp(-i t P / 2); U3 is
 * [[c, -e^{i l} s], [e^{i p} s, e^{i(p+l)} c]] with c, s = cos, sin(t/2);
 * CRZ(t) = |0><0|_q0 (x) I + |1><1|_q0 (x) RZ_q1(t); RZZ(t) = exp(-i t Z Z / 2);
 * CX/CRZ control is q0, target q1.
 *
 * Ownership.  The caller owns every device buffer and the CUDA stream.
 * vqc_compile copies the gate list; the plan owns its host and device copies
 * and is released with vqc_free.  Calls are stream-ordered and asynchronous:
 * a returned VQC_OK means the work was enqueued.  No C++ exception crosses
 * this ABI.  A plan may be used from several threads; calls that share a
 * workspace must be ordered on one stream.
 *
 * Errors.  Every call returns a vqc_status; vqc_last_error() gives a
 * thread-local message for the last failing call on the calling thread.
 */
#ifndef VQC_ABI_H_INCLUDED
#define VQC_ABI_H_INCLUDED

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define VQC_ABI_VERSION 1
#define VQC_MAX_QUBITS 24

typedef struct vqc_plan vqc_plan;   /* opaque */

typedef enum {
    VQC_OK = 0,
    VQC_ERR_INVALID_ARG = 1,       /* NULL where a pointer is required, bad size or dtype */
    VQC_ERR_UNSUPPORTED_GATE = 2,  /* opcode outside vqc_gate_op */
    VQC_ERR_QUBIT_RANGE = 3,       /* qubit >= num_qubits, or q0 == q1 on a 2q gate */
    VQC_ERR_TOO_MANY_QUBITS = 4,   /* num_qubits outside 1..VQC_MAX_QUBITS */
    VQC_ERR_PARAM_RANGE = 5,       /* angle source kind or index out of range */
    VQC_ERR_OUT_OF_MEMORY = 6,     /* host or device allocation failed */
    VQC_ERR_CUDA = 7,              /* a CUDA runtime call failed (message has the name) */
    VQC_ERR_WORKSPACE = 8,         /* workspace NULL, too small or not 256-byte aligned */
    VQC_ERR_DEVICE_CHECK = 9,      /* a kernel's own bounds/consistency check tripped */
    VQC_ERR_UNSUPPORTED = 10       /* valid request the library cannot run (e.g. too large) */
} vqc_status;

/* VQC_C128_DF: complex128 in memory (every array, layout, workspace size and
 * plan schedule exactly as VQC_C128) with the kernels computing in double-float
 * arithmetic on the FP32 units: each real is an unevaluated sum of two floats
 * (about 48 significant bits; error-free sums and FMA products, Dekker 1971),
 * split when read and rejoined when written.  Results agree with VQC_C128 to
 * about 1e-13 (the complex128 parity bound, 1e-10, holds); on parts whose FP64
 * rate is a small fraction of the FP32 rate (GB300: about 1/75) it is the
 * faster way to complex128 accuracy.  vqc_plan_export gives the same bytes as
 * for VQC_C128 (the arithmetic is chosen at launch, not in the plan). */
typedef enum { VQC_C64 = 0, VQC_C128 = 1, VQC_C128_DF = 2 } vqc_dtype;

/* The 16-gate set.  Angles per gate: RX/RY/RZ/CRZ/RZZ one (theta),
 * U3 three (theta, phi, lambda), the rest none. */
typedef enum {
    VQC_H = 0, VQC_X = 1, VQC_Y = 2, VQC_Z = 3, VQC_S = 4, VQC_T = 5, VQC_SX = 6,
    VQC_RX = 7, VQC_RY = 8, VQC_RZ = 9, VQC_U3 = 10,
    VQC_CX = 11, VQC_CZ = 12, VQC_SWAP = 13, VQC_CRZ = 14, VQC_RZZ = 15,
    VQC_NUM_GATE_OPS = 16
} vqc_gate_op;

/* Source of one angle (Alg. 1 compile phase: constant gates are cached,
 * parametric gates are instantiated from theta at run time). */
typedef enum {
    VQC_P_NONE = 0,    /* unused slot */
    VQC_P_CONST = 1,   /* pconst[i] */
    VQC_P_X = 2,       /* per-sample angle x[b, pidx[i]] */
    VQC_P_W = 3        /* shared angle w[pidx[i]] */
} vqc_pkind;

/* One gate of the input list (48 bytes, natural alignment, no implicit padding). */
typedef struct {
    uint8_t op;          /* vqc_gate_op */
    uint8_t q0;          /* first qubit (control of CX / CRZ) */
    uint8_t q1;          /* second qubit (target); ignored for 1q gates */
    uint8_t pkind[3];    /* vqc_pkind of each angle slot; slots beyond the gate's arity ignored */
    uint8_t reserved[2]; /* must be zero */
    int32_t pidx[3];     /* column of x or index of w for VQC_P_X / VQC_P_W */
    int32_t reserved2;   /* must be zero */
    double pconst[3];    /* angle for VQC_P_CONST */
} vqc_gate;

/* Execution paths a plan can take. */
typedef enum {
    VQC_PATH_RESIDENT = 0,  /* each sample's state stays in one CTA's shared memory */
    VQC_PATH_HBM = 1,       /* state in HBM, swept in shared-memory tiles, one launch per pass */
    VQC_PATH_CLUSTER = 2    /* each sample's state (forward) or its psi and lambda (backward)
                               spread over the shared memory of a thread-block cluster (2..8
                               CTAs of 512 threads), one launch (plus the fixed-order dw sum);
                               taken by default for 2-CTA clusters (forward: complex64 15
                               qubits, complex128 14; backward: complex64 14, complex128 13),
                               for larger ones only when the environment sets
                               VQC_FORCE_PATH=cluster (they measured slower than VQC_PATH_HBM);
                               VQC_FORCE_PATH=hbm turns it off.  The backward's workspace is a
                               256-byte control block and one dw partial per cluster. */
} vqc_path;

typedef struct {
    int32_t num_qubits, num_x, num_w, dtype;   /* dtype as given to vqc_compile */
    int32_t num_gates_in;        /* gates given to vqc_compile */
    int32_t num_ops;             /* fused ops after lowering (1q runs, CX, CZ, phase ops) */
    int32_t num_runs;            /* fused single-qubit runs */
    int32_t num_terms;           /* parametrised angle occurrences carrying a gradient */
    int32_t fwd_path, bwd_path;  /* vqc_path chosen for the batch given to vqc_plan_info (-1: none) */
    int32_t fwd_k, bwd_k;        /* register-block qubits per thread */
    int32_t fwd_stages, bwd_stages;
    int32_t fwd_passes, bwd_passes;      /* HBM passes (1 on the resident path) */
    int32_t fwd_threads_per_sample, bwd_threads_per_sample;
    int32_t fwd_tile_qubits, bwd_tile_qubits;
    double fwd_flops_per_eval;   /* algorithmic flops of one forward evaluation */
    double bwd_flops_per_eval;   /* algorithmic flops of one backward evaluation (from psi_final) */
    double recompute_flops_per_eval;     /* extra flops when the backward recomputes psi_final */
    double fwd_hbm_bytes_per_eval;       /* state bytes moved through HBM per forward evaluation */
    double bwd_hbm_bytes_per_eval;
} vqc_plan_stats;

/* Compile a gate list (paper, Alg. 1 compile phase).  Validates every gate,
 * fuses runs of single-qubit gates, pre-multiplies constant matrices, and
 * builds the register-block stage schedules.  When the process sees a CUDA
 * device, uploads the plan to the current device (one synchronous copy);
 * otherwise the plan is host-only (vqc_plan_info / vqc_plan_export work) and
 * the first vqc_forward / vqc_backward uploads it, so that first call must
 * not be made inside CUDA stream capture.  dtype is VQC_C64, VQC_C128 or
 * VQC_C128_DF (a VQC_C128 plan whose kernels compute in double-float; see
 * vqc_dtype).  On success *out_plan owns the result.
 * Errors: VQC_ERR_INVALID_ARG (NULL gates with num_gates > 0, NULL out_plan,
 * negative counts, bad dtype, nonzero reserved bytes), VQC_ERR_UNSUPPORTED_GATE,
 * VQC_ERR_QUBIT_RANGE, VQC_ERR_TOO_MANY_QUBITS, VQC_ERR_PARAM_RANGE,
 * VQC_ERR_OUT_OF_MEMORY, VQC_ERR_CUDA. */
vqc_status vqc_compile(const vqc_gate* gates, int32_t num_gates, int32_t num_qubits,
                       int32_t num_x, int32_t num_w, vqc_dtype dtype, vqc_plan** out_plan);

/* OpenQASM 2 front end (paper, Sec. 3 "Static Circuit Scope" and Fig. 2: the
 * circuit is given as normalised OpenQASM and parsed once).  Accepted:
 * "OPENQASM 2.0;", include "qelib1.inc", qreg / creg declarations (quantum
 * registers are numbered in declaration order, qubit 0 first), the gate set
 * under its qelib1 names -- h x y z s t sx rx ry rz u3 (also u, U) cx (CX) cz
 * swap crz rzz -- and the exact U3 special cases u1 / p, u2, sdg, tdg, id;
 * `barrier` and terminal `measure` are accepted and ignored (the engine
 * returns <Z>); a gate or barrier on a qubit after its measurement is rejected
 * with VQC_ERR_UNSUPPORTED_GATE (a mid-circuit measurement is outside the
 * static-circuit scope).
 * Whole-register operands broadcast over equal-sized registers.  An angle is a
 * constant expression (numbers, pi, + - * / ^, unary minus, parentheses, sin
 * cos tan exp ln sqrt) or, as the variational extension, exactly one parameter
 * reference: x[i] (per-sample column i) or w[j] (shared weight j).  Gate
 * definitions, opaque, if and reset are rejected (VQC_ERR_UNSUPPORTED_GATE),
 * as are gates outside the set; errors name the source line.
 *
 * vqc_parse_qasm lowers `source` to vqc_gate records: *inout_num_gates is the
 * capacity of `gates` on entry and the program's gate count on return; pass
 * gates = NULL to query the count.  num_qubits, num_x (largest x index + 1) and
 * num_w (largest w index + 1) are written on success.  Host only. */
vqc_status vqc_parse_qasm(const char* source, vqc_gate* gates, int32_t* inout_num_gates,
                          int32_t* num_qubits, int32_t* num_x, int32_t* num_w);

/* vqc_parse_qasm followed by vqc_compile.  num_x / num_w < 0 take the counts
 * the program implies; given counts must cover every referenced index
 * (VQC_ERR_PARAM_RANGE otherwise).  Other errors as vqc_compile. */
vqc_status vqc_compile_qasm(const char* source, int32_t num_x, int32_t num_w, vqc_dtype dtype,
                            vqc_plan** out_plan);

/* Release a plan (NULL-safe).  The caller must make sure no enqueued call
 * still uses it (synchronise the streams first). */
void vqc_free(vqc_plan* plan);

/* Bytes of device workspace a call needs: mode 0 = vqc_forward, 1 = vqc_backward,
 * 2 = vqc_probabilities, 3 = vqc_forward_backward.  Returns 0 when no workspace is needed; (size_t)-1 for
 * a NULL plan. */
size_t vqc_workspace_bytes(const vqc_plan* plan, int32_t batch, int32_t mode);

/* Zero a workspace's control block on `stream` (enqueued memset).  A freshly
 * allocated workspace must be initialised once with this call (or zeroed by
 * the caller) before its first use; every call leaves it initialised. */
vqc_status vqc_workspace_init(void* workspace, size_t workspace_bytes, void* stream);

/* Forward sweep (paper, Alg. 1 execute phase).
 *   batch     B >= 0 (B == 0 enqueues nothing).
 *   x         device [B, num_x] real, or NULL when num_x == 0.
 *   w         device [num_w] real, or NULL when num_w == 0.
 *   psi0      device [B, 2^n] complex initial states, or NULL for |0...0>.
 *   expz_out  device [B, n] real: E[b, j] (required).
 *   state_out device [B, 2^n] complex final states, or NULL.
 *   workspace device scratch of vqc_workspace_bytes(plan, B, 0) bytes, 256-byte
 *             aligned (may be NULL when that size is 0).
 *   stream    cudaStream_t (NULL = legacy default stream).
 * Buffers must not overlap, except that state_out may equal psi0. */
vqc_status vqc_forward(const vqc_plan* plan, int32_t batch, const void* x, const void* w,
                       const void* psi0, void* expz_out, void* state_out,
                       void* workspace, size_t workspace_bytes, void* stream);

/* Adjoint backward (paper, Sec. 3 gradients).  For L = sum gE * E:
 *   psi_final device [B, 2^n] complex: the state_out of a vqc_forward with the
 *             same plan, x, w and psi0, or NULL to recompute it in the kernel.
 *   grad_expz device [B, n] real gE (required).
 *   grad_x    device [B, num_x] real, overwritten with dL/dx (or NULL: not computed).
 *   grad_w    device [num_w] real, overwritten with dL/dw summed over the
 *             batch in a fixed order (deterministic for a given plan and B),
 *             or NULL.
 *   workspace vqc_workspace_bytes(plan, B, 1) bytes, 256-byte aligned,
 *             initialised once with vqc_workspace_init.
 * Other arguments as vqc_forward. */
vqc_status vqc_backward(const vqc_plan* plan, int32_t batch, const void* x, const void* w,
                        const void* psi0, const void* psi_final, const void* grad_expz,
                        void* grad_x, void* grad_w, void* workspace, size_t workspace_bytes,
                        void* stream);

/* Forward and adjoint backward together, for a loss whose gradient gE is known
 * before the call (L = sum gE * E with fixed weights; the paper's own objective,
 * the mean of <Z_j>, has gE = 1/n): E, dL/dx and dL/dw of one batch.  Where the
 * state fits one SM (the resident path) it is ONE launch: the backward kernel
 * runs the forward sweep itself, keeps the final states in shared memory,
 * writes E and sweeps back, so no state goes through HBM -- unless the forward
 * alone would take larger register blocks than the backward, when it is
 * vqc_forward saving the final states in the workspace followed by
 * vqc_backward from them (faster there).  Beyond one SM it is vqc_forward
 * (final states into the workspace) followed by the backward passes or the
 * cluster backward from them.
 *   expz_out  device [B, n] real (required); grad_expz device [B, n] (required);
 *   grad_x, grad_w as vqc_backward; psi0 as vqc_forward.
 *   workspace vqc_workspace_bytes(plan, B, 3) bytes, 256-byte aligned,
 *             initialised once with vqc_workspace_init.
 * E agrees with vqc_forward and the gradients with vqc_backward to rounding (the
 * sweeps may group the gates into different stages).  Errors as vqc_backward. */
vqc_status vqc_forward_backward(const vqc_plan* plan, int32_t batch, const void* x, const void* w,
                                const void* psi0, const void* grad_expz, void* expz_out, void* grad_x,
                                void* grad_w, void* workspace, size_t workspace_bytes, void* stream);

/* Measurement probabilities |psi_b[k]|^2 of the final states (paper, Sec. 3:
 * the engine's outputs are the statevector or its probabilities, and <Z>):
 * probs_out [B, 2^n] real (float / double), logical amplitude order.  Runs the
 * forward sweep into the workspace (vqc_workspace_bytes mode 2: the forward's
 * own workspace, then the states and <Z> of the batch; 256-byte aligned, the
 * first 256 bytes cleared once by vqc_workspace_init), then one elementwise
 * kernel.  Inputs as vqc_forward.  Errors as vqc_forward, VQC_ERR_WORKSPACE for
 * a missing, short or misaligned workspace. */
vqc_status vqc_probabilities(const vqc_plan* plan, int32_t batch, const void* x, const void* w,
                             const void* psi0, void* probs_out, void* workspace,
                             size_t workspace_bytes, void* stream);

/* Bytes of device scratch built into the library for vqc_backward_noalloc
 * (one array per GPU that loads the library, held until the process exits). */
#define VQC_NOALLOC_SCRATCH_BYTES (1u << 20)

/* vqc_backward without a workspace argument, for callers that cannot allocate
 * device memory (a plugin whose host application owns all device memory, a
 * real-time loop that must not pay cudaMalloc's latency or implicit device
 * synchronisation, code under a fixed device-memory budget).  The paper has no
 * counterpart; it is a deployment convenience of this library.
 *   Arguments, outputs and results are those of vqc_backward.  The scratch is
 *   a fixed array of VQC_NOALLOC_SCRATCH_BYTES inside the library; a batch
 *   whose scratch need (vqc_workspace_bytes(plan, batch, 1)) exceeds it is
 *   rejected with VQC_ERR_WORKSPACE and a message giving both sizes.
 *   No cudaMalloc, cudaFree or allocating library call is made.  Each call
 *   clears the array's control block on `stream` before its launch; all calls
 *   on a device share the array, so calls that overlap on the GPU race and must
 *   be ordered by the caller.  The first call on a device (with that device
 *   current) looks up the array's device address; make it before any CUDA
 *   stream capture begins.  That address is cached for the process: the entry
 *   point assumes the CUDA runtime's primary context and no cudaDeviceReset
 *   while the library is loaded. */
vqc_status vqc_backward_noalloc(const vqc_plan* plan, int32_t batch, const void* x,
                                const void* w, const void* psi0, const void* psi_final,
                                const void* grad_expz, void* grad_x, void* grad_w, void* stream);

/* One evaluation with inputs and outputs in HOST memory (pageable or pinned):
 * the forward sweep and, when grad_expz is given, the adjoint backward from the
 * forward's final states (paper, Alg. 1 execute phase and Sec. 3 gradients;
 * the loss is L = sum gE * E with gE known before the call, e.g. fixed
 * observable weights).  For callers whose data live on the host.  Where the
 * device accesses pageable host memory coherently (vqc_host_direct() == 1,
 * e.g. Grace-Blackwell over NVLink-C2C) the kernels read and write the
 * caller's arrays in place and no copy is made; otherwise the inputs are packed
 * into a pinned staging area and moved in ONE host-to-device copy and the
 * outputs come back in ONE device-to-host copy.
 *   x         host [B, num_x] real (NULL when num_x == 0).
 *   w         host [num_w] real (NULL when num_w == 0).
 *   grad_expz host [B, n] real gE, or NULL for the forward only.
 *   expz_out  host [B, n] real: E (required).
 *   grad_x    host [B, num_x] real dL/dx, or NULL (ignored without grad_expz).
 *   grad_w    host [num_w] real dL/dw summed over the batch, or NULL.
 *   stream    cudaStream_t the work is enqueued on.
 * The work is vqc_forward_backward (vqc_forward without grad_expz).
 * Initial states are |0...0>.  The plan owns a device arena (packed inputs and
 * outputs, the workspace) and a pinned host mirror, sized for
 * the largest batch seen on the current device and released by vqc_free; calls
 * on one plan are serialised by the plan.  Blocking: returns after `stream`
 * has finished the call's work.  Errors as vqc_forward / vqc_backward, plus
 * VQC_ERR_OUT_OF_MEMORY when the arena or the staging area cannot be allocated. */
vqc_status vqc_evaluate_host(const vqc_plan* plan, int32_t batch, const void* x, const void* w,
                             const void* grad_expz, void* expz_out, void* grad_x, void* grad_w,
                             void* stream);

/* 1 when vqc_evaluate_host on `device` lets the kernels access host arrays in
 * place (cudaDevAttrPageableMemoryAccess is set and the environment does not
 * set VQC_HOST_DIRECT=0), else 0 (staged copies). */
int32_t vqc_host_direct(int32_t device);

/* The fused multiply-add rate of the current device for the arithmetic of
 * `dtype`'s sweeps (VQC_C64 and VQC_C128_DF: packed FP32 pairs, the FP32
 * lanes double-float also runs on; VQC_C128: FP64), in TFLOP/s
 * (an FMA counts as two flops), measured: a kernel of independent FMA chains
 * over every SM, calibrated to launches of about 5 ms, best of five timed
 * launches.  This is the arithmetic ceiling against which the sweep kernels'
 * algorithmic flop rates are reported (roofline of the resident path, Sec. 3
 * complexity O(B * G * 2^n)).  Blocking; runs on a private stream; takes
 * about 50 ms.  Errors: VQC_ERR_INVALID_ARG (NULL out, bad dtype),
 * VQC_ERR_CUDA. */
vqc_status vqc_fma_peak(vqc_dtype dtype, double* tflops_out);

/* One batch-shared 5-qubit stage applied to a batch of complex64 states, on
 * the tensor cores or on the FP32 CUDA cores: the measurement behind the
 * engine's choice of FP32 register blocks over tensor-core stages (paper,
 * Sec. 3 "Gate Application and Differentiation": the prior art applies gates
 * as batched matrix products).  Not used by the evaluation calls above.
 *   method    1: the dense 32 x 32 complex Kronecker product of the factors
 *             as a real 64 x 64 matrix product on tcgen05 tensor cores (tf32
 *             operands split into high and low parts, three products
 *             accumulated in FP32 in tensor memory); 0: the five 2x2 factors in
 *             packed FP32 register blocks.
 *   batch, num_qubits  B >= 0 states of n (5..VQC_MAX_QUBITS) qubits.
 *   factors   host [5][8] doubles: factor q (row-major 2x2, (re, im) pairs)
 *             acts on qubit q; the stage is U_4 (x) ... (x) U_0 on qubits 0..4.
 *   psi_in, psi_out  device [B, 2^n] complex64, 16-byte aligned (may be equal).
 *   repeats   the stage is applied this many times to data kept on chip
 *             (psi_out = U^repeats psi_in), so that timing the call measures
 *             arithmetic rather than HBM traffic.
 *   stream    cudaStream_t.
 * Asynchronous.  A tensor-core completion wait that runs out (about a second)
 * is reported by the next vqc_sync_check as VQC_ERR_DEVICE_CHECK.  Errors:
 * VQC_ERR_INVALID_ARG, VQC_ERR_CUDA. */
vqc_status vqc_stage_apply(int32_t method, int32_t batch, int32_t num_qubits, const double* factors,
                           const void* psi_in, void* psi_out, int32_t repeats, void* stream);

/* Plan statistics (paths, stage counts, algorithmic flop and byte counts per
 * evaluation) for a batch of `batch` samples. */
vqc_status vqc_plan_info(const vqc_plan* plan, int32_t batch, vqc_plan_stats* out);

/* Serialise the host plan (fused ops, runs, constituents, term table and all
 * stage schedules) into buf.  *inout_bytes holds buf's capacity on entry and
 * the bytes needed on return; buf may be NULL to query the size.  The bytes
 * are a deterministic function of the vqc_compile arguments. */
vqc_status vqc_plan_export(const vqc_plan* plan, void* buf, size_t* inout_bytes);

/* Synchronise `stream` and report any CUDA error, then read (and clear) the
 * error word of every plan of this process on the current device: each kernel
 * checks its launch geometry against the plan before touching memory and, on
 * a mismatch (an engine bug, never the caller's data), records it there and
 * skips its work; such a record returns VQC_ERR_DEVICE_CHECK naming the
 * kernel kind. */
vqc_status vqc_sync_check(void* stream);

/* Thread-local message of the last failing call ("" if none). */
const char* vqc_last_error(void);

/* VQC_ABI_VERSION of the loaded library. */
int32_t vqc_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* VQC_ABI_H_INCLUDED */
