/*
 * vqc_oracle.c -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously-correct complex128 statevector simulator used as the
 * correctness oracle for the GPU engine.  Only the test suite, the smoke entry
 * point and the benchmark's CPU-baseline leg may load it.  It shares no code,
 * header, table or constant with the CUDA path.
 *
 * What it computes (paper, Alg. 1 and Sec. 3 "Compile-Once Lowering and
 * Execution" / "Gate Application and Differentiation"):
 *   psi_G = U_G ... U_1 psi_0            (psi_0 = |0...0> unless given)
 *   E[b,j] = sum_k (-1)^{k_j} |psi_G[b,k]|^2   (Alg. 1, return statement)
 * and the exact gradient of L = sum_{b,j} gE[b,j] * E[b,j] with respect to the
 * per-sample angles x[b,.] and the shared angles w[.] (Sec. 3, gradients with
 * respect to trainable parameters).  The paper obtains this gradient with
 * autograd; the oracle obtains it with the adjoint recursion written with
 * explicit derivative matrices dU/dp (no generator shortcut), one gate at a
 * time, in time order reversed.
 *
 * Conventions (the paper does not print them; its semantic reference is Qiskit,
 * Sec. 4 "Preprocessing and Semantic Validation"):
 *   - qubit q is bit q of the amplitude index (little endian);
 *   - a circuit is listed in time order (first gate applied first);
 *   - 1q matrices act on the pair (bit q = 0, bit q = 1);
 *   - 2q matrices act on the local index s = b0 + 2*b1, b0 = bit of the first
 *     qubit (control for CX/CRZ), b1 = bit of the second qubit (target);
 *   - RX/RY/RZ(t) = exp(-i t P / 2); U3 is Qiskit's U(theta, phi, lambda);
 *     CRZ(t) = |0><0| x I + |1><1| x RZ(t); RZZ(t) = exp(-i t Z x Z / 2).
 *
 * Arithmetic is in double precision throughout.  Each gate is applied to the
 * full state by a loop over index pairs (1q) or index quadruples (2q) with the
 * gate's dense 2x2 or 4x4 matrix.
 */
#define _DEFAULT_SOURCE 1
#include <complex.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef double complex cplx;

/* Oracle opcodes (its own numbering; the Python wrapper maps gate names). */
enum {
    OR_H = 0, OR_X, OR_Y, OR_Z, OR_S, OR_T, OR_SX,
    OR_RX, OR_RY, OR_RZ, OR_U3,
    OR_CX, OR_CZ, OR_SWAP, OR_CRZ, OR_RZZ,
    OR_NUM_OPS
};

/* Parameter-source kinds for each of a gate's (up to) three angles. */
enum { OR_P_NONE = 0, OR_P_CONST = 1, OR_P_X = 2, OR_P_W = 3 };

static int op_arity(int op) { return op >= OR_CX ? 2 : 1; }

static int op_nparams(int op)
{
    switch (op) {
    case OR_RX: case OR_RY: case OR_RZ: case OR_CRZ: case OR_RZZ: return 1;
    case OR_U3: return 3;
    default: return 0;
    }
}

/* Dense matrix of a gate, row-major, dimension d = 2 (1q) or 4 (2q).
 * Returns d.  th[] holds the gate's angles (unused entries ignored). */
static int gate_matrix(int op, const double* th, cplx* U)
{
    const double r2 = 1.0 / sqrt(2.0);
    double c, s;
    int d = op_arity(op) == 1 ? 2 : 4;
    for (int i = 0; i < d * d; ++i) U[i] = 0.0;
    switch (op) {
    case OR_H:  U[0] = r2; U[1] = r2; U[2] = r2; U[3] = -r2; break;
    case OR_X:  U[1] = 1.0; U[2] = 1.0; break;
    case OR_Y:  U[1] = -I; U[2] = I; break;
    case OR_Z:  U[0] = 1.0; U[3] = -1.0; break;
    case OR_S:  U[0] = 1.0; U[3] = I; break;
    case OR_T:  U[0] = 1.0; U[3] = cexp(I * M_PI / 4.0); break;
    case OR_SX: U[0] = 0.5 * (1.0 + I); U[1] = 0.5 * (1.0 - I);
                U[2] = 0.5 * (1.0 - I); U[3] = 0.5 * (1.0 + I); break;
    case OR_RX: c = cos(th[0] / 2); s = sin(th[0] / 2);
                U[0] = c; U[1] = -I * s; U[2] = -I * s; U[3] = c; break;
    case OR_RY: c = cos(th[0] / 2); s = sin(th[0] / 2);
                U[0] = c; U[1] = -s; U[2] = s; U[3] = c; break;
    case OR_RZ: U[0] = cexp(-I * th[0] / 2); U[3] = cexp(I * th[0] / 2); break;
    case OR_U3: c = cos(th[0] / 2); s = sin(th[0] / 2);
                U[0] = c;
                U[1] = -cexp(I * th[2]) * s;
                U[2] = cexp(I * th[1]) * s;
                U[3] = cexp(I * (th[1] + th[2])) * c; break;
    /* 2q: local index s = b0 + 2*b1, U[out*4 + in] */
    case OR_CX:   U[0] = 1; U[1 * 4 + 3] = 1; U[2 * 4 + 2] = 1; U[3 * 4 + 1] = 1; break;
    case OR_CZ:   U[0] = 1; U[5] = 1; U[10] = 1; U[15] = -1; break;
    case OR_SWAP: U[0] = 1; U[1 * 4 + 2] = 1; U[2 * 4 + 1] = 1; U[15] = 1; break;
    case OR_CRZ:  U[0] = 1; U[5] = cexp(-I * th[0] / 2); U[10] = 1;
                  U[15] = cexp(I * th[0] / 2); break;
    case OR_RZZ:  U[0] = cexp(-I * th[0] / 2); U[5] = cexp(I * th[0] / 2);
                  U[10] = cexp(I * th[0] / 2); U[15] = cexp(-I * th[0] / 2); break;
    default: return 0;
    }
    return d;
}

/* Derivative dU/d th[p] of a parametrised gate, written out by hand from the
 * matrices above.  Returns d, or 0 if the gate has no parameter p. */
static int gate_matrix_deriv(int op, const double* th, int p, cplx* D)
{
    double c, s;
    int d = op_arity(op) == 1 ? 2 : 4;
    if (p >= op_nparams(op)) return 0;
    for (int i = 0; i < d * d; ++i) D[i] = 0.0;
    switch (op) {
    case OR_RX: c = cos(th[0] / 2); s = sin(th[0] / 2);
                D[0] = -0.5 * s; D[1] = -0.5 * I * c; D[2] = -0.5 * I * c; D[3] = -0.5 * s; break;
    case OR_RY: c = cos(th[0] / 2); s = sin(th[0] / 2);
                D[0] = -0.5 * s; D[1] = -0.5 * c; D[2] = 0.5 * c; D[3] = -0.5 * s; break;
    case OR_RZ: D[0] = -0.5 * I * cexp(-I * th[0] / 2); D[3] = 0.5 * I * cexp(I * th[0] / 2); break;
    case OR_U3:
        c = cos(th[0] / 2); s = sin(th[0] / 2);
        if (p == 0) {          /* d/d theta */
            D[0] = -0.5 * s;
            D[1] = -cexp(I * th[2]) * 0.5 * c;
            D[2] = cexp(I * th[1]) * 0.5 * c;
            D[3] = -cexp(I * (th[1] + th[2])) * 0.5 * s;
        } else if (p == 1) {   /* d/d phi */
            D[2] = I * cexp(I * th[1]) * s;
            D[3] = I * cexp(I * (th[1] + th[2])) * c;
        } else {               /* d/d lambda */
            D[1] = -I * cexp(I * th[2]) * s;
            D[3] = I * cexp(I * (th[1] + th[2])) * c;
        }
        break;
    case OR_CRZ: D[5] = -0.5 * I * cexp(-I * th[0] / 2); D[15] = 0.5 * I * cexp(I * th[0] / 2); break;
    case OR_RZZ: D[0] = -0.5 * I * cexp(-I * th[0] / 2); D[5] = 0.5 * I * cexp(I * th[0] / 2);
                 D[10] = 0.5 * I * cexp(I * th[0] / 2); D[15] = -0.5 * I * cexp(-I * th[0] / 2); break;
    default: return 0;
    }
    return d;
}

/* out = M applied on the qubits (q0[, q1]) of the n-qubit state in (full
 * Hilbert-space operator I x ... x M x ... x I, little endian).  in != out. */
static void apply_local(int n, const cplx* M, int d, int q0, int q1,
                        const cplx* in, cplx* out)
{
    const int64_t dim = (int64_t)1 << n;
    if (d == 2) {
        const int64_t m0 = (int64_t)1 << q0;
        for (int64_t k = 0; k < dim; ++k) {
            if (k & m0) continue;
            cplx a = in[k], b = in[k | m0];
            out[k] = M[0] * a + M[1] * b;
            out[k | m0] = M[2] * a + M[3] * b;
        }
    } else {
        const int64_t m0 = (int64_t)1 << q0, m1 = (int64_t)1 << q1;
        for (int64_t k = 0; k < dim; ++k) {
            if ((k & m0) || (k & m1)) continue;
            int64_t idx[4] = { k, k | m0, k | m1, k | m0 | m1 };  /* s = b0 + 2 b1 */
            cplx v[4];
            for (int s = 0; s < 4; ++s) v[s] = in[idx[s]];
            for (int r = 0; r < 4; ++r) {
                cplx acc = 0.0;
                for (int s = 0; s < 4; ++s) acc += M[r * 4 + s] * v[s];
                out[idx[r]] = acc;
            }
        }
    }
}

static void dagger(const cplx* M, int d, cplx* Md)
{
    for (int r = 0; r < d; ++r)
        for (int c = 0; c < d; ++c) Md[c * d + r] = conj(M[r * d + c]);
}

typedef struct {
    int n, G;
    const int32_t* op; const int32_t* q0; const int32_t* q1;
    const int32_t* pkind; const int32_t* pidx; const double* pconst;  /* [G*3] */
    int Px, Pw;
} circuit_t;

/* Resolve the angles of gate g for sample row xb. */
static void gate_angles(const circuit_t* c, int g, const double* xb, const double* w, double* th)
{
    for (int p = 0; p < 3; ++p) {
        int kind = c->pkind[g * 3 + p], idx = c->pidx[g * 3 + p];
        th[p] = 0.0;
        if (kind == OR_P_CONST) th[p] = c->pconst[g * 3 + p];
        else if (kind == OR_P_X) th[p] = xb[idx];
        else if (kind == OR_P_W) th[p] = w[idx];
    }
}

static int validate(const circuit_t* c)
{
    if (c->n < 1 || c->n > 24 || c->G < 0) return -1;
    for (int g = 0; g < c->G; ++g) {
        int op = c->op[g];
        if (op < 0 || op >= OR_NUM_OPS) return -2;
        if (c->q0[g] < 0 || c->q0[g] >= c->n) return -3;
        if (op_arity(op) == 2 && (c->q1[g] < 0 || c->q1[g] >= c->n || c->q1[g] == c->q0[g])) return -3;
        for (int p = 0; p < op_nparams(op); ++p) {
            int kind = c->pkind[g * 3 + p], idx = c->pidx[g * 3 + p];
            if (kind == OR_P_X && (idx < 0 || idx >= c->Px)) return -4;
            if (kind == OR_P_W && (idx < 0 || idx >= c->Pw)) return -4;
            if (kind != OR_P_CONST && kind != OR_P_X && kind != OR_P_W) return -4;
        }
    }
    return 0;
}

/* Evolve one sample: psi (in/out) of dimension 2^n. tmp is scratch. */
static void evolve(const circuit_t* c, const double* xb, const double* w, cplx* psi, cplx* tmp)
{
    const int64_t dim = (int64_t)1 << c->n;
    cplx U[16]; double th[3];
    for (int g = 0; g < c->G; ++g) {
        gate_angles(c, g, xb, w, th);
        int d = gate_matrix(c->op[g], th, U);
        apply_local(c->n, U, d, c->q0[g], c->q1[g], psi, tmp);
        memcpy(psi, tmp, (size_t)dim * sizeof(cplx));
    }
}

static void init_state(int n, const double* psi0b, cplx* psi)
{
    const int64_t dim = (int64_t)1 << n;
    for (int64_t k = 0; k < dim; ++k)
        psi[k] = psi0b ? psi0b[2 * k] + I * psi0b[2 * k + 1] : (k == 0 ? 1.0 : 0.0);
}

/* E_j = sum_k (-1)^{k_j} |psi_k|^2 (Alg. 1, return statement). */
static void expect_z(int n, const cplx* psi, double* E)
{
    const int64_t dim = (int64_t)1 << n;
    for (int j = 0; j < n; ++j) {
        double acc = 0.0;
        for (int64_t k = 0; k < dim; ++k) {
            double p = creal(psi[k]) * creal(psi[k]) + cimag(psi[k]) * cimag(psi[k]);
            acc += ((k >> j) & 1) ? -p : p;
        }
        E[j] = acc;
    }
}

/* ---- public entry points (loaded by the test wrapper through ctypes) ---- */

int oracle_num_ops(void) { return OR_NUM_OPS; }

/* Dense matrix of one gate (d*d complex as interleaved doubles). Returns d. */
int oracle_gate_matrix(int op, const double* th, double* out)
{
    cplx U[16];
    int d = gate_matrix(op, th, U);
    for (int i = 0; i < d * d; ++i) { out[2 * i] = creal(U[i]); out[2 * i + 1] = cimag(U[i]); }
    return d;
}

int oracle_gate_matrix_deriv(int op, const double* th, int p, double* out)
{
    cplx D[16];
    int d = gate_matrix_deriv(op, th, p, D);
    for (int i = 0; i < d * d; ++i) { out[2 * i] = creal(D[i]); out[2 * i + 1] = cimag(D[i]); }
    return d;
}

/* Forward: E[B*n] and optionally the final states state[B*2^n*2].
 * psi0: NULL or [B*2^n*2] interleaved (re, im).  Returns 0 or a negative code. */
int oracle_forward(int n, int G, const int32_t* op, const int32_t* q0, const int32_t* q1,
                   const int32_t* pkind, const int32_t* pidx, const double* pconst,
                   int Px, int Pw, int B, const double* x, const double* w,
                   const double* psi0, double* E, double* state)
{
    circuit_t c = { n, G, op, q0, q1, pkind, pidx, pconst, Px, Pw };
    int rc = validate(&c);
    if (rc) return rc;
    const int64_t dim = (int64_t)1 << n;
    cplx* psi = (cplx*)malloc((size_t)dim * sizeof(cplx));
    cplx* tmp = (cplx*)malloc((size_t)dim * sizeof(cplx));
    if (!psi || !tmp) { free(psi); free(tmp); return -5; }
    for (int b = 0; b < B; ++b) {
        init_state(n, psi0 ? psi0 + (size_t)b * dim * 2 : NULL, psi);
        evolve(&c, x ? x + (size_t)b * Px : NULL, w, psi, tmp);
        expect_z(n, psi, E + (size_t)b * n);
        if (state)
            for (int64_t k = 0; k < dim; ++k) {
                state[((size_t)b * dim + k) * 2] = creal(psi[k]);
                state[((size_t)b * dim + k) * 2 + 1] = cimag(psi[k]);
            }
    }
    free(psi); free(tmp);
    return 0;
}

/* Adjoint backward: dx[B*Px] (overwritten) and dw[Pw] (overwritten, summed
 * over the batch) for L = sum_{b,j} gE[b,j] E[b,j].
 *
 *   psi_G  = forward state,  lam_G = O psi_G with O = sum_j gE_j Z_j.
 *   for g = G..1:  psi_{g-1} = U_g^dag psi_g
 *                  dL/dp += 2 Re <lam_g| dU_g/dp |psi_{g-1}>   (each angle p)
 *                  lam_{g-1} = U_g^dag lam_g
 */
int oracle_backward(int n, int G, const int32_t* op, const int32_t* q0, const int32_t* q1,
                    const int32_t* pkind, const int32_t* pidx, const double* pconst,
                    int Px, int Pw, int B, const double* x, const double* w,
                    const double* psi0, const double* gE, double* dx, double* dw)
{
    circuit_t c = { n, G, op, q0, q1, pkind, pidx, pconst, Px, Pw };
    int rc = validate(&c);
    if (rc) return rc;
    const int64_t dim = (int64_t)1 << n;
    cplx* psi = (cplx*)malloc((size_t)dim * sizeof(cplx));
    cplx* lam = (cplx*)malloc((size_t)dim * sizeof(cplx));
    cplx* tmp = (cplx*)malloc((size_t)dim * sizeof(cplx));
    if (!psi || !lam || !tmp) { free(psi); free(lam); free(tmp); return -5; }
    if (dx) memset(dx, 0, (size_t)B * Px * sizeof(double));
    if (dw) memset(dw, 0, (size_t)Pw * sizeof(double));
    cplx U[16], Ud[16], D[16]; double th[3];
    for (int b = 0; b < B; ++b) {
        const double* xb = x ? x + (size_t)b * Px : NULL;
        const double* gb = gE + (size_t)b * n;
        init_state(n, psi0 ? psi0 + (size_t)b * dim * 2 : NULL, psi);
        evolve(&c, xb, w, psi, tmp);
        for (int64_t k = 0; k < dim; ++k) {
            double o = 0.0;
            for (int j = 0; j < n; ++j) o += ((k >> j) & 1) ? -gb[j] : gb[j];
            lam[k] = o * psi[k];
        }
        for (int g = G - 1; g >= 0; --g) {
            gate_angles(&c, g, xb, w, th);
            int d = gate_matrix(op[g], th, U);
            dagger(U, d, Ud);
            apply_local(n, Ud, d, q0[g], q1[g], psi, tmp);   /* psi_{g-1} */
            memcpy(psi, tmp, (size_t)dim * sizeof(cplx));
            for (int p = 0; p < op_nparams(op[g]); ++p) {
                int kind = pkind[g * 3 + p], idx = pidx[g * 3 + p];
                if (kind != OR_P_X && kind != OR_P_W) continue;
                gate_matrix_deriv(op[g], th, p, D);
                apply_local(n, D, d, q0[g], q1[g], psi, tmp);  /* dU/dp psi_{g-1} */
                cplx ip = 0.0;
                for (int64_t k = 0; k < dim; ++k) ip += conj(lam[k]) * tmp[k];
                double term = 2.0 * creal(ip);
                if (kind == OR_P_X) { if (dx) dx[(size_t)b * Px + idx] += term; }
                else if (dw) dw[idx] += term;
            }
            apply_local(n, Ud, d, q0[g], q1[g], lam, tmp);   /* lam_{g-1} */
            memcpy(lam, tmp, (size_t)dim * sizeof(cplx));
        }
    }
    free(psi); free(lam); free(tmp);
    return 0;
}
