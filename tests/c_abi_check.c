/* The C ABI used from plain C (no Python, no torch): compile a small circuit,
 * query and export the plan, check the documented error codes and, when built
 * with VQC_CHECK_GPU and run on a CUDA device, evaluate it and compare E with
 * its closed form.
 *
 * Circuit (2 qubits): RY(x0) on q0, CX q0 -> q1, RZ(w0) on q1.  RY(t)|0> has
 * <Z> = cos t; the CX copies the Z value of q0 onto q1; RZ is diagonal and
 * leaves both unchanged: E[b] = (cos x[b], cos x[b]).
 *
 * The same circuit compiled for complex128 and for complex128 in double-float
 * arithmetic gives identical plan bytes and, on a device, E = cos x to 1e-12.
 *
 * Exit status 0 and a last line "ok" on success. */
#include <math.h>
#include <stdio.h>
#include <string.h>

#include "vqc.h"

#ifdef VQC_CHECK_GPU
#include <cuda_runtime.h>
#endif

static int fail(const char* what) {
    printf("FAILED: %s (%s)\n", what, vqc_last_error());
    return 1;
}

int main(void) {
    vqc_gate g[3];
    memset(g, 0, sizeof g);
    g[0].op = VQC_RY;
    g[0].q0 = 0;
    g[0].pkind[0] = VQC_P_X;
    g[0].pidx[0] = 0;
    g[1].op = VQC_CX;
    g[1].q0 = 0;
    g[1].q1 = 1;
    g[2].op = VQC_RZ;
    g[2].q0 = 1;
    g[2].pkind[0] = VQC_P_W;
    g[2].pidx[0] = 0;

    if (vqc_abi_version() != VQC_ABI_VERSION) return fail("abi version");
    vqc_plan* plan = NULL;
    if (vqc_compile(g, 3, 2, 1, 1, VQC_C64, &plan) != VQC_OK || !plan) return fail("vqc_compile");

    vqc_plan_stats st;
    if (vqc_plan_info(plan, 4, &st) != VQC_OK) return fail("vqc_plan_info");
    if (st.num_qubits != 2 || st.num_x != 1 || st.num_w != 1 || st.num_gates_in != 3 || st.num_terms != 2)
        return fail("plan statistics");

    size_t nbytes = 0;
    if (vqc_plan_export(plan, NULL, &nbytes) != VQC_OK || nbytes == 0) return fail("export size");
    static unsigned char blob[1 << 20];
    if (nbytes > sizeof blob) return fail("export too large");
    if (vqc_plan_export(plan, blob, &nbytes) != VQC_OK || memcmp(blob, "VQCP", 4) != 0)
        return fail("export bytes");
    size_t small = 4;
    if (vqc_plan_export(plan, blob, &small) != VQC_ERR_INVALID_ARG) return fail("export capacity check");

    /* complex128 with double-float arithmetic: the complex128 plan, reported as such */
    vqc_plan *p128 = NULL, *pdf = NULL;
    if (vqc_compile(g, 3, 2, 1, 1, VQC_C128, &p128) != VQC_OK ||
        vqc_compile(g, 3, 2, 1, 1, VQC_C128_DF, &pdf) != VQC_OK)
        return fail("vqc_compile complex128");
    {
        static unsigned char b1[1 << 20], b2[1 << 20];
        size_t n1 = sizeof b1, n2 = sizeof b2;
        if (vqc_plan_export(p128, b1, &n1) != VQC_OK || vqc_plan_export(pdf, b2, &n2) != VQC_OK ||
            n1 != n2 || memcmp(b1, b2, n1) != 0)
            return fail("double-float plan bytes");
        vqc_plan_stats s2;
        if (vqc_plan_info(pdf, 4, &s2) != VQC_OK || s2.dtype != VQC_C128_DF) return fail("double-float dtype");
    }

    /* documented errors of vqc_compile */
    vqc_plan* bad = NULL;
    vqc_gate h = g[1];
    h.q1 = 0; /* q0 == q1 */
    if (vqc_compile(&h, 1, 2, 0, 0, VQC_C64, &bad) != VQC_ERR_QUBIT_RANGE || bad) return fail("q0 == q1");
    h = g[0];
    h.op = 99;
    if (vqc_compile(&h, 1, 2, 1, 0, VQC_C64, &bad) != VQC_ERR_UNSUPPORTED_GATE) return fail("bad opcode");
    h = g[0];
    h.pidx[0] = 5; /* x column beyond num_x */
    if (vqc_compile(&h, 1, 2, 1, 0, VQC_C64, &bad) != VQC_ERR_PARAM_RANGE) return fail("param range");
    if (vqc_compile(g, 3, VQC_MAX_QUBITS + 1, 1, 1, VQC_C64, &bad) != VQC_ERR_TOO_MANY_QUBITS)
        return fail("too many qubits");
    if (vqc_compile(g, 3, 2, 1, 1, VQC_C64, NULL) != VQC_ERR_INVALID_ARG) return fail("NULL out_plan");

#ifdef VQC_CHECK_GPU
    {
        enum { B = 5 };
        float hx[B], hw[1] = {0.7f}, hE[B * 2];
        for (int b = 0; b < B; ++b) hx[b] = -2.0f + 0.9f * (float)b;
        float *dx = NULL, *dw = NULL, *dE = NULL;
        if (cudaMalloc((void**)&dx, sizeof hx) != cudaSuccess || cudaMalloc((void**)&dw, sizeof hw) != cudaSuccess ||
            cudaMalloc((void**)&dE, sizeof hE) != cudaSuccess)
            return fail("cudaMalloc");
        cudaMemcpy(dx, hx, sizeof hx, cudaMemcpyHostToDevice);
        cudaMemcpy(dw, hw, sizeof hw, cudaMemcpyHostToDevice);
        if (vqc_workspace_bytes(plan, B, 0) != 0) return fail("forward workspace");
        if (vqc_forward(plan, B, dx, dw, NULL, dE, NULL, NULL, 0, NULL) != VQC_OK) return fail("vqc_forward");
        if (vqc_sync_check(NULL) != VQC_OK) return fail("vqc_sync_check");
        cudaMemcpy(hE, dE, sizeof hE, cudaMemcpyDeviceToHost);
        for (int b = 0; b < B; ++b) {
            const double c = cos((double)hx[b]);
            if (fabs(hE[2 * b] - c) > 1e-5 || fabs(hE[2 * b + 1] - c) > 1e-5) return fail("E closed form");
        }
        /* host buffers through vqc_evaluate_host: same E */
        float hE2[B * 2];
        if (vqc_evaluate_host(plan, B, hx, hw, NULL, hE2, NULL, NULL, NULL) != VQC_OK)
            return fail("vqc_evaluate_host");
        for (int i = 0; i < 2 * B; ++i)
            if (hE2[i] != hE[i]) return fail("host evaluation differs");
        cudaFree(dx);
        cudaFree(dw);
        cudaFree(dE);
        /* complex128, native and double-float, from host buffers: E = cos x to 1e-12 */
        double x2[B], w2[1] = {0.7}, e128[B * 2], edf[B * 2];
        for (int b = 0; b < B; ++b) x2[b] = -2.0 + 0.9 * b;
        if (vqc_evaluate_host(p128, B, x2, w2, NULL, e128, NULL, NULL, NULL) != VQC_OK ||
            vqc_evaluate_host(pdf, B, x2, w2, NULL, edf, NULL, NULL, NULL) != VQC_OK)
            return fail("vqc_evaluate_host complex128");
        for (int b = 0; b < B; ++b)
            for (int j = 0; j < 2; ++j)
                if (fabs(e128[2 * b + j] - cos(x2[b])) > 1e-12 || fabs(edf[2 * b + j] - cos(x2[b])) > 1e-12)
                    return fail("complex128 E closed form");
        printf("gpu ok\n");
    }
#endif
    vqc_free(plan);
    vqc_free(p128);
    vqc_free(pdf);
    vqc_free(NULL);
    printf("ok\n");
    return 0;
}
