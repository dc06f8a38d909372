// sweep.cuh -- sm_103a kernels of the batched statevector engine.
//
// Forward (paper, Alg. 1 execute phase): per sample, psi = U_G ... U_1 psi0
// and E[b, j] = sum_k (-1)^{k_j} |psi[k]|^2 (Alg. 1, return statement).
// Backward (paper, Sec. 3, gradients w.r.t. trainable parameters), adjoint
// method: lam = O psi with O = sum_j gE[b, j] Z_j; the plan is swept in
// reverse, un-applying every op on psi and lam, and for every parametrised
// angle t of a gate exp(-i t P / 2) the term dL/dt = Im <lam|P|psi> is taken
// at the gate's output.  For a fused single-qubit run V the kernel
// accumulates rho = sum_pairs psi_pair lam_pair^dag (a 2x2 matrix) once at
// the run's output; each constituent j of the run then gives
// dL/dt_j = Im Tr(W_j P_j W_j^dag rho) with W_j the constituents after j.
//
// Execution model ("resident" path).  A sample's state lives in shared
// memory.  A group of T = 2^(n-K) threads owns one sample; in each stage a
// thread loads the 2^K amplitudes spanned by the stage's K active qubits into
// registers (its block; the other n-K index bits come from the thread index),
// applies all of the stage's ops there, and stores the block back.  Blocks of
// different threads are disjoint, so one group barrier per stage suffices.
// Gate matrices are evaluated once per sample (sincos once per angle) into a
// shared-memory table before the sweep.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

#include "dd.cuh"
#include "plan.h"

namespace vqc {

template <typename R> struct V2;
template <> struct V2<float> { using t = float2; };
template <> struct V2<double> { using t = double2; };
template <> struct V2<dd> { using t = dd2; };
template <typename R> using C2 = typename V2<R>::t;

// The real type arrays have outside a kernel (caller memory, workspaces,
// partials) for the kernel's arithmetic type R: R itself, except double for
// double-float kernels, which split values on reading and rejoin them on
// writing.  For float and double every conversion below is the identity.
template <typename R> struct StoreOf { using t = R; };
template <> struct StoreOf<dd> { using t = double; };
template <typename R> using St = typename StoreOf<R>::t;
template <typename R> using SC2 = C2<St<R>>;

template <typename R, typename T>
__device__ __forceinline__ R as_r(T v) {
    if constexpr (std::is_same<T, R>::value) return v;
    else return R(v);
}
template <typename O, typename R>
__device__ __forceinline__ O as_out(R v) {
    if constexpr (std::is_same<O, R>::value) return v;
    else return v.to_double();
}
template <typename R>
__device__ __forceinline__ C2<R> c2_in(SC2<R> v) {
    if constexpr (std::is_same<St<R>, R>::value) return v;
    else { C2<R> r; r.x = R(v.x); r.y = R(v.y); return r; }
}
template <typename R>
__device__ __forceinline__ SC2<R> c2_out(C2<R> v) {
    if constexpr (std::is_same<St<R>, R>::value) return v;
    else { SC2<R> r; r.x = v.x.to_double(); r.y = v.y.to_double(); return r; }
}

template <typename R>
__device__ __forceinline__ C2<R> cm(R x, R y) { C2<R> r; r.x = x; r.y = y; return r; }

template <typename R>
__device__ __forceinline__ C2<R> cmul(C2<R> a, C2<R> b) {
    return cm<R>(fma(a.x, b.x, -a.y * b.y), fma(a.x, b.y, a.y * b.x));
}
// m0 * u + m1 * v
template <typename R>
__device__ __forceinline__ C2<R> cmv2(C2<R> m0, C2<R> u, C2<R> m1, C2<R> v) {
    if constexpr (std::is_same<R, dd>::value) {   // each component one compensated dot product
        C2<R> r;
        r.x = dot4(m0.x, u.x, -m0.y, u.y, m1.x, v.x, -m1.y, v.y);
        r.y = dot4(m0.x, u.y, m0.y, u.x, m1.x, v.y, m1.y, v.x);
        return r;
    }
    R x = fma(m0.x, u.x, fma(-m0.y, u.y, fma(m1.x, v.x, -m1.y * v.y)));
    R y = fma(m0.x, u.y, fma(m0.y, u.x, fma(m1.x, v.y, m1.y * v.x)));
    return cm<R>(x, y);
}
template <typename R>
__device__ __forceinline__ C2<R> cconj(C2<R> a) { return cm<R>(a.x, -a.y); }

template <typename R> struct M2 { C2<R> a, b, c, d; };   // [[a, b], [c, d]]

template <typename R>
__device__ __forceinline__ M2<R> mmul(const M2<R>& p, const M2<R>& q) {   // p * q
    M2<R> r;
    r.a = cmv2<R>(p.a, q.a, p.b, q.c);
    r.b = cmv2<R>(p.a, q.b, p.b, q.d);
    r.c = cmv2<R>(p.c, q.a, p.d, q.c);
    r.d = cmv2<R>(p.c, q.b, p.d, q.d);
    return r;
}
template <typename R>
__device__ __forceinline__ M2<R> mdag(const M2<R>& p) {
    M2<R> r;
    r.a = cconj<R>(p.a); r.b = cconj<R>(p.c); r.c = cconj<R>(p.b); r.d = cconj<R>(p.d);
    return r;
}
template <typename R>
__device__ __forceinline__ M2<R> mident() {
    M2<R> r;
    r.a = cm<R>(1, 0); r.b = cm<R>(0, 0); r.c = cm<R>(0, 0); r.d = cm<R>(1, 0);
    return r;
}

// Plain load: plan arrays may live in shared memory (copied at kernel start)
// or, when too large, in global memory.
template <typename T>
__device__ __forceinline__ T vqc_ld(const T* p) { return *p; }

// Copy [src, src + bytes) (16-byte multiple) into shared memory; all loads are
// independent, so a CTA pulls the whole plan in about one memory latency.
__device__ __forceinline__ void copy_region(unsigned char* dst, const unsigned char* src, int bytes) {
    const uint4* s = reinterpret_cast<const uint4*>(src);
    uint4* d = reinterpret_cast<uint4*>(dst);
    for (int i = threadIdx.x; i < bytes / 16; i += blockDim.x) d[i] = s[i];
}

// Asynchronous global -> shared copies (cp.async, 4/8/16 bytes, both addresses
// aligned to the size).  They hold no registers while in flight, so a thread
// can issue all of a CTA's staging loads before the first wait; async_wait()
// then blocks until this thread's copies have landed (a __syncthreads must
// follow before other threads read them).
template <int BYTES>
__device__ __forceinline__ void async_copy(void* sdst, const void* gsrc) {
    const unsigned sa = static_cast<unsigned>(__cvta_generic_to_shared(sdst));
    asm volatile("cp.async.ca.shared.global [%0], [%1], %2;\n" ::"r"(sa), "l"(gsrc), "n"(BYTES)
                 : "memory");
}
__device__ __forceinline__ void async_wait() { asm volatile("cp.async.wait_all;\n" ::: "memory"); }

__device__ __forceinline__ void async_region(unsigned char* dst, const unsigned char* src, int bytes) {
    for (int i = threadIdx.x; i < bytes / 16; i += blockDim.x) async_copy<16>(dst + 16 * i, src + 16 * i);
}
template <typename T>
__device__ __forceinline__ void async_elem(T* sdst, const T* gsrc) {
    async_copy<sizeof(T)>(sdst, gsrc);
}

// Programmatic dependent launch.  Every kernel of the library is launched so
// that it may start while the previous kernel in the stream is finishing; it
// reads and writes no caller memory (inputs, outputs, workspace) before
// grid_dep_wait(), which returns once that kernel has completed and its writes
// are visible (immediately when the launch had no such predecessor).  Only the
// plan, which no kernel writes, is read before it.  grid_dep_launch() then lets
// the next kernel in the stream begin its own prologue.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() {
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

// Pointer into the shared copy of a plan region (or the global one).
template <typename T>
__device__ __forceinline__ const T* rebase(const T* g, const unsigned char* plan, int region_off,
                                           const unsigned char* sm_region) {
    if (!sm_region) return g;
    return reinterpret_cast<const T*>(sm_region +
                                      (reinterpret_cast<const unsigned char*>(g) - plan - region_off));
}

// sin and cos for complex64 table entries, written out so that the half-angle
// evaluation is a short chain of FMAs: Cody-Waite reduction t = k pi/2 + r
// with pi/2 split in three parts (the head has 8 significant bits, so k *
// head is exact for |k| < 2^16), |r| <= pi/4, then the Taylor polynomials of
// sin (through r^9) and cos (through r^10), whose truncation errors on
// [-pi/4, pi/4] are below 2e-9, and the quadrant of k.  The reduction is exact
// only while |k| < 2^16; arguments beyond |t| = 65536 (|k| <= 41722), and NaN,
// go to the library sincosf instead.  complex128 uses the library routine.
__device__ __forceinline__ void sc(float t, float* s, float* c) {
    if (!(fabsf(t) <= 65536.0f)) {
        sincosf(t, s, c);
        return;
    }
    const float k = rintf(t * 0.636619772367581343f);   // t / (pi/2)
    float r = fmaf(-k, 1.5703125f, t);
    r = fmaf(-k, 4.838267923332751e-4f, r);
    r = fmaf(-k, 2.5633440682570896e-12f, r);
    const float r2 = r * r;
    float ps = fmaf(r2, 2.75573192239858907e-6f, -1.98412698412698413e-4f);   // 1/9!, -1/7!
    ps = fmaf(r2, ps, 8.33333333333333333e-3f);                               // 1/5!
    ps = fmaf(r2, ps, -1.66666666666666667e-1f);                              // -1/3!
    const float sr = fmaf(r * r2, ps, r);
    float pc = fmaf(r2, -2.75573192239858907e-7f, 2.48015873015873016e-5f);   // -1/10!, 1/8!
    pc = fmaf(r2, pc, -1.38888888888888889e-3f);                              // -1/6!
    pc = fmaf(r2, pc, 4.16666666666666667e-2f);                               // 1/4!
    pc = fmaf(r2, pc, -0.5f);                                                 // -1/2!
    const float cr = fmaf(r2, pc, 1.0f);
    const int q = (int)k & 3;
    const float sv = (q & 1) ? cr : sr, cv = (q & 1) ? sr : cr;
    *s = (q & 2) ? -sv : sv;
    *c = ((q + 1) & 2) ? -cv : cv;
}
__device__ __forceinline__ void sc(double t, double* s, double* c) { sincos(t, s, c); }
// double-float: the library routine in double (once per angle), then split
__device__ __forceinline__ void sc(dd t, dd* s, dd* c) {
    double sd, cd;
    sincos(t.to_double(), &sd, &cd);
    *s = dd(sd);
    *c = dd(cd);
}

// ---------------------------------------------------------------- kernel args
// R here is the storage real type (kernels take KArgs<St<R>>).
template <typename R>
struct KArgs {
    // plan
    const DOp* ops;
    const DStage* stages;
    int nstages;
    const DEntry* entries;
    const int32_t* ps_list;   // per-sample entry ids
    const int32_t* sh_list;   // shared entry ids
    const DConst* consts;
    const R* cmat;
    const R* cang;
    const DAcc* accs;
    const int32_t* xocc_ptr;
    const int32_t* xocc;
    const int32_t* wocc_ptr;
    const int32_t* wocc;
    unsigned* err;
    int n, K, tbits, G, S;     // S = samples per CTA
    int tpg, bpt;              // threads per sample group, register blocks per thread (tpg * bpt = 2^tbits)
    int n_ps, n_sh, n_accs, n_terms, Px, Pw;
    // batch
    int B, nunits;
    const R* x;
    const R* w;
    const C2<R>* psi0;
    const C2<R>* psi_final;
    const R* gE;
    R* E;
    C2<R>* state_out;
    R* dx;
    R* dw;
    R* dw_part;          // [gridDim.x, Pw]
    unsigned* counter;
    // shared-memory carve-up (byte offsets)
    int sm_sh, sm_ps, sm_psi, sm_lam, sm_acc, sm_terms, sm_dw, sm_red;
    int sm_w, sm_xg;   // shared copies of w [Pw] and of the unit's x / gE rows [S][Px + n]
    // plan regions copied to shared memory at sm_plan when plan_smem is set:
    // table data [tab_off, tab_off + tab_bytes) and this schedule's
    // [sched_off, sched_off + sched_bytes) of the plan's device blob.
    const unsigned char* plan;
    int tab_off, tab_bytes, sched_off, sched_bytes, sm_plan, plan_smem;
    // cluster path only (cluster.cuh): log2 CTAs per sample, rank 0's <Z> gather area
    int cl, sm_ecl;
};

struct PlanPtrs {
    const DOp* ops;
    const DStage* stages;
    const DEntry* entries;
    const int32_t* ps_list;
    const int32_t* sh_list;
    const DConst* consts;
    const void* cmat;
    const void* cang;
    const DAcc* accs;
    const int32_t* xocc_ptr;
    const int32_t* xocc;
    const int32_t* wocc_ptr;
    const int32_t* wocc;
};

// ---------------------------------------------------------------- tables
// Reals per table entry.  complex64 stores each 2x2 run matrix U twice in the
// operand form of the packed-FP32 update (see m1_apply_f2w): U at [0, 16) and
// U^dag at [16, 32), each as the pairs (m, i m) = (Re m, Im m), (-Im m, Re m) of
// its four entries m.
// complex128 stores U once (8 reals).  Phase entries use the first 8 reals.
template <typename R> struct EntryWords { static constexpr int value = sizeof(R) == 4 ? 32 : 8; };


template <typename R>
__device__ __forceinline__ void store_matrix(const M2<R>& m, R* out) {
    if constexpr (sizeof(R) == 4) {   // 16-byte stores (entries are 128-byte aligned)
        const C2<R> e[4] = {m.a, m.b, m.c, m.d};
        const C2<R> d[4] = {cconj<R>(m.a), cconj<R>(m.c), cconj<R>(m.b), cconj<R>(m.d)};
        float4* o4 = reinterpret_cast<float4*>(out);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            o4[k] = make_float4(e[k].x, e[k].y, -e[k].y, e[k].x);        // (m, i m)
            o4[4 + k] = make_float4(d[k].x, d[k].y, -d[k].y, d[k].x);
        }
    } else {
        out[0] = m.a.x; out[1] = m.a.y; out[2] = m.b.x; out[3] = m.b.y;
        out[4] = m.c.x; out[5] = m.c.y; out[6] = m.d.x; out[7] = m.d.y;
    }
}
template <typename R, typename XI, typename WI>
__device__ __forceinline__ R angle_of(uint8_t src, int32_t idx, const XI* xb, const WI* w,
                                      const R* cang) {
    if (src == SRC_X) return as_r<R>(xb[idx]);
    if (src == SRC_W) return as_r<R>(w[idx]);
    return cang[idx];
}

// Matrix of one constituent of a run.
template <typename R, typename XI, typename WI>
__device__ __forceinline__ M2<R> constituent(const DConst& c, const XI* xb, const WI* w, const R* cang,
                             const R* cmat) {
    M2<R> u;
    if (c.kind == CK_CONST) {
        const R* m = cmat + 8 * c.idx0;
        u.a = cm<R>(m[0], m[1]); u.b = cm<R>(m[2], m[3]);
        u.c = cm<R>(m[4], m[5]); u.d = cm<R>(m[6], m[7]);
        return u;
    }
    R t = angle_of<R>(c.src0, c.idx0, xb, w, cang);
    if (c.kind == CK_GPHASE) t += angle_of<R>(c.src1, c.idx1, xb, w, cang);
    R s, co;
    sc(t * R(0.5), &s, &co);
    const C2<R> z = cm<R>(0, 0);
    switch (c.kind) {
    case CK_RX: u.a = cm<R>(co, 0); u.b = cm<R>(0, -s); u.c = cm<R>(0, -s); u.d = cm<R>(co, 0); break;
    case CK_RY: u.a = cm<R>(co, 0); u.b = cm<R>(-s, 0); u.c = cm<R>(s, 0); u.d = cm<R>(co, 0); break;
    case CK_RZ: u.a = cm<R>(co, -s); u.b = z; u.c = z; u.d = cm<R>(co, s); break;
    default:    u.a = cm<R>(co, s); u.b = z; u.c = z; u.d = cm<R>(co, s); break;   // CK_GPHASE
    }
    return u;
}

// Evaluate one table entry (8 reals) for sample row xb.
template <typename R, typename XI, typename WI>
__device__ __forceinline__ void eval_entry(const DEntry& e, const DConst* consts, const XI* xb, const WI* w,
                           const R* cang, const R* cmat, R* out) {
    if (e.phase) {
        const DConst c = consts[e.cfirst];
        R t = angle_of<R>(c.src0, c.idx0, xb, w, cang);
        R s, co;
        sc(t * R(0.5), &s, &co);
        if (c.kind == CK_CRZ) {
            out[0] = 1; out[1] = 0; out[2] = co; out[3] = -s;
            out[4] = 1; out[5] = 0; out[6] = co; out[7] = s;
        } else {   // CK_RZZ: parity 0 -> e^{-it/2}, parity 1 -> e^{it/2}
            out[0] = co; out[1] = -s; out[2] = co; out[3] = s;
            out[4] = co; out[5] = s; out[6] = co; out[7] = -s;
        }
        return;
    }
    M2<R> m = mident<R>();
    for (int k = 0; k < e.ccount; ++k) {
        const DConst c = consts[e.cfirst + k];
        m = mmul<R>(constituent<R>(c, xb, w, cang, cmat), m);
    }
    store_matrix<R>(m, out);
}

template <typename R>
__device__ __forceinline__ M2<R> load_m2(const R* p) {
    M2<R> m;
    m.a = cm<R>(p[0], p[1]); m.b = cm<R>(p[2], p[3]);
    m.c = cm<R>(p[4], p[5]); m.d = cm<R>(p[6], p[7]);
    return m;
}

// ---------------------------------------------------------------- block ops
// Pair (i0, i1) = (r with bit T clear, r with bit T set), p enumerates pairs.
template <int T>
__host__ __device__ constexpr int pair_lo(int p) { return ((p >> T) << (T + 1)) | (p & ((1 << T) - 1)); }

template <typename R, int K, int T>
__device__ __forceinline__ void m1_apply(C2<R> (&a)[1 << K], const M2<R>& m) {
#pragma unroll
    for (int p = 0; p < (1 << (K - 1)); ++p) {
        const int i0 = pair_lo<T>(p), i1 = i0 | (1 << T);
        C2<R> u = a[i0], v = a[i1];
        a[i0] = cmv2<R>(m.a, u, m.b, v);
        a[i1] = cmv2<R>(m.c, u, m.d, v);
    }
}

// Gradient accumulator of a fused run.  With rho = sum_pairs psi conj(lam)^T
// (2x2, rho[a][b] = psi_a conj(lam_b)), every term the run needs is
// Im Tr(P rho') for a Pauli P and rho' = W^dag rho W, i.e. it depends only on
// the traceless anti-Hermitian part of rho, (i/2)(tx X + ty Y + tz Z), and that
// part stays traceless anti-Hermitian under W^dag . W.  So three reals per
// thread are summed instead of rho's eight:
//   tx = Im(rho01 + rho10), ty = Re(rho01 - rho10), tz = Im(rho00 - rho11).
// One running sum per component: two partial sums (shorter FMA chains) held
// more registers and measured 2-4% slower in the backward kernels.
template <typename R, int K, int T>
__device__ __forceinline__ void m1_t3(const C2<R> (&ps)[1 << K], const C2<R> (&la)[1 << K],
                                      R (&v)[4]) {
    R xa = 0, ya = 0, za = 0;
#pragma unroll
    for (int p = 0; p < (1 << (K - 1)); ++p) {
        const int i0 = pair_lo<T>(p), i1 = i0 | (1 << T);
        const C2<R> u = ps[i0], w = ps[i1], q0 = la[i0], q1 = la[i1];
        // Im(u conj q1) + Im(w conj q0)
        xa = fma(u.y, q1.x, fma(-u.x, q1.y, fma(w.y, q0.x, fma(-w.x, q0.y, xa))));
        // Re(u conj q1) - Re(w conj q0)
        ya = fma(u.x, q1.x, fma(u.y, q1.y, fma(-w.x, q0.x, fma(-w.y, q0.y, ya))));
        // Im(u conj q0) - Im(w conj q1)
        za = fma(u.y, q0.x, fma(-u.x, q0.y, fma(-w.y, q1.x, fma(w.x, q1.y, za))));
    }
    v[0] += xa;
    v[1] += ya;
    v[2] += za;
}

// complex64 2x2 update with Blackwell's packed FP32 instructions (FFMA2 on
// (re, im) pairs), the operand pairs read directly from a table entry (w: 8
// float2 = a, i a, b, i b, c, i c, d, i d).  With each state component
// broadcast to both lanes,
//   m u = (u.re, u.re) * m + (u.im, u.im) * (i m)
// so a complex multiply-add is two FFMA2 and a pair update eight.  (The form
// with the table's (Re m, Re m), (-Im m, Im m) pairs needs the swapped state
// pair (u.im, u.re) instead and measured 2-8% slower.)
template <int K, int T>
__device__ __forceinline__ void m1_apply_f2w(float2 (&a)[1 << K], const float* wp) {
    const float4 w0 = *reinterpret_cast<const float4*>(wp);
    const float4 w1 = *reinterpret_cast<const float4*>(wp + 4);
    const float4 w2 = *reinterpret_cast<const float4*>(wp + 8);
    const float4 w3 = *reinterpret_cast<const float4*>(wp + 12);
    const float2 ar = make_float2(w0.x, w0.y), ai = make_float2(w0.z, w0.w);
    const float2 br = make_float2(w1.x, w1.y), bi = make_float2(w1.z, w1.w);
    const float2 cr = make_float2(w2.x, w2.y), ci = make_float2(w2.z, w2.w);
    const float2 dr = make_float2(w3.x, w3.y), di = make_float2(w3.z, w3.w);
#pragma unroll
    for (int p = 0; p < (1 << (K - 1)); ++p) {
        const int i0 = pair_lo<T>(p), i1 = i0 | (1 << T);
        const float2 u = a[i0], v = a[i1];
        // entries hold (m, i m): m u = u.re (m) + u.im (i m)
        const float2 ux = make_float2(u.x, u.x), uy = make_float2(u.y, u.y);
        const float2 vx = make_float2(v.x, v.x), vy = make_float2(v.y, v.y);
        float2 nu = __fmul2_rn(ar, ux);
        nu = __ffma2_rn(ai, uy, nu);
        nu = __ffma2_rn(br, vx, nu);
        nu = __ffma2_rn(bi, vy, nu);
        float2 nv = __fmul2_rn(cr, ux);
        nv = __ffma2_rn(ci, uy, nv);
        nv = __ffma2_rn(dr, vx, nv);
        nv = __ffma2_rn(di, vy, nv);
        a[i0] = nu;
        a[i1] = nv;
    }
}

// Apply the table entry at tp (forward: U; adjoint: U^dag).
template <typename R, int K, int T, bool ADJ>
__device__ __forceinline__ void m1_entry(C2<R> (&a)[1 << K], const R* tp) {
    if constexpr (sizeof(R) == 4) {
        m1_apply_f2w<K, T>(a, tp + (ADJ ? 16 : 0));
    } else {
        M2<R> m = load_m2<R>(tp);
        if (ADJ) m = mdag<R>(m);
        m1_apply<R, K, T>(a, m);
    }
}

// X on local T when the predicate holds (control outside the block).
template <typename R, int K, int T>
__device__ __forceinline__ void x_pred(C2<R> (&a)[1 << K], bool p) {
#pragma unroll
    for (int q = 0; q < (1 << (K - 1)); ++q) {
        const int i0 = pair_lo<T>(q), i1 = i0 | (1 << T);
        C2<R> u = a[i0], v = a[i1];
        a[i0] = p ? v : u;
        a[i1] = p ? u : v;
    }
}

template <typename R, int K>
__device__ __forceinline__ void x_pred_dispatch(int t, C2<R> (&a)[1 << K], bool p) {
    switch (t) {
    case 0: x_pred<R, K, 0>(a, p); break;
    case 1: if constexpr (K > 1) x_pred<R, K, 1>(a, p); break;
    case 2: if constexpr (K > 2) x_pred<R, K, 2>(a, p); break;
    case 3: if constexpr (K > 3) x_pred<R, K, 3>(a, p); break;
    case 4: if constexpr (K > 4) x_pred<R, K, 4>(a, p); break;
    default: break;
    }
}

// Negate amplitudes with local bits A and Bq set (when p) -- CZ inside the block.
template <typename R, int K, int A, int Bq>
__device__ __forceinline__ void z2_ll(C2<R> (&a)[1 << K]) {
#pragma unroll
    for (int r = 0; r < (1 << K); ++r)
        if (((r >> A) & 1) && ((r >> Bq) & 1)) a[r] = cm<R>(-a[r].x, -a[r].y);
}
template <typename R, int K, int A>
__device__ __forceinline__ void z1_pred(C2<R> (&a)[1 << K], bool p) {
    const R s = p ? R(-1) : R(1);
#pragma unroll
    for (int r = 0; r < (1 << K); ++r)
        if ((r >> A) & 1) a[r] = cm<R>(s * a[r].x, s * a[r].y);
}

template <typename R, int K>
__device__ __forceinline__ void cz_dispatch(int ra, int rb, uint32_t pb, C2<R> (&a)[1 << K]) {
    if (ra >= kRefPhys && rb >= kRefPhys) {
        const bool p = ((pb >> (ra - kRefPhys)) & (pb >> (rb - kRefPhys)) & 1u) != 0;
        const R s = p ? R(-1) : R(1);
#pragma unroll
        for (int r = 0; r < (1 << K); ++r) a[r] = cm<R>(s * a[r].x, s * a[r].y);
        return;
    }
    if (ra >= kRefPhys || rb >= kRefPhys) {
        const int l = ra >= kRefPhys ? rb : ra;
        const int ph = ra >= kRefPhys ? ra : rb;
        const bool p = ((pb >> (ph - kRefPhys)) & 1u) != 0;
        switch (l) {
        case 0: z1_pred<R, K, 0>(a, p); break;
        case 1: if constexpr (K > 1) z1_pred<R, K, 1>(a, p); break;
        case 2: if constexpr (K > 2) z1_pred<R, K, 2>(a, p); break;
        case 3: if constexpr (K > 3) z1_pred<R, K, 3>(a, p); break;
        case 4: if constexpr (K > 4) z1_pred<R, K, 4>(a, p); break;
        default: break;
        }
        return;
    }
    const int lo = ra < rb ? ra : rb, hi = ra < rb ? rb : ra;
#define VQC_ZCASE(A_, B_) \
    case A_ * 8 + B_: if constexpr (A_ < K && B_ < K) z2_ll<R, K, A_, B_>(a); break;
    switch (lo * 8 + hi) {
        VQC_ZCASE(0, 1) VQC_ZCASE(0, 2) VQC_ZCASE(0, 3) VQC_ZCASE(0, 4)
        VQC_ZCASE(1, 2) VQC_ZCASE(1, 3) VQC_ZCASE(1, 4)
        VQC_ZCASE(2, 3) VQC_ZCASE(2, 4) VQC_ZCASE(3, 4)
        default: break;
    }
#undef VQC_ZCASE
}

__device__ __forceinline__ int refbit(int ref, int r, uint32_t pb) {
    return ref >= kRefPhys ? (int)((pb >> (ref - kRefPhys)) & 1u) : ((r >> ref) & 1);
}

// ---------------------------------------------------------------- reductions
// Butterfly exchange with lane ^ m (double-float: both parts).
template <typename R>
__device__ __forceinline__ R shx(R v, int m, unsigned mask) {
    if constexpr (std::is_same<R, dd>::value)
        return dd(__shfl_xor_sync(mask, v.hi, m), __shfl_xor_sync(mask, v.lo, m));
    else
        return __shfl_xor_sync(mask, v, m);
}

// Reduce 4 values over a group of `lanes` lanes (power of two <= 32) and write
// the 4 sums to dst[0..3] (reduce-scatter: 2 + 1 exchanges, then plain steps).
template <typename R>
__device__ __forceinline__ void reduce4_store(R (&v)[4], int lanes, int lane, R* dst,
                                              unsigned mask, bool add) {
    int u0 = 0, u1 = 0;
    if (lanes >= 2) {
        const int m = lanes >> 1;
        u0 = (lane & m) ? 1 : 0;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            R send = u0 ? v[i] : v[i + 2];
            R keep = u0 ? v[i + 2] : v[i];
            v[i] = keep + shx<R>(send, m, mask);
        }
    }
    if (lanes >= 4) {
        const int m = lanes >> 2;
        u1 = (lane & m) ? 1 : 0;
        R send = u1 ? v[0] : v[1];
        R keep = u1 ? v[1] : v[0];
        v[0] = keep + shx<R>(send, m, mask);
        for (int mm = lanes >> 3; mm >= 1; mm >>= 1) v[0] += shx<R>(v[0], mm, mask);
        if ((lane & ((lanes >> 2) - 1)) == 0) {
            R* d = dst + 2 * u0 + u1;
            *d = add ? *d + v[0] : v[0];
        }
    } else if (lanes == 2) {
        for (int i = 0; i < 2; ++i) dst[2 * u0 + i] = add ? dst[2 * u0 + i] + v[i] : v[i];
    } else {
        for (int i = 0; i < 4; ++i) dst[i] = add ? dst[i] + v[i] : v[i];
    }
}

// reduce4_store for a full warp, branch-free: 2 + 1 scatter shuffles and 3
// plain ones; lanes with (lane & 7) == 0 write their sum.
template <typename R>
__device__ __forceinline__ void reduce4_full(R (&v)[4], int lane, R* dst, bool add) {
    const unsigned full = 0xffffffffu;
    const int u0 = (lane >> 4) & 1, u1 = (lane >> 3) & 1;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const R send = u0 ? v[i] : v[i + 2];
        const R keep = u0 ? v[i + 2] : v[i];
        v[i] = keep + shx<R>(send, 16, full);
    }
    {
        const R send = u1 ? v[0] : v[1];
        const R keep = u1 ? v[1] : v[0];
        v[0] = keep + shx<R>(send, 8, full);
    }
    v[0] += shx<R>(v[0], 4, full);
    v[0] += shx<R>(v[0], 2, full);
    v[0] += shx<R>(v[0], 1, full);
    if ((lane & 7) == 0) {
        R* d = dst + 2 * u0 + u1;
        *d = add ? *d + v[0] : v[0];
    }
}

template <typename R>
__device__ __forceinline__ R reduce1(R v, int lanes, unsigned mask) {
    for (int m = lanes >> 1; m >= 1; m >>= 1) v += shx<R>(v, m, mask);
    return v;
}

// ---------------------------------------------------------------- addressing
struct Geo {
    int T;        // threads per sample group
    int lanes;    // min(T, 32)
    int wg;       // warps per group (>= 1)
    int g;        // group (sample slot) index in the CTA
    int t;        // thread index in the group
    int h;        // per-sample XOR on the slot index (bank spreading of small groups)
    unsigned mask;   // lanes of this warp that exist (a CTA smaller than a warp)
};

__device__ __forceinline__ uint32_t swz(uint32_t u, int G) {
    uint32_t v = u >> G, f = 0;
    while (v) { f ^= v; v >>= G; }
    return u ^ (f & ((1u << G) - 1));
}

template <typename R>
__device__ __forceinline__ void group_sync(const Geo& q) {
    if (q.T > 32) __syncthreads(); else __syncwarp(q.mask);
}

template <int K>
__device__ __forceinline__ uint32_t block_off(int r, const int32_t (&sg)[K]) {
    uint32_t o = 0;
#pragma unroll
    for (int j = 0; j < K; ++j)
        if ((r >> j) & 1) o ^= (uint32_t)sg[j];
    return o;
}

struct StageView {
    uint32_t swb, pb;
};

// XOR of the entries of v[0 .. 16) selected by the set bits of t, with all
// loads independent (no loop-carried branch): a thread's slot base.  Entries
// past the stage's thread bits are zero in the record, and t has no bits there.
__device__ __forceinline__ uint32_t xor_select(const int32_t* v, int nb, int t) {
    uint32_t b = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) b ^= ((t >> i) & 1) ? (uint32_t)vqc_ld(&v[i]) : 0u;
    if (nb > 8) {
#pragma unroll
        for (int i = 8; i < kMaxThreadBits; ++i) b ^= ((t >> i) & 1) ? (uint32_t)vqc_ld(&v[i]) : 0u;
    }
    return b;
}

template <int K>
__device__ __forceinline__ StageView stage_view(const DStage* sp, int t, int h, int32_t (&sg)[K]) {
#pragma unroll
    for (int j = 0; j < K; ++j) sg[j] = vqc_ld(&sp->sigma[j]);
    const int nb = vqc_ld(&sp->nthreadbits);   // uint8 load
    StageView v;
    v.swb = (uint32_t)h ^ xor_select(sp->tau, nb, t);
    v.pb = xor_select(reinterpret_cast<const int32_t*>(sp->tmask), nb, t);   // disjoint bits
    return v;
}

// Slot base of thread t and the local offsets of a stage's load map (ST false)
// or store map (ST true), read from the stage record.
template <int K, bool ST>
__device__ __forceinline__ uint32_t map_base(const DStage* sp, int t, int h, int32_t (&sg)[K]) {
    const int32_t* sig = ST ? sp->sigma_st : sp->sigma;
#pragma unroll
    for (int j = 0; j < K; ++j) sg[j] = vqc_ld(&sig[j]);
    const int nb = vqc_ld(&sp->nthreadbits);
    return (uint32_t)h ^ xor_select(ST ? sp->tau_st : sp->tau, nb, t);
}

template <typename R, int K>
__device__ __forceinline__ void block_load(C2<R> (&a)[1 << K], const C2<R>* st, uint32_t swb,
                                           const int32_t (&sg)[K]) {
#pragma unroll
    for (int r = 0; r < (1 << K); ++r) a[r] = st[swb ^ block_off<K>(r, sg)];
}
// The store recomputes the 2^K slot offsets (an empty asm hides swb's value
// from the compiler) instead of keeping the load's offsets live in registers
// across the stage's ops.
template <typename R, int K>
__device__ __forceinline__ void block_store(const C2<R> (&a)[1 << K], C2<R>* st, uint32_t swb,
                                            const int32_t (&sg)[K]) {
    asm volatile("" : "+r"(swb));
    int32_t s2[K];
#pragma unroll
    for (int j = 0; j < K; ++j) {
        s2[j] = sg[j];
        asm volatile("" : "+r"(s2[j]));
    }
#pragma unroll
    for (int r = 0; r < (1 << K); ++r) st[swb ^ block_off<K>(r, s2)] = a[r];
}

// Diagonal two-qubit phase (CRZ, RZZ): amplitude r is multiplied by ph[s],
// s = bit a + 2 bit b (a, b = the gate's first and second qubit), conjugated in
// the backward, where the gradient term Im <lam|P|psi> = sum_r g[s] Im(conj(lam_r)
// psi_r) is taken first (g = the generator's diagonal: CRZ (0, 1, 0, -1), RZZ
// (1, -1, -1, 1)).  Three forms by where a and b live; each resolves s per
// amplitude at compile time except for one per-op selection.
template <typename R>
__device__ __forceinline__ void ph2_gen(uint8_t flags, R (&g)[4]) {
    if (flags & OPF_GEN_CRZ) { g[0] = 0; g[1] = 1; g[2] = 0; g[3] = -1; }
    else { g[0] = 1; g[1] = -1; g[2] = -1; g[3] = 1; }
}
template <typename R>
__device__ __forceinline__ R gen_at(uint8_t flags, int s) {   // g[s] for a runtime s
    if (flags & OPF_GEN_CRZ) return s == 1 ? R(1) : s == 3 ? R(-1) : R(0);
    return (s == 0 || s == 3) ? R(1) : R(-1);
}
template <typename R>
__device__ __forceinline__ R im_conj_mul(const C2<R>& la, const C2<R>& ps) {
    return la.x * ps.y - la.y * ps.x;
}
template <typename R, bool FULL>
__device__ __forceinline__ void ph2_term_store(R tv, const Geo& q, R* accp, bool acc_add) {
    if (FULL) {
#pragma unroll
        for (int m = 16; m >= 1; m >>= 1) tv += shx<R>(tv, m, 0xffffffffu);
    } else {
        tv = reduce1<R>(tv, q.lanes, q.mask);
    }
    if ((q.t & (q.lanes - 1)) == 0) accp[0] = acc_add ? accp[0] + tv : tv;
}
template <typename R, int K, int MODE, bool FULL, int LO, int HI>
__device__ __forceinline__ void ph2_ll(bool swapped, const R* tp, uint8_t flags,
                                       C2<R> (&a)[1 << K], C2<R> (&l)[1 << K], const Geo& q,
                                       R* accp, bool acc_add) {
    // index by (bit LO) + 2 (bit HI): swap entries 1 and 2 when a is the higher position
    C2<R> ph[4] = {cm<R>(tp[0], tp[1]), cm<R>(tp[2], tp[3]), cm<R>(tp[4], tp[5]), cm<R>(tp[6], tp[7])};
    R g[4];
    ph2_gen<R>(flags, g);
    if (swapped) {
        const C2<R> t = ph[1]; ph[1] = ph[2]; ph[2] = t;
        const R u = g[1]; g[1] = g[2]; g[2] = u;
    }
    if (MODE == 1) {
#pragma unroll
        for (int s = 0; s < 4; ++s) ph[s].y = -ph[s].y;
        if (flags & OPF_HAS_ACC) {
            R tv = 0;
#pragma unroll
            for (int r = 0; r < (1 << K); ++r)
                tv = fma(g[((r >> LO) & 1) + 2 * ((r >> HI) & 1)], im_conj_mul<R>(l[r], a[r]), tv);
            ph2_term_store<R, FULL>(tv, q, accp, acc_add);
        }
    }
#pragma unroll
    for (int r = 0; r < (1 << K); ++r) {
        const int s = ((r >> LO) & 1) + 2 * ((r >> HI) & 1);
        a[r] = cmul<R>(a[r], ph[s]);
        if (MODE == 1) l[r] = cmul<R>(l[r], ph[s]);
    }
}
template <typename R, int K, int MODE, bool FULL, int L>
__device__ __forceinline__ void ph2_pl(bool a_local, bool p, const R* tp, uint8_t flags,
                                       C2<R> (&a)[1 << K], C2<R> (&l)[1 << K], const Geo& q,
                                       R* accp, bool acc_add) {
    // s = bit L + 2 p (a local) or p + 2 bit L (b local)
    const int s0 = a_local ? 2 * (int)p : (int)p, s1 = a_local ? 1 + 2 * (int)p : (int)p + 2;
    C2<R> f0 = cm<R>(tp[2 * s0], tp[2 * s0 + 1]), f1 = cm<R>(tp[2 * s1], tp[2 * s1 + 1]);
    const R g0 = gen_at<R>(flags, s0), g1 = gen_at<R>(flags, s1);
    if (MODE == 1) {
        f0.y = -f0.y;
        f1.y = -f1.y;
        if (flags & OPF_HAS_ACC) {
            R tv = 0;
#pragma unroll
            for (int r = 0; r < (1 << K); ++r)
                tv = fma(((r >> L) & 1) ? g1 : g0, im_conj_mul<R>(l[r], a[r]), tv);
            ph2_term_store<R, FULL>(tv, q, accp, acc_add);
        }
    }
#pragma unroll
    for (int r = 0; r < (1 << K); ++r) {
        const C2<R> f = ((r >> L) & 1) ? f1 : f0;
        a[r] = cmul<R>(a[r], f);
        if (MODE == 1) l[r] = cmul<R>(l[r], f);
    }
}
template <typename R, int K, int MODE, bool FULL>
__device__ __forceinline__ void ph2_pp(int s, const R* tp, uint8_t flags, C2<R> (&a)[1 << K],
                                       C2<R> (&l)[1 << K], const Geo& q, R* accp, bool acc_add) {
    C2<R> f = cm<R>(tp[2 * s], tp[2 * s + 1]);
    if (MODE == 1) {
        f.y = -f.y;
        if (flags & OPF_HAS_ACC) {
            R tv = 0;
#pragma unroll
            for (int r = 0; r < (1 << K); ++r) tv += im_conj_mul<R>(l[r], a[r]);
            ph2_term_store<R, FULL>(gen_at<R>(flags, s) * tv, q, accp, acc_add);
        }
    }
#pragma unroll
    for (int r = 0; r < (1 << K); ++r) {
        a[r] = cmul<R>(a[r], f);
        if (MODE == 1) l[r] = cmul<R>(l[r], f);
    }
}

// ---------------------------------------------------------------- op dispatch
template <typename R> __device__ __forceinline__ M2<R> load_m2v(const R* p);
template <> __device__ __forceinline__ M2<float> load_m2v<float>(const float* p) {
    const float4 u = *reinterpret_cast<const float4*>(p);
    const float4 v = *reinterpret_cast<const float4*>(p + 4);
    M2<float> m;
    m.a = make_float2(u.x, u.y); m.b = make_float2(u.z, u.w);
    m.c = make_float2(v.x, v.y); m.d = make_float2(v.z, v.w);
    return m;
}
template <> __device__ __forceinline__ M2<double> load_m2v<double>(const double* p) {
    const double2* q = reinterpret_cast<const double2*>(p);
    M2<double> m;
    m.a = q[0]; m.b = q[1]; m.c = q[2]; m.d = q[3];
    return m;
}
template <> __device__ __forceinline__ M2<dd> load_m2v<dd>(const dd* p) {
    const dd2* q = reinterpret_cast<const dd2*>(p);
    M2<dd> m;
    m.a = q[0]; m.b = q[1]; m.c = q[2]; m.d = q[3];
    return m;
}

__device__ __forceinline__ bool physbit(uint32_t pb, int ref) {
    return ((pb >> (ref - kRefPhys)) & 1u) != 0;
}

// Apply op `raw` to the block(s).  MODE 0: forward on a.  MODE 1: backward --
// accumulate the op's gradient slot, then un-apply on a (psi) and l (lam).
// One switch over the dispatch code; every case has fixed local positions.
// WITH_CX: the schedule may hold CX ops (HBM passes); resident schedules fold
// every CX into stage store maps, and leaving those cases out of the switch
// keeps the other cases' register allocation tight.  A pass schedule holds
// only CX gates whose control lies outside the tile (the compiler folds every
// CX with both qubits in the tile into a store map), so the switch has no case
// for a local control: its code alone made the pass kernels spill (about 2.5x
// the spill traffic under the 128-register cap).
// WITH_PH2: the schedule may hold diagonal two-qubit phase ops (CRZ, RZZ).
// Kernels for plans without them are instantiated with the cases left out:
// their register allocation then needs fewer spills (measured 8-11% faster on
// the 12-qubit resident sweeps and the 16-qubit forward passes); the launch
// code picks the instantiation from the plan.
template <typename R, int K, int MODE, bool WITH_CX, bool FULL, bool WITH_PH2 = true>
__device__ __forceinline__ void apply_op(uint2 raw, uint32_t pb, C2<R> (&a)[1 << K],
                                         C2<R> (&l)[1 << K], const R* sh_tab, const R* ps_tab,
                                         R* acc, const Geo& q, int lane, int warp_in_group,
                                         bool acc_add) {
    const int code = raw.x & 0xff, ra = (raw.x >> 8) & 0xff, rb = (raw.x >> 16) & 0xff;
    const int flags = raw.x >> 24, slot = raw.y & 0xffff, aux = raw.y >> 16;
    const R* tp = ((flags & OPF_PER_SAMPLE) ? ps_tab : sh_tab) + EntryWords<R>::value * slot;
    R* accp = acc + ((size_t)aux * q.wg + warp_in_group) * 8;
    const int rlane = FULL ? lane : q.t;
    switch (code) {
#define VQC_M1(T_)                                                                   \
    case DC_M1 + T_:                                                                 \
        if constexpr (T_ < K) {                                                      \
            if (MODE == 0) {                                                         \
                m1_entry<R, K, T_, false>(a, tp);                                    \
            } else {                                                                 \
                if constexpr (FULL) {                                                \
                    /* one basic block; the butterfly is issued before the    */     \
                    /* adjoint updates so that the accumulator registers are */     \
                    /* free while both blocks are updated (fewer spills under */     \
                    /* the pass kernels' 128-register cap)                    */     \
                    if (flags & OPF_HAS_ACC) {                                       \
                        R rh[4] = {0, 0, 0, 0};                                      \
                        m1_t3<R, K, T_>(a, l, rh);                                   \
                        reduce4_full<R>(rh, lane, accp, acc_add);                    \
                        m1_entry<R, K, T_, true>(a, tp);                             \
                        m1_entry<R, K, T_, true>(l, tp);                             \
                    } else {                                                         \
                        m1_entry<R, K, T_, true>(a, tp);                             \
                        m1_entry<R, K, T_, true>(l, tp);                             \
                    }                                                                \
                } else {                                                             \
                    if (flags & OPF_HAS_ACC) {                                       \
                        R rh[4] = {0, 0, 0, 0};                                      \
                        m1_t3<R, K, T_>(a, l, rh);                                   \
                        reduce4_store<R>(rh, q.lanes, rlane, accp, q.mask, acc_add); \
                    }                                                                \
                    m1_entry<R, K, T_, true>(a, tp);                                 \
                    m1_entry<R, K, T_, true>(l, tp);                                 \
                }                                                                    \
            }                                                                        \
        }                                                                            \
        break;
        VQC_M1(0) VQC_M1(1) VQC_M1(2) VQC_M1(3) VQC_M1(4)
#undef VQC_M1
#define VQC_CXPL(T_)                                                                 \
    case DC_CX_PL + T_:                                                              \
        if constexpr (WITH_CX && T_ < K) {                                           \
            const bool p_ = physbit(pb, ra);                                         \
            x_pred<R, K, T_>(a, p_);                                                 \
            if (MODE == 1) x_pred<R, K, T_>(l, p_);                                  \
        }                                                                            \
        break;
        VQC_CXPL(0) VQC_CXPL(1) VQC_CXPL(2) VQC_CXPL(3) VQC_CXPL(4)
#undef VQC_CXPL
#define VQC_CZLL(A_, B_)                                                             \
    case DC_CZ_LL + cz_pair_index(A_, B_):                                           \
        if constexpr (A_ < K && B_ < K) {                                            \
            z2_ll<R, K, A_, B_>(a);                                                  \
            if (MODE == 1) z2_ll<R, K, A_, B_>(l);                                   \
        }                                                                            \
        break;
        VQC_CZLL(0, 1) VQC_CZLL(0, 2) VQC_CZLL(0, 3) VQC_CZLL(0, 4)
        VQC_CZLL(1, 2) VQC_CZLL(1, 3) VQC_CZLL(1, 4)
        VQC_CZLL(2, 3) VQC_CZLL(2, 4) VQC_CZLL(3, 4)
#undef VQC_CZLL
#define VQC_CZPL(L_)                                                                 \
    case DC_CZ_PL + L_:                                                              \
        if constexpr (L_ < K) {                                                      \
            const bool p_ = physbit(pb, rb);                                         \
            z1_pred<R, K, L_>(a, p_);                                                \
            if (MODE == 1) z1_pred<R, K, L_>(l, p_);                                 \
        }                                                                            \
        break;
        VQC_CZPL(0) VQC_CZPL(1) VQC_CZPL(2) VQC_CZPL(3) VQC_CZPL(4)
#undef VQC_CZPL
    case DC_CZ_PP: {
        const R sgn = (physbit(pb, ra) && physbit(pb, rb)) ? R(-1) : R(1);
#pragma unroll
        for (int r = 0; r < (1 << K); ++r) {
            a[r] = cm<R>(sgn * a[r].x, sgn * a[r].y);
            if (MODE == 1) l[r] = cm<R>(sgn * l[r].x, sgn * l[r].y);
        }
        break;
    }
#define VQC_PH2LL(LO_, HI_)                                                          \
    case DC_PH2_LL + cz_pair_index(LO_, HI_):                                        \
        if constexpr (WITH_PH2 && LO_ < K && HI_ < K) ph2_ll<R, K, MODE, FULL, LO_, HI_>(ra > rb, tp, flags, a, l, q, accp, acc_add); \
        break;
        VQC_PH2LL(0, 1) VQC_PH2LL(0, 2) VQC_PH2LL(0, 3) VQC_PH2LL(0, 4)
        VQC_PH2LL(1, 2) VQC_PH2LL(1, 3) VQC_PH2LL(1, 4)
        VQC_PH2LL(2, 3) VQC_PH2LL(2, 4) VQC_PH2LL(3, 4)
#undef VQC_PH2LL
#define VQC_PH2PL(L_)                                                                \
    case DC_PH2_PL + L_:                                                             \
        if constexpr (WITH_PH2 && L_ < K) ph2_pl<R, K, MODE, FULL, L_>(ra < kRefPhys, physbit(pb, ra < kRefPhys ? rb : ra), tp, flags, a, l, q, accp, acc_add); \
        break;
        VQC_PH2PL(0) VQC_PH2PL(1) VQC_PH2PL(2) VQC_PH2PL(3) VQC_PH2PL(4)
#undef VQC_PH2PL
    case DC_PH2_PP:
        if constexpr (WITH_PH2)
            ph2_pp<R, K, MODE, FULL>((int)physbit(pb, ra) + 2 * (int)physbit(pb, rb), tp, flags, a, l, q,
                                     accp, acc_add);
        break;
    default:
        break;
    }
}

// Run ops [ob, oe) of a stage (forward: in order; backward: reversed).  The
// descriptor is read when the op starts: keeping a prefetched one live across
// the dispatch switch costs more registers than the load latency it hides.
template <typename R, int K, int MODE, bool WITH_CX, bool FULL, bool WITH_PH2 = true>
__device__ __forceinline__ void run_ops(const DOp* ops, int ob, int oe, uint32_t pb,
                                        C2<R> (&a)[1 << K], C2<R> (&l)[1 << K], const R* sh_tab,
                                        const R* ps_tab, R* acc, const Geo& q, int lane,
                                        int warp_in_group, bool acc_add = false) {
    const uint2* op2 = reinterpret_cast<const uint2*>(ops);
    if (MODE == 0) {
        for (int o = ob; o < oe; ++o)
            apply_op<R, K, MODE, WITH_CX, FULL, WITH_PH2>(vqc_ld(op2 + o), pb, a, l, sh_tab, ps_tab, acc, q, lane,
                                          warp_in_group, acc_add);
    } else {
        for (int o = oe - 1; o >= ob; --o)
            apply_op<R, K, MODE, WITH_CX, FULL, WITH_PH2>(vqc_ld(op2 + o), pb, a, l, sh_tab, ps_tab, acc, q, lane,
                                          warp_in_group, acc_add);
    }
}

// lam = O psi on the block, O = sum_j gE_j Z_j (diagonal): the sign of Z_j comes
// from local bit j of r for active qubits and from the block base pb otherwise.
template <typename R, int K, typename GI>
__device__ __forceinline__ void lambda_init(const DStage* sp, uint32_t pb, const GI* gb, int n,
                                            const C2<R> (&a)[1 << K], C2<R> (&l)[1 << K]) {
    R ge_loc[K];
    R cst = 0;
    uint32_t actmask = 0;
#pragma unroll
    for (int j = 0; j < K; ++j) {
        const int aq = vqc_ld(&sp->active[j]);
        actmask |= 1u << aq;
        ge_loc[j] = as_r<R>(gb[aq]);
    }
    for (int j = 0; j < n; ++j)
        if (!((actmask >> j) & 1)) cst += ((pb >> j) & 1u) ? -as_r<R>(gb[j]) : as_r<R>(gb[j]);
#pragma unroll
    for (int r = 0; r < (1 << K); ++r) {
        R o = cst;
#pragma unroll
        for (int j = 0; j < K; ++j) o += ((r >> j) & 1) ? -ge_loc[j] : ge_loc[j];
        l[r] = cm<R>(o * a[r].x, o * a[r].y);
    }
}

// Adds this block's contributions to E_j = sum (-1)^{bit j} |a|^2 for qubits
// j < NV into ez[j] (a qubit outside the block contributes +-(block norm) by
// its bit in pb; entries j >= n stay untouched and are never read).
template <typename R, int K, int NV>
__device__ __forceinline__ void expz_accum(const DStage* sp, uint32_t pb, const C2<R> (&a)[1 << K],
                                           R (&ez)[NV]) {
    R ptot = 0;
    R dloc[K];
#pragma unroll
    for (int j = 0; j < K; ++j) dloc[j] = 0;
#pragma unroll
    for (int r = 0; r < (1 << K); ++r) {
        const R pr = fma(a[r].x, a[r].x, a[r].y * a[r].y);
        ptot += pr;
#pragma unroll
        for (int j = 0; j < K; ++j) dloc[j] += ((r >> j) & 1) ? -pr : pr;
    }
    uint32_t actmask = 0;
    int aq[K];
#pragma unroll
    for (int j = 0; j < K; ++j) {
        aq[j] = vqc_ld(&sp->active[j]);
        actmask |= 1u << aq[j];
    }
#pragma unroll
    for (int j = 0; j < NV; ++j) {
        R val = ((pb >> j) & 1u) ? -ptot : ptot;
#pragma unroll
        for (int k = 0; k < K; ++k) val = aq[k] == j ? dloc[k] : val;
        ez[j] += val;
    }
}

// Sum NV values over the 32 lanes of a warp (reduce-scatter butterfly, NV - 1
// + log2(32 / NV) shuffles).  Returns the value index this lane ends up with;
// v[0] then holds that value's warp sum in every lane whose bits below the
// scatter bits are zero (and in their partners).
template <typename R, int NV>
__device__ __forceinline__ int warp_reduce_scatter(R (&v)[NV], int lane) {
    int idx = 0;
    int m = 16;
#pragma unroll
    for (int w = NV; w > 1; w >>= 1, m >>= 1) {
        const int u = (lane & m) ? 1 : 0;
        const int h = w >> 1;
#pragma unroll
        for (int i = 0; i < h; ++i) {
            const R send = u ? v[i] : v[i + h];
            const R keep = u ? v[i + h] : v[i];
            v[i] = keep + shx<R>(send, m, 0xffffffffu);
        }
        idx = 2 * idx + u;
    }
#pragma unroll
    for (; m >= 1; m >>= 1) v[0] += shx<R>(v[0], m, 0xffffffffu);
    return idx;
}

// Per-warp partial sums of E_j = sum (-1)^{bit j} |a|^2 over this group's
// blocks, written to red[warp_in_group * n + j].
template <typename R, int K>
__device__ __forceinline__ void expz_partials(const DStage* sp, uint32_t pb,
                                              const C2<R> (&a)[1 << K], int n, R* red,
                                              const Geo& q, int warp_in_group, bool add = false) {
    R ptot = 0;
    R dloc[K];
#pragma unroll
    for (int j = 0; j < K; ++j) dloc[j] = 0;
#pragma unroll
    for (int r = 0; r < (1 << K); ++r) {
        const R pr = fma(a[r].x, a[r].x, a[r].y * a[r].y);
        ptot += pr;
#pragma unroll
        for (int j = 0; j < K; ++j) dloc[j] += ((r >> j) & 1) ? -pr : pr;
    }
    uint32_t actmask = 0;
    int aq[K];
#pragma unroll
    for (int j = 0; j < K; ++j) {
        aq[j] = vqc_ld(&sp->active[j]);
        actmask |= 1u << aq[j];
    }
    for (int j = 0; j < n; ++j) {
        R val;
        if ((actmask >> j) & 1) {
            val = 0;
#pragma unroll
            for (int k = 0; k < K; ++k) if (aq[k] == j) val = dloc[k];
        } else {
            val = ((pb >> j) & 1u) ? -ptot : ptot;
        }
        val = reduce1<R>(val, q.lanes, q.mask);
        if ((q.t & (q.lanes - 1)) == 0) {
            R* d = red + warp_in_group * n + j;
            *d = add ? *d + val : val;
        }
    }
}

// Gradient terms of one accumulator slot (summed over the wg per-warp
// partials at ap): a phase op's scalar, or Im Tr(W_j P_j W_j^dag rho) for each
// parametrised constituent j of a run.  Writes out[term].
template <typename R, typename XI, typename WI, typename O>
__device__ void acc_terms(const DAcc& ac, const DEntry& e, const R* ap, int wg,
                          const DConst* consts, const XI* xg, const WI* w, const R* cang,
                          const R* cmat, O* out) {
    if (ac.kind == 1) {
        R sum = 0;
        for (int k2 = 0; k2 < wg; ++k2) sum += ap[k2 * 8];
        out[consts[e.cfirst].term] = as_out<O>(sum);
        return;
    }
    R vx = 0, vy = 0, vz = 0;
    for (int k2 = 0; k2 < wg; ++k2) {
        vx += ap[k2 * 8 + 0];
        vy += ap[k2 * 8 + 1];
        vz += ap[k2 * 8 + 2];
    }
    // The accumulator holds (tx, ty, tz) of rho's traceless anti-Hermitian part
    // rho' = (i/2)(tx X + ty Y + tz Z).  term_j = Im Tr(W_j P_j W_j^dag rho) =
    // Im Tr(P_j rho_j) = the P_j component of rho_j = W_j^dag rho' W_j, carried
    // from the last constituent backwards: rho' <- U^dag rho' U after each one.
    // For U = exp(-i t P / 2) that turns (tx, ty, tz) by the full angle t about
    // P's axis; a scalar phase leaves it; a constant 2x2 goes through its matrix.
    for (int c = e.ccount - 1; c >= 0; --c) {
        const DConst cn = consts[e.cfirst + c];
        if (cn.term >= 0) out[cn.term] = as_out<O>(cn.kind == CK_RX ? vx : cn.kind == CK_RY ? vy : vz);
        if (c == 0) break;
        if (cn.kind == CK_RX || cn.kind == CK_RY || cn.kind == CK_RZ) {
            R sn, co;
            sc(angle_of<R>(cn.src0, cn.idx0, xg, w, cang), &sn, &co);
            if (cn.kind == CK_RX) {
                const R y2 = vy * co + vz * sn, z2 = vz * co - vy * sn;
                vy = y2; vz = z2;
            } else if (cn.kind == CK_RY) {
                const R x2 = vx * co - vz * sn, z2 = vz * co + vx * sn;
                vx = x2; vz = z2;
            } else {
                const R x2 = vx * co + vy * sn, y2 = vy * co - vx * sn;
                vx = x2; vy = y2;
            }
        } else if (cn.kind == CK_CONST) {
            const R h = R(0.5);
            M2<R> rho;
            rho.a = cm<R>(0, h * vz); rho.b = cm<R>(h * vy, h * vx);
            rho.c = cm<R>(-h * vy, h * vx); rho.d = cm<R>(0, -h * vz);
            const M2<R> u = constituent<R>(cn, xg, w, cang, cmat);
            rho = mmul<R>(mdag<R>(u), mmul<R>(rho, u));
            // Im Tr(X rho) = Im r01 + Im r10, Im Tr(Y rho) = Re r01 - Re r10,
            // Im Tr(Z rho) = Im r00 - Im r11
            vx = rho.b.y + rho.c.y;
            vy = rho.b.x - rho.c.x;
            vz = rho.a.y - rho.d.y;
        }
    }
}


// ---------------------------------------------------------------- kernel
// MODE 0: forward, MODE 1: backward.
// FULL: every sample group spans whole warps (2^(n-K) >= 32 threads), so warp
// reductions are fixed full-warp butterflies; the launch picks the variant.
// FUSED (MODE 1 only): the backward that recomputes the states also writes E
// (vqc_forward_backward); a separate instantiation keeps that code out of the
// plain backward kernel.
// Launch-geometry self-check (kernel side): the host derives the block size,
// the sample groups and the register blocks from one plan; a launch whose
// numbers disagree records `code` in the plan's error word (read back by
// vqc_sync_check) and does no work.  Uniform over the grid: every thread takes
// the same branch.
__device__ __forceinline__ bool geometry_bad(bool bad, unsigned* err, unsigned code) {
    if (bad && threadIdx.x == 0 && err) atomicOr(err, code);
    return bad;
}
enum : unsigned { kErrSweepGeometry = 1u, kErrPassGeometry = 2u, kErrClusterGeometry = 4u };

template <typename R, int K, int MODE, bool FULL, bool FUSED, bool PH2 = true>
__global__ void __launch_bounds__(512) sweep_kernel(const __grid_constant__ KArgs<St<R>> A) {
    if (geometry_bad(blockDim.x != (unsigned)(A.S * A.tpg) || A.bpt * A.tpg != (1 << A.tbits) ||
                         A.tbits != A.n - K || A.nstages < 1,
                     A.err, kErrSweepGeometry))
        return;
    extern __shared__ __align__(16) unsigned char smem[];
    R* sh_tab = reinterpret_cast<R*>(smem + A.sm_sh);
    R* ps_all = reinterpret_cast<R*>(smem + A.sm_ps);
    C2<R>* psi_all = reinterpret_cast<C2<R>*>(smem + A.sm_psi);
    C2<R>* lam_all = reinterpret_cast<C2<R>*>(smem + A.sm_lam);
    R* acc_all = reinterpret_cast<R*>(smem + A.sm_acc);
    R* terms_all = reinterpret_cast<R*>(smem + A.sm_terms);
    R* dw_cta = reinterpret_cast<R*>(smem + A.sm_dw);
    R* red_all = reinterpret_cast<R*>(smem + A.sm_red);

    const int n = A.n, G = A.G;
    const int dim = 1 << n;
    Geo q;
    q.T = A.tpg;
    q.lanes = q.T < 32 ? q.T : 32;
    q.wg = q.T > 32 ? q.T / 32 : 1;
    q.g = threadIdx.x / q.T;
    q.t = threadIdx.x % q.T;
    q.h = 0;
    if (A.tbits < G) q.h = ((q.g & ((1 << (G - A.tbits)) - 1)) << A.tbits) & (dim - 1);
    q.mask = blockDim.x >= 32 ? 0xffffffffu : ((1u << blockDim.x) - 1u);
    const int lane = q.t & 31;
    const int warp_in_group = q.t >> 5;
    const int nthr = blockDim.x;

    R* w_sm = reinterpret_cast<R*>(smem + A.sm_w);
    R* xg_all = reinterpret_cast<R*>(smem + A.sm_xg);
    const int xgw = A.Px + n;   // row width of the x / gE staging area
    C2<R>* psi = psi_all + (size_t)q.g * dim;
    C2<R>* lam = lam_all + (size_t)q.g * dim;

    // initial (forward) or final (backward) state source; null: |0...0>
    const SC2<R>* src = MODE == 1 ? A.psi_final : A.psi0;
    if (MODE == 1 && !src) src = A.psi0;
    const bool from_global = src != nullptr;

    // One unit's inputs to shared memory, asynchronously: x (and, backward,
    // gE) rows of its samples and each sample's initial / final state
    // (coalesced reads, swizzled slots).
    // (Double-float kernels copy the stored doubles as they are and split them
    // in place afterwards, unit_to_dd: both types are 8 bytes.)
    St<R>* xg_st = reinterpret_cast<St<R>*>(xg_all);
    SC2<R>* psi_st = reinterpret_cast<SC2<R>*>(psi);
    auto stage_unit = [&](int unit) {
        for (int i = threadIdx.x; i < A.S * xgw; i += nthr) {
            const int gg = i / xgw, c = i % xgw;
            const int bb = min(unit * A.S + gg, A.B - 1);
            if (c < A.Px) async_elem<St<R>>(xg_st + i, A.x + (size_t)bb * A.Px + c);
            else if (MODE == 1) async_elem<St<R>>(xg_st + i, A.gE + (size_t)bb * n + (c - A.Px));
        }
        if (from_global) {
            const int b = min(unit * A.S + q.g, A.B - 1);
            const SC2<R>* gs = src + (size_t)b * dim;
            for (int u = q.t; u < dim; u += q.T) async_elem<SC2<R>>(psi_st + (swz(u, G) ^ q.h), gs + u);
        }
    };
    // after async_wait(): stored doubles -> dd in place, each by the thread that
    // issued its copy (its own copies are visible to it); a barrier follows
    auto unit_to_dd = [&]() {
        if constexpr (!std::is_same<St<R>, R>::value) {
            for (int i = threadIdx.x; i < A.S * xgw; i += nthr) {
                const int c = i % xgw;
                if (c < A.Px || MODE == 1) xg_all[i] = R(xg_st[i]);
            }
            if (from_global)
                for (int u = q.t; u < dim; u += q.T) {
                    const int sl = swz(u, G) ^ q.h;
                    psi[sl] = c2_in<R>(psi_st[sl]);
                }
        }
    };

    // Prologue: the plan regions, w and the first unit's inputs all in flight
    // at once, one wait.
    const unsigned char* smt = nullptr;
    const unsigned char* sms = nullptr;
    if (A.plan_smem) {
        unsigned char* t = smem + A.sm_plan;
        unsigned char* u = t + ((A.tab_bytes + 15) & ~15);
        async_region(t, A.plan + A.tab_off, A.tab_bytes);
        async_region(u, A.plan + A.sched_off, A.sched_bytes);
        smt = t;
        sms = u;
    }
    grid_dep_wait();
    grid_dep_launch();
    for (int i = threadIdx.x; i < A.Pw; i += nthr)
        async_elem<St<R>>(reinterpret_cast<St<R>*>(w_sm) + i, A.w + i);
    if ((int)blockIdx.x < A.nunits) stage_unit(blockIdx.x);
    if (MODE == 1)
        for (int i = threadIdx.x; i < A.Pw; i += nthr) dw_cta[i] = 0;
    PlanPtrs P;
    P.ops = rebase(A.ops, A.plan, A.sched_off, sms);
    P.stages = rebase(A.stages, A.plan, A.sched_off, sms);
    P.entries = rebase(A.entries, A.plan, A.tab_off, smt);
    P.ps_list = rebase(A.ps_list, A.plan, A.tab_off, smt);
    P.sh_list = rebase(A.sh_list, A.plan, A.tab_off, smt);
    P.consts = rebase(A.consts, A.plan, A.tab_off, smt);
    P.cmat = rebase(reinterpret_cast<const unsigned char*>(A.cmat), A.plan, A.tab_off, smt);
    P.cang = rebase(reinterpret_cast<const unsigned char*>(A.cang), A.plan, A.tab_off, smt);
    P.accs = rebase(A.accs, A.plan, A.tab_off, smt);
    P.xocc_ptr = rebase(A.xocc_ptr, A.plan, A.tab_off, smt);
    P.xocc = rebase(A.xocc, A.plan, A.tab_off, smt);
    P.wocc_ptr = rebase(A.wocc_ptr, A.plan, A.tab_off, smt);
    P.wocc = rebase(A.wocc, A.plan, A.tab_off, smt);
    const R* Pcmat = reinterpret_cast<const R*>(P.cmat);
    const R* Pcang = reinterpret_cast<const R*>(P.cang);
    async_wait();
    if constexpr (!std::is_same<St<R>, R>::value) {
        for (int i = threadIdx.x; i < A.Pw; i += nthr) w_sm[i] = R(reinterpret_cast<const St<R>*>(w_sm)[i]);
        if ((int)blockIdx.x < A.nunits) unit_to_dd();
    }
    __syncthreads();

    // shared table (w and constants) once per CTA, on the CTA's last threads
    // so that it runs beside the first unit's per-sample table
    for (int i = nthr - 1 - threadIdx.x; i < A.n_sh; i += nthr) {
        const int id = vqc_ld(&P.sh_list[i]);
        const DEntry e = P.entries[id];
        eval_entry<R>(e, P.consts, static_cast<const R*>(nullptr), w_sm, Pcang, Pcmat,
                      sh_tab + EntryWords<R>::value * e.slot);
    }

    R* ps_tab = ps_all + (size_t)q.g * A.n_ps * EntryWords<R>::value;
    R* acc = acc_all + (size_t)q.g * A.n_accs * q.wg * 8;
    R* terms = terms_all + (size_t)q.g * A.n_terms;

    for (int unit = blockIdx.x; unit < A.nunits; unit += gridDim.x) {
        const int b_raw = unit * A.S + q.g;
        const bool valid = b_raw < A.B;
        const int b = valid ? b_raw : A.B - 1;
        if (unit != (int)blockIdx.x) {
            stage_unit(unit);
            async_wait();
            if constexpr (!std::is_same<St<R>, R>::value) unit_to_dd();
            __syncthreads();
        }
        const R* xrow = xg_all + (size_t)q.g * xgw;

        // per-sample table (x-dependent runs): threads of the CTA over (sample, entry)
        for (int i = threadIdx.x; i < A.S * A.n_ps; i += nthr) {
            const int gg = i / A.n_ps, k = i % A.n_ps;
            const int id = vqc_ld(&P.ps_list[k]);
            const DEntry e = P.entries[id];
            eval_entry<R>(e, P.consts, xg_all + (size_t)gg * xgw, w_sm, Pcang, Pcmat,
                          ps_all + ((size_t)gg * A.n_ps + e.slot) * EntryWords<R>::value);
        }
        __syncthreads();

        C2<R> a[1 << K];
        int32_t sg[K];
        StageView v{0, 0};
        const bool recompute = MODE == 1 && A.psi_final == nullptr;
        const int ns = A.nstages;

        // -------- forward sweep (forward mode, or backward recompute; the
        // recompute also writes E when the caller asks for it)
        R* red = red_all + (size_t)q.g * q.wg * n;
        const bool want_E = MODE == 0 || (FUSED && recompute && A.E != nullptr);
        if (MODE == 0 || recompute) {
            for (int s = 0; s < ns; ++s) {
                const DStage* sp = P.stages + s;
                const bool last = s + 1 == ns;
                const bool store = !last || (MODE == 0 && A.state_out) || (MODE == 1 && A.bpt > 1);
                R eacc = 0;   // full-warp groups: this lane's share of the warp's <Z> sums
                int eidx = 0;
                for (int bj = 0; bj < A.bpt; ++bj) {
                    v = stage_view<K>(sp, q.t + bj * q.T, q.h, sg);
                    if (s == 0 && !from_global) {
#pragma unroll
                        for (int r = 0; r < (1 << K); ++r) a[r] = cm<R>(0, 0);
                        if (v.pb == 0) a[0] = cm<R>(1, 0);
                    } else {
                        block_load<R, K>(a, psi, v.swb, sg);
                    }
                    run_ops<R, K, 0, false, FULL, PH2>(P.ops, vqc_ld(&sp->op_begin), vqc_ld(&sp->op_end), v.pb, a, a,
                                     sh_tab, ps_tab, nullptr, q, lane, warp_in_group);
                    if (want_E && last) {   // <Z_j> partials from the final blocks
                        if constexpr (FULL) {   // butterfly over the warp (n <= 16 here)
                            if (n <= 8) {
                                R ez[8];
#pragma unroll
                                for (int j = 0; j < 8; ++j) ez[j] = 0;
                                expz_accum<R, K, 8>(sp, v.pb, a, ez);
                                eidx = warp_reduce_scatter<R, 8>(ez, lane);
                                eacc += ez[0];
                            } else {
                                R ez[16];
#pragma unroll
                                for (int j = 0; j < 16; ++j) ez[j] = 0;
                                expz_accum<R, K, 16>(sp, v.pb, a, ez);
                                eidx = warp_reduce_scatter<R, 16>(ez, lane);
                                eacc += ez[0];
                            }
                        } else {
                            expz_partials<R, K>(sp, v.pb, a, n, red, q, warp_in_group, bj > 0);
                        }
                    }
                    if (store) {   // through the store map (absorbed CX gates)
                        // a permuting store writes slots other threads load in this
                        // stage: every load of the group must be done first
                        if (vqc_ld(&sp->nperm)) group_sync<R>(q);
                        int32_t s2[K];
                        const uint32_t b2 = map_base<K, true>(sp, q.t + bj * q.T, q.h, s2);
                        block_store<R, K>(a, psi, b2, s2);
                    }
                }
                if (want_E && last && FULL) {
                    // a single-warp group writes E itself
                    const int low = n <= 8 ? 3 : 1;   // lane bits below the scatter bits
                    if ((lane & low) == 0 && eidx < n) {
                        if (q.wg == 1) {
                            if (valid) A.E[(size_t)b * n + eidx] = as_out<St<R>>(eacc);
                        } else {
                            red[warp_in_group * n + eidx] = eacc;
                        }
                    }
                }
                if (store) group_sync<R>(q);
            }
        }

        if (MODE == 0) {
            const bool direct = FULL && q.wg == 1;   // E already written
            if (!direct || A.state_out) {
                __syncthreads();
                if (valid) {
                    if (!direct) {
                        for (int j = q.t; j < n; j += q.T) {
                            R e = 0;
                            for (int k = 0; k < q.wg; ++k) e += red[k * n + j];
                            A.E[(size_t)b * n + j] = as_out<St<R>>(e);
                        }
                    }
                    if (A.state_out) {
                        SC2<R>* go = A.state_out + (size_t)b * dim;
                        for (int u = q.t; u < dim; u += q.T) go[u] = c2_out<R>(psi[swz(u, G) ^ q.h]);
                    }
                }
            }
            if (unit + (int)gridDim.x < A.nunits) __syncthreads();
            continue;
        }

        if (MODE == 1 && want_E && !(FULL && q.wg == 1)) {   // E of the recomputed states
            __syncthreads();
            if (valid)
                for (int j = q.t; j < n; j += q.T) {
                    R e = 0;
                    for (int k = 0; k < q.wg; ++k) e += red[k * n + j];
                    A.E[(size_t)b * n + j] = as_out<St<R>>(e);
                }
        }

        // -------- backward: reverse sweep with psi and lam
        for (int s = ns - 1; s >= 0; --s) {
            const DStage* sp = P.stages + s;
            for (int bj = 0; bj < A.bpt; ++bj) {
                C2<R> l[1 << K];
                v = stage_view<K>(sp, q.t + bj * q.T, q.h, sg);
                if (s == ns - 1) {
                    if (!recompute || A.bpt > 1) block_load<R, K>(a, psi, v.swb, sg);
                    lambda_init<R, K>(sp, v.pb, xrow + A.Px, n, a, l);
                } else {   // the forward left this stage's output in its store map
                    int32_t s2[K];
                    const uint32_t b2 = map_base<K, true>(sp, q.t + bj * q.T, q.h, s2);
                    block_load<R, K>(a, psi, b2, s2);
                    block_load<R, K>(l, lam, b2, s2);
                }
                run_ops<R, K, 1, false, FULL, PH2>(P.ops, vqc_ld(&sp->op_begin), vqc_ld(&sp->op_end), v.pb, a, l,
                                 sh_tab, ps_tab, acc, q, lane, warp_in_group, bj > 0);
                if (s > 0) {   // back to the stage's input layout (load map)
                    if (vqc_ld(&sp->nperm)) group_sync<R>(q);   // see the forward's store
                    int32_t s2[K];
                    const uint32_t b2 = map_base<K, false>(sp, q.t + bj * q.T, q.h, s2);
                    block_store<R, K>(a, psi, b2, s2);
                    block_store<R, K>(l, lam, b2, s2);
                }
            }
            group_sync<R>(q);
        }
        __syncthreads();

        // -------- gradient terms from the accumulated rho / scalars
        for (int i = threadIdx.x; i < A.S * A.n_accs; i += nthr) {
            const int gg = i / A.n_accs, k = i % A.n_accs;
            const DAcc ac = P.accs[k];
            acc_terms<R>(ac, P.entries[ac.entry], acc_all + ((size_t)gg * A.n_accs + k) * q.wg * 8,
                         q.wg, P.consts, xg_all + (size_t)gg * xgw, w_sm, Pcang, Pcmat,
                         terms_all + (size_t)gg * A.n_terms);
        }
        __syncthreads();
        // dx rows of this CTA's samples; dw partial of this CTA (fixed order)
        if (A.dx) {
            for (int i = threadIdx.x; i < A.S * A.Px; i += nthr) {
                const int gg = i / A.Px, p = i % A.Px;
                const int bb = unit * A.S + gg;
                if (bb >= A.B) continue;
                const R* tm = terms_all + (size_t)gg * A.n_terms;
                const int k0 = vqc_ld(&P.xocc_ptr[p]), k1 = vqc_ld(&P.xocc_ptr[p + 1]);
                R sum = 0;
                for (int k = k0; k < k1; ++k) sum += tm[vqc_ld(&P.xocc[k])];
                A.dx[(size_t)bb * A.Px + p] = as_out<St<R>>(sum);
            }
        }
        const int nvalid = min(A.S, A.B - unit * A.S);
        for (int p = threadIdx.x; p < A.Pw; p += nthr) {
            // samples in order, each sample's occurrences in order
            const int k0 = vqc_ld(&P.wocc_ptr[p]), k1 = vqc_ld(&P.wocc_ptr[p + 1]);
            R sum = dw_cta[p];
            if (k1 - k0 == 1) {   // the common case: independent loads
                const int j = vqc_ld(&P.wocc[k0]);
                for (int gg = 0; gg < nvalid; ++gg) sum += terms_all[(size_t)gg * A.n_terms + j];
            } else {
                for (int gg = 0; gg < nvalid; ++gg) {
                    const R* tm = terms_all + (size_t)gg * A.n_terms;
                    for (int k = k0; k < k1; ++k) sum += tm[vqc_ld(&P.wocc[k])];
                }
            }
            dw_cta[p] = sum;
        }
        __syncthreads();
    }

    if (MODE == 1 && A.Pw > 0 && A.dw) {
        // per-CTA partial of dw; reduce_cols sums the partials in CTA order
        for (int p = threadIdx.x; p < A.Pw; p += nthr)
            A.dw_part[(size_t)blockIdx.x * A.Pw + p] = as_out<St<R>>(dw_cta[p]);
    }
}

// out[c] = sum over rows r of part[r * cols + c]: one block per column,
// fixed strided partial sums, then a fixed-shape tree (deterministic).
template <typename R>
__global__ void __launch_bounds__(256) reduce_cols(const R* part, int rows, int cols, R* out) {
    __shared__ R buf[256];
    const int c = blockIdx.x;
    grid_dep_wait();
    grid_dep_launch();
    R s = 0;
    for (int r = threadIdx.x; r < rows; r += 256) s += part[(size_t)r * cols + c];
    buf[threadIdx.x] = s;
    __syncthreads();
    for (int w = 128; w >= 1; w >>= 1) {
        if (threadIdx.x < w) buf[threadIdx.x] += buf[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) out[c] = buf[0];
}

}  // namespace vqc
