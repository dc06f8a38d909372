// cluster.cuh -- forward and backward sweeps with a sample's state (forward) or
// its psi and lam (backward) spread over a thread-block cluster (distributed
// shared memory), for states larger than one SM's shared memory but small
// enough for 2..8 SMs (forward: complex64 15-16 qubits, complex128 14-16;
// backward: complex64 14-16, complex128 13-15).
//
// Same stage program as the resident path (sweep.cuh): the stage maps give
// every register amplitude a slot in [0, 2^n); slot s lives in the shared memory
// of cluster rank s >> (n - CL) at local position s & (2^(n-CL) - 1).  The
// swizzle only XORs the lowest G index bits, so a CTA holds exactly the
// amplitudes whose top CL qubits equal its rank.  Loads and stores go through
// the cluster window (mapa + ld/st.shared::cluster); a cluster barrier replaces
// the group barrier between stages.  A stage whose maps keep every block inside
// its thread's own CTA (the compiler's cl_local flags) uses plain shared loads
// and stores and, when no data crosses CTAs at its end, the CTA barrier.  One
// sample per cluster at a time; the 2^(n-K) threads of its group are spread
// over the cluster's CTAs in rank order.  The forward's <Z> sums go from each
// CTA to rank 0, which writes E; the backward's rho sums likewise (rank 0
// writes dx and the cluster's dw partial).
#pragma once

#include "sweep.cuh"

namespace vqc {

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// Every thread of every CTA of the cluster arrives; memory operations before
// it (including shared::cluster stores) are visible to all of them after it.
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n"
                 "barrier.cluster.wait.acquire.aligned;\n" ::: "memory");
}
// Address of local shared address `sa` in the shared memory of cluster rank r.
__device__ __forceinline__ uint32_t cluster_map(uint32_t sa, uint32_t r) {
    uint32_t d;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(sa), "r"(r));
    return d;
}
__device__ __forceinline__ float2 dsm_load(uint32_t a, float2*) {
    float2 v;
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ double2 dsm_load(uint32_t a, double2*) {
    double2 v;
    asm volatile("ld.shared::cluster.v2.f64 {%0, %1}, [%2];" : "=d"(v.x), "=d"(v.y) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ void dsm_store(uint32_t a, float2 v) {
    asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(a), "f"(v.x), "f"(v.y) : "memory");
}
__device__ __forceinline__ void dsm_store(uint32_t a, double2 v) {
    asm volatile("st.shared::cluster.v2.f64 [%0], {%1, %2};" ::"r"(a), "d"(v.x), "d"(v.y) : "memory");
}
__device__ __forceinline__ void dsm_store(uint32_t a, float v) {
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(a), "f"(v) : "memory");
}
__device__ __forceinline__ void dsm_store(uint32_t a, double v) {
    asm volatile("st.shared::cluster.f64 [%0], %1;" ::"r"(a), "d"(v) : "memory");
}
__device__ __forceinline__ void dsm_load_r(uint32_t a, float* v) {
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(*v) : "r"(a) : "memory");
}
__device__ __forceinline__ void dsm_load_r(uint32_t a, double* v) {
    asm volatile("ld.shared::cluster.f64 %0, [%1];" : "=d"(*v) : "r"(a) : "memory");
}
__device__ __forceinline__ void dsm_load_r(uint32_t a, dd* v) {
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v->hi), "=f"(v->lo) : "r"(a) : "memory");
}
// double-float: (hi, lo) pairs, complex values as (re.hi, re.lo, im.hi, im.lo)
__device__ __forceinline__ dd2 dsm_load(uint32_t a, dd2*) {
    dd2 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x.hi), "=f"(v.x.lo), "=f"(v.y.hi), "=f"(v.y.lo) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ void dsm_store(uint32_t a, dd2 v) {
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(a), "f"(v.x.hi), "f"(v.x.lo),
                 "f"(v.y.hi), "f"(v.y.lo) : "memory");
}
__device__ __forceinline__ void dsm_store(uint32_t a, dd v) {
    asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(a), "f"(v.hi), "f"(v.lo) : "memory");
}

// Cluster address of slot s of the distributed state (psi_sa: this CTA's local
// shared address of its slice; slices are 2^slice amplitudes).
template <typename R>
__device__ __forceinline__ uint32_t slot_addr(uint32_t psi_sa, uint32_t s, int slice) {
    const uint32_t owner = s >> slice, off = s & ((1u << slice) - 1u);
    return cluster_map(psi_sa + off * (uint32_t)sizeof(C2<R>), owner);
}

template <typename R, int K>
__device__ __forceinline__ void cl_block_load(C2<R> (&a)[1 << K], uint32_t psi_sa, int slice,
                                              uint32_t swb, const int32_t (&sg)[K]) {
#pragma unroll
    for (int r = 0; r < (1 << K); ++r)
        a[r] = dsm_load(slot_addr<R>(psi_sa, swb ^ block_off<K>(r, sg), slice), (C2<R>*)nullptr);
}
template <typename R, int K>
__device__ __forceinline__ void cl_block_store(const C2<R> (&a)[1 << K], uint32_t psi_sa, int slice,
                                               uint32_t swb, const int32_t (&sg)[K]) {
#pragma unroll
    for (int r = 0; r < (1 << K); ++r) dsm_store(slot_addr<R>(psi_sa, swb ^ block_off<K>(r, sg), slice), a[r]);
}

// KArgs fields used: the plan, n, K, G, tpg (= 2^(n-K), threads per sample over
// the cluster), nunits (= B), x, w, psi0, E, state_out, the shared-memory
// carve-up (sm_psi holds this CTA's slice of 2^(n - cl) amplitudes, sm_red the
// per-warp <Z> sums, sm_ecl rank 0's [2^cl][n] gather of per-CTA sums), cl.
template <typename R, int K>
__global__ void __launch_bounds__(512) cluster_fwd_kernel(const __grid_constant__ KArgs<St<R>> A) {
    // every CTA of every cluster takes the same branch, before any cluster barrier
    uint32_t nrank;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(nrank));
    if (geometry_bad(((unsigned)blockDim.x << A.cl) != (unsigned)A.tpg || nrank != (1u << A.cl) ||
                         A.tpg != (1 << (A.n - K)) || A.nstages < 1,
                     A.err, kErrClusterGeometry))
        return;
    extern __shared__ __align__(16) unsigned char smem[];
    R* sh_tab = reinterpret_cast<R*>(smem + A.sm_sh);
    R* ps_tab = reinterpret_cast<R*>(smem + A.sm_ps);
    C2<R>* psi = reinterpret_cast<C2<R>*>(smem + A.sm_psi);
    R* red = reinterpret_cast<R*>(smem + A.sm_red);
    R* ecl = reinterpret_cast<R*>(smem + A.sm_ecl);
    R* w_sm = reinterpret_cast<R*>(smem + A.sm_w);
    R* xrow = reinterpret_cast<R*>(smem + A.sm_xg);

    const int n = A.n, G = A.G, CL = A.cl;
    const int slice = n - CL;
    const uint32_t smask = (1u << slice) - 1u;
    const uint32_t rank = cluster_rank();
    const int cid = (int)(blockIdx.x >> CL), ncl = (int)(gridDim.x >> CL);
    const int nthr = blockDim.x;
    const int tg = (int)rank * nthr + (int)threadIdx.x;   // thread index in the sample group
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = nthr >> 5;
    Geo q;
    q.T = A.tpg;
    q.lanes = 32;
    q.wg = nwarps;
    q.g = 0;
    q.t = tg;
    q.h = 0;
    q.mask = 0xffffffffu;
    const uint32_t psi_sa = static_cast<uint32_t>(__cvta_generic_to_shared(psi));
    const uint32_t ecl_sa = static_cast<uint32_t>(__cvta_generic_to_shared(ecl));

    // plan regions (immutable) before the dependency wait; then caller memory
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
    async_wait();
    if constexpr (!std::is_same<St<R>, R>::value)   // each thread splits the values it copied
        for (int i = threadIdx.x; i < A.Pw; i += nthr) w_sm[i] = R(reinterpret_cast<const St<R>*>(w_sm)[i]);
    PlanPtrs P;
    P.ops = rebase(A.ops, A.plan, A.sched_off, sms);
    P.stages = rebase(A.stages, A.plan, A.sched_off, sms);
    P.entries = rebase(A.entries, A.plan, A.tab_off, smt);
    P.ps_list = rebase(A.ps_list, A.plan, A.tab_off, smt);
    P.sh_list = rebase(A.sh_list, A.plan, A.tab_off, smt);
    P.consts = rebase(A.consts, A.plan, A.tab_off, smt);
    P.cmat = rebase(reinterpret_cast<const unsigned char*>(A.cmat), A.plan, A.tab_off, smt);
    P.cang = rebase(reinterpret_cast<const unsigned char*>(A.cang), A.plan, A.tab_off, smt);
    const R* Pcmat = reinterpret_cast<const R*>(P.cmat);
    const R* Pcang = reinterpret_cast<const R*>(P.cang);
    __syncthreads();
    for (int i = threadIdx.x; i < A.n_sh; i += nthr) {
        const DEntry e = P.entries[vqc_ld(&P.sh_list[i])];
        eval_entry<R>(e, P.consts, static_cast<const R*>(nullptr), w_sm, Pcang, Pcmat,
                      sh_tab + EntryWords<R>::value * e.slot);
    }

    const int ns = A.nstages;
    for (int b = cid; b < A.nunits; b += ncl) {
        // this sample's x row, per-sample table and (given psi0) this CTA's slice
        for (int i = threadIdx.x; i < A.Px; i += nthr) xrow[i] = as_r<R>(A.x[(size_t)b * A.Px + i]);
        if (A.psi0) {
            const SC2<R>* gs = A.psi0 + ((size_t)b << n) + ((size_t)rank << slice);
            const uint32_t u0 = rank << slice;
            for (uint32_t v = threadIdx.x; v < (1u << slice); v += nthr)
                psi[swz(u0 + v, G) & ((1u << slice) - 1u)] = c2_in<R>(gs[v]);
        }
        __syncthreads();
        for (int i = threadIdx.x; i < A.n_ps; i += nthr) {
            const DEntry e = P.entries[vqc_ld(&P.ps_list[i])];
            eval_entry<R>(e, P.consts, xrow, w_sm, Pcang, Pcmat, ps_tab + EntryWords<R>::value * e.slot);
        }
        cluster_sync();   // tables ready here, every slice loaded cluster-wide

        C2<R> a[1 << K];
        int32_t sg[K];
        R eacc = 0;
        int eidx = 0;
        for (int s = 0; s < ns; ++s) {
            const DStage* sp = P.stages + s;
            const bool last = s + 1 == ns;
            const StageView v = stage_view<K>(sp, tg, 0, sg);
            const int loc = vqc_ld(&sp->cl_local);
            const int loc_next = last ? 1 : vqc_ld(&sp[1].cl_local);
            if (s == 0 && !A.psi0) {
#pragma unroll
                for (int r = 0; r < (1 << K); ++r) a[r] = cm<R>(0, 0);
                if (v.pb == 0) a[0] = cm<R>(1, 0);
            } else if (loc & 1) {   // every block in this CTA: plain shared loads
                block_load<R, K>(a, psi, v.swb & smask, sg);
            } else {
                cl_block_load<R, K>(a, psi_sa, slice, v.swb, sg);
            }
            run_ops<R, K, 0, false, true>(P.ops, vqc_ld(&sp->op_begin), vqc_ld(&sp->op_end), v.pb, a, a,
                                         sh_tab, ps_tab, nullptr, q, lane, warp);
            if (last) {   // <Z_j> partials: one butterfly per warp (n <= 16 here)
                R ez[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) ez[j] = 0;
                expz_accum<R, K, 16>(sp, v.pb, a, ez);
                eidx = warp_reduce_scatter<R, 16>(ez, lane);
                eacc = ez[0];
            }
            if (!last || A.state_out) {
                // Permuting store: every load that reads a slot it overwrites first
                // (only this CTA's threads read this CTA's slice when the loads are local).
                if (vqc_ld(&sp->nperm)) {
                    if (loc == 3) __syncthreads();
                    else cluster_sync();
                }
                int32_t s2[K];
                const uint32_t b2 = map_base<K, true>(sp, tg, 0, s2);
                if (loc & 2) block_store<R, K>(a, psi, b2 & smask, s2);
                else cl_block_store<R, K>(a, psi_sa, slice, b2, s2);
                // Data crosses CTAs only through a remote store here or a remote
                // load next; otherwise the CTA's own barrier orders the stages.
                if ((loc & 2) && (loc_next & 1)) __syncthreads();
                else cluster_sync();
            }
        }
        // E: warps -> CTA -> rank 0, summed in fixed order
        if ((lane & 1) == 0 && eidx < n) red[warp * n + eidx] = eacc;
        __syncthreads();
        for (int j = threadIdx.x; j < n; j += nthr) {
            R e = 0;
            for (int k = 0; k < nwarps; ++k) e += red[k * n + j];
            dsm_store(cluster_map(ecl_sa + (uint32_t)((rank * n + j) * sizeof(R)), 0), e);
        }
        cluster_sync();
        if (rank == 0)
            for (int j = threadIdx.x; j < n; j += nthr) {
                R e = 0;
                for (int r = 0; r < (1 << CL); ++r) e += ecl[r * n + j];
                A.E[(size_t)b * n + j] = as_out<St<R>>(e);
            }
        if (A.state_out) {   // this CTA's slice, logical order
            SC2<R>* go = A.state_out + ((size_t)b << n) + ((size_t)rank << slice);
            const uint32_t u0 = rank << slice;
            for (uint32_t v = threadIdx.x; v < (1u << slice); v += nthr)
                go[v] = c2_out<R>(psi[swz(u0 + v, G) & ((1u << slice) - 1u)]);
        }
        cluster_sync();   // slices and rank 0's gather area are reused by the next sample
    }
}

// Backward (adjoint) sweep of one sample per cluster, psi and lam each spread
// over the CTAs' shared memory in the forward's slice layout.  The stage walk is
// the resident backward's: stages in reverse, each loading both blocks through
// its store map, un-applying its ops with the rho accumulation, and storing
// through its load map; maps that leave the thread's CTA go through the cluster
// window.  Without psi_final the kernel first sweeps forward from psi0 (or
// |0...0>) with the same stages and keeps the last stage's block in registers.
//
// rho partials: the ops write one slot per (accumulator, warp) of which they
// use four reals, so two warps share each eight-real slot and the area holds
// [n_accs][warps][4].  After the sweep each CTA sums its warps in order, rank
// 0 sums the CTAs in rank order through the cluster window, turns the sums
// into gradient terms (with wg = 1), writes the sample's dx row and adds its
// dw terms to the cluster's running partial, written at the end to dw_part
// [cluster][Pw] (reduce_cols sums the rows in cluster order).
//
// KArgs fields used beyond the forward's: psi_final, gE, dx, dw_part, n_accs,
// n_terms, the accs / xocc / wocc tables, sm_lam, sm_acc, sm_terms, sm_dw, and
// sm_xg holding the sample's x row followed by its gE row.
template <typename R, int K>
__global__ void __launch_bounds__(512) cluster_bwd_kernel(const __grid_constant__ KArgs<St<R>> A) {
    uint32_t nrank;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(nrank));
    if (geometry_bad(((unsigned)blockDim.x << A.cl) != (unsigned)A.tpg || nrank != (1u << A.cl) ||
                         A.tpg != (1 << (A.n - K)) || A.nstages < 1 || (blockDim.x & 63u) != 0,
                     A.err, kErrClusterGeometry))
        return;
    extern __shared__ __align__(16) unsigned char smem[];
    R* sh_tab = reinterpret_cast<R*>(smem + A.sm_sh);
    R* ps_tab = reinterpret_cast<R*>(smem + A.sm_ps);
    C2<R>* psi = reinterpret_cast<C2<R>*>(smem + A.sm_psi);
    C2<R>* lam = reinterpret_cast<C2<R>*>(smem + A.sm_lam);
    R* acc = reinterpret_cast<R*>(smem + A.sm_acc);
    R* terms = reinterpret_cast<R*>(smem + A.sm_terms);
    R* dw_cta = reinterpret_cast<R*>(smem + A.sm_dw);
    R* w_sm = reinterpret_cast<R*>(smem + A.sm_w);
    R* xrow = reinterpret_cast<R*>(smem + A.sm_xg);

    const int n = A.n, G = A.G, CL = A.cl;
    const int slice = n - CL;
    const uint32_t smask = (1u << slice) - 1u;
    const uint32_t rank = cluster_rank();
    const int cid = (int)(blockIdx.x >> CL), ncl = (int)(gridDim.x >> CL);
    const int nthr = blockDim.x;
    const int tg = (int)rank * nthr + (int)threadIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = nthr >> 5;
    Geo q;
    q.T = A.tpg;
    q.lanes = 32;
    q.wg = nwarps;
    q.g = 0;
    q.t = tg;
    q.h = 0;
    q.mask = 0xffffffffu;
    // the ops address slot (k * wg + w) * 8: with wg halved, warp w / 2 and the
    // base moved by 4 reals for odd w, warp w's four reals sit at (k * warps + w) * 4
    Geo qa = q;
    qa.wg = nwarps >> 1;
    R* acc_w = acc + (warp & 1) * 4;
    const int warp_a = warp >> 1;
    const uint32_t psi_sa = static_cast<uint32_t>(__cvta_generic_to_shared(psi));
    const uint32_t lam_sa = static_cast<uint32_t>(__cvta_generic_to_shared(lam));
    const uint32_t acc_sa = static_cast<uint32_t>(__cvta_generic_to_shared(acc));

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
    async_wait();
    if constexpr (!std::is_same<St<R>, R>::value)
        for (int i = threadIdx.x; i < A.Pw; i += nthr) w_sm[i] = R(reinterpret_cast<const St<R>*>(w_sm)[i]);
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
    __syncthreads();
    for (int i = threadIdx.x; i < A.n_sh; i += nthr) {
        const DEntry e = P.entries[vqc_ld(&P.sh_list[i])];
        eval_entry<R>(e, P.consts, static_cast<const R*>(nullptr), w_sm, Pcang, Pcmat,
                      sh_tab + EntryWords<R>::value * e.slot);
    }

    const int ns = A.nstages;
    const bool recompute = A.psi_final == nullptr;
    const SC2<R>* src = recompute ? A.psi0 : A.psi_final;
    for (int b = cid; b < A.nunits; b += ncl) {
        // the sample's x and gE rows, per-sample table and this CTA's slice of
        // its final (or, recomputing from psi0, initial) state
        for (int i = threadIdx.x; i < A.Px + n; i += nthr)
            xrow[i] = i < A.Px ? as_r<R>(A.x[(size_t)b * A.Px + i]) : as_r<R>(A.gE[(size_t)b * n + (i - A.Px)]);
        if (src) {
            const SC2<R>* gs = src + ((size_t)b << n) + ((size_t)rank << slice);
            const uint32_t u0 = rank << slice;
            for (uint32_t v = threadIdx.x; v < (1u << slice); v += nthr)
                psi[swz(u0 + v, G) & smask] = c2_in<R>(gs[v]);
        }
        __syncthreads();
        for (int i = threadIdx.x; i < A.n_ps; i += nthr) {
            const DEntry e = P.entries[vqc_ld(&P.ps_list[i])];
            eval_entry<R>(e, P.consts, xrow, w_sm, Pcang, Pcmat, ps_tab + EntryWords<R>::value * e.slot);
        }
        cluster_sync();   // tables ready, every slice loaded cluster-wide

        C2<R> a[1 << K];
        C2<R> l[1 << K];
        int32_t sg[K];
        if (recompute) {   // forward with the same stages; the last block stays in registers
            for (int s = 0; s < ns; ++s) {
                const DStage* sp = P.stages + s;
                const StageView v = stage_view<K>(sp, tg, 0, sg);
                const int loc = vqc_ld(&sp->cl_local);
                if (s == 0 && !A.psi0) {
#pragma unroll
                    for (int r = 0; r < (1 << K); ++r) a[r] = cm<R>(0, 0);
                    if (v.pb == 0) a[0] = cm<R>(1, 0);
                } else if (loc & 1) {
                    block_load<R, K>(a, psi, v.swb & smask, sg);
                } else {
                    cl_block_load<R, K>(a, psi_sa, slice, v.swb, sg);
                }
                run_ops<R, K, 0, false, true>(P.ops, vqc_ld(&sp->op_begin), vqc_ld(&sp->op_end), v.pb, a, a,
                                             sh_tab, ps_tab, nullptr, q, lane, warp);
                if (s + 1 == ns) break;
                if (vqc_ld(&sp->nperm)) {
                    if (loc == 3) __syncthreads();
                    else cluster_sync();
                }
                int32_t s2[K];
                const uint32_t b2 = map_base<K, true>(sp, tg, 0, s2);
                if (loc & 2) block_store<R, K>(a, psi, b2 & smask, s2);
                else cl_block_store<R, K>(a, psi_sa, slice, b2, s2);
                if ((loc & 2) && (vqc_ld(&sp[1].cl_local) & 1)) __syncthreads();
                else cluster_sync();
            }
        }

        for (int s = ns - 1; s >= 0; --s) {
            const DStage* sp = P.stages + s;
            const StageView v = stage_view<K>(sp, tg, 0, sg);
            const int loc = vqc_ld(&sp->cl_local);
            if (s == ns - 1) {   // the final state in the last stage's frame (its store map is the identity)
                if (!recompute) {
                    if (loc & 1) block_load<R, K>(a, psi, v.swb & smask, sg);
                    else cl_block_load<R, K>(a, psi_sa, slice, v.swb, sg);
                }
                lambda_init<R, K>(sp, v.pb, xrow + A.Px, n, a, l);
            } else {   // stage s's output, where its store map left it
                int32_t s2[K];
                const uint32_t b2 = map_base<K, true>(sp, tg, 0, s2);
                if (loc & 2) {
                    block_load<R, K>(a, psi, b2 & smask, s2);
                    block_load<R, K>(l, lam, b2 & smask, s2);
                } else {
                    cl_block_load<R, K>(a, psi_sa, slice, b2, s2);
                    cl_block_load<R, K>(l, lam_sa, slice, b2, s2);
                }
            }
            run_ops<R, K, 1, false, true>(P.ops, vqc_ld(&sp->op_begin), vqc_ld(&sp->op_end), v.pb, a, l,
                                         sh_tab, ps_tab, acc_w, qa, lane, warp_a);
            if (s > 0) {   // back to the stage's input layout (load map)
                if (vqc_ld(&sp->nperm)) {
                    if (loc == 3) __syncthreads();
                    else cluster_sync();
                }
                int32_t s2[K];
                const uint32_t b2 = map_base<K, false>(sp, tg, 0, s2);
                if (loc & 1) {
                    block_store<R, K>(a, psi, b2 & smask, s2);
                    block_store<R, K>(l, lam, b2 & smask, s2);
                } else {
                    cl_block_store<R, K>(a, psi_sa, slice, b2, s2);
                    cl_block_store<R, K>(l, lam_sa, slice, b2, s2);
                }
                // stage s - 1 loads through its store map next
                if ((loc & 1) && (vqc_ld(&sp[-1].cl_local) & 2)) __syncthreads();
                else cluster_sync();
            }
        }
        __syncthreads();
        // this CTA's warps, in warp order, into warp 0's four reals
        for (int k = threadIdx.x; k < A.n_accs; k += nthr) {
            R* ap = acc + (size_t)k * nwarps * 4;
            R t0 = 0, t1 = 0, t2 = 0, t3 = 0;
            for (int w = 0; w < nwarps; ++w) {
                t0 += ap[w * 4 + 0];
                t1 += ap[w * 4 + 1];
                t2 += ap[w * 4 + 2];
                t3 += ap[w * 4 + 3];
            }
            ap[0] = t0; ap[1] = t1; ap[2] = t2; ap[3] = t3;
        }
        cluster_sync();
        if (rank == 0)   // the CTAs in rank order
            for (int k = threadIdx.x; k < A.n_accs; k += nthr) {
                const uint32_t off = (uint32_t)((size_t)k * nwarps * 4 * sizeof(R));
                R t[4] = {0, 0, 0, 0};
                for (uint32_t r = 0; r < (1u << CL); ++r)
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        R vr;
                        dsm_load_r(cluster_map(acc_sa + off + (uint32_t)(i * sizeof(R)), r), &vr);
                        t[i] += vr;
                    }
                R* ap = acc + (size_t)k * nwarps * 4;
#pragma unroll
                for (int i = 0; i < 4; ++i) ap[i] = t[i];
            }
        // rank 0 has read every CTA's sums: slices and accumulators are free again
        cluster_sync();
        if (rank == 0) {
            for (int k = threadIdx.x; k < A.n_accs; k += nthr) {
                const DAcc ac = P.accs[k];
                acc_terms<R>(ac, P.entries[ac.entry], acc + (size_t)k * nwarps * 4, 1, P.consts, xrow, w_sm,
                             Pcang, Pcmat, terms);
            }
            __syncthreads();
            if (A.dx)
                for (int p = threadIdx.x; p < A.Px; p += nthr) {
                    const int k0 = vqc_ld(&P.xocc_ptr[p]), k1 = vqc_ld(&P.xocc_ptr[p + 1]);
                    R sum = 0;
                    for (int k = k0; k < k1; ++k) sum += terms[vqc_ld(&P.xocc[k])];
                    A.dx[(size_t)b * A.Px + p] = as_out<St<R>>(sum);
                }
            for (int p = threadIdx.x; p < A.Pw; p += nthr) {
                const int k0 = vqc_ld(&P.wocc_ptr[p]), k1 = vqc_ld(&P.wocc_ptr[p + 1]);
                R sum = dw_cta[p];
                for (int k = k0; k < k1; ++k) sum += terms[vqc_ld(&P.wocc[k])];
                dw_cta[p] = sum;
            }
        }
    }
    if (rank == 0 && A.Pw > 0 && A.dw_part)
        for (int p = threadIdx.x; p < A.Pw; p += nthr)
            A.dw_part[(size_t)cid * A.Pw + p] = as_out<St<R>>(dw_cta[p]);
}

}  // namespace vqc
