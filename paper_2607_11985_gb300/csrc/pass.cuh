// pass.cuh -- HBM-tiled path for states that do not fit one SM's shared memory
// (paper, Sec. 3 "Complexity and Tradeoffs": the state, O(B 2^n), is the
// memory wall; here it lives in HBM between passes).
//
// The compiler cuts the op list into passes.  A pass acts on tiles of m
// qubits: the tile qubits always include the low qubits whose 2^G amplitudes
// form one 128-byte chunk, so a tile is gathered from HBM as whole chunks.
// One launch per pass: each CTA loads S tiles (the other n - m qubits fix the
// tile), runs the pass's register-block stages on them in shared memory
// exactly as the resident path does, and writes them back.  The forward's last
// pass emits per-tile <Z> partials; the backward emits per-tile rho sums of
// the pass's accumulators, which reduce_terms adds up per sample and turns into
// gradient terms.  reduce_* kernels sum partials in a fixed order
// (deterministic).
#pragma once

#include "sweep.cuh"

namespace vqc {

// R here is the storage real type (pass kernels take PArgs<St<R>>).
template <typename R>
struct PArgs {
    const DOp* ops;
    const DStage* stages;
    const int32_t* pass_entries;
    const int32_t* pass_accs;
    const DEntry* entries;
    const DConst* consts;
    const R* cmat;
    const R* cang;
    const DAcc* accs;
    int n, m, K, tbits, G, S, nout, ntiles;
    int stage_begin, stage_end;
    int ps_begin, ps_count, sh_begin, sh_count, acc_begin, acc_count, n_accs, Px;
    const void* ps_g;       // per-sample tables of every sample [B][n_ps][entry words] (ps_tables),
                            // kernel real type (not read by the complex64 backward)
    int n_ps;
    int B;
    long long nunits;
    uint8_t tile_q[24], out_q[24];
    const R* x;
    const R* w;
    const R* gE;
    const C2<R>* src_psi;   // tiles are read from here (nullptr: start from |0...0>)
    C2<R>* dst_psi;         // and written back here (nullptr: not written)
    const C2<R>* src_lam;   // backward: lam tiles (nullptr: lam = O psi in the first stage)
    C2<R>* dst_lam;
    R* E_part;              // forward, last pass: [B * ntiles, n]
    R* rho;                 // backward: per-tile rho sums [B * ntiles][n_accs][4] (3 used)
    int sm_sh, sm_ps, sm_psi, sm_lam, sm_acc, sm_red;
    const unsigned char* plan;   // plan regions copied to shared memory (see KArgs)
    int tab_off, tab_bytes, sched_off, sched_bytes, sm_plan, plan_smem;
    int sm_koff;                 // per-pass tile-copy offsets: [ceil(2^m / (APV * T))] uint2
    unsigned* err;               // the plan's error word (launch self-check)
    // double-float kernels only: src_psi / src_lam / dst_psi and dst_lam hold
    // raw (hi, lo) float pairs (workspace state passed between passes) rather
    // than complex128 values (caller buffers); ignored by other kernels
    int src_raw, lam_raw, dst_raw;
};

// Global amplitude index of tile-local index u (the low G tile bits are the
// low G qubits; the rest follow tile_q).
__device__ __forceinline__ uint32_t tile_global(uint32_t u, uint32_t tile_base, const uint8_t* tq,
                                                int G) {
    uint32_t g = tile_base | (u & ((1u << G) - 1u));
    uint32_t hi = u >> G;
    for (int i = G; hi; ++i, hi >>= 1)
        if (hi & 1u) g |= 1u << tq[i];
    return g;
}

// 16-byte vectors of amplitudes, moved without taking register addresses.
template <typename R> struct Vec16;
template <> struct Vec16<float> {
    float2 a[2];
    __device__ __forceinline__ void ld(const float2* p) {
        const float4 v = __ldcs(reinterpret_cast<const float4*>(p));
        a[0] = make_float2(v.x, v.y);
        a[1] = make_float2(v.z, v.w);
    }
    __device__ __forceinline__ void st(float2* p) const {
        __stcs(reinterpret_cast<float4*>(p), make_float4(a[0].x, a[0].y, a[1].x, a[1].y));
    }
};
template <> struct Vec16<double> {
    double2 a[1];
    __device__ __forceinline__ void ld(const double2* p) { a[0] = __ldcs(p); }
    __device__ __forceinline__ void st(double2* p) const { __stcs(p, a[0]); }
};
// double-float kernels: complex128 in HBM, split on the way in, rejoined on the way out
template <> struct Vec16<dd> {
    dd2 a[1];
    __device__ __forceinline__ void ld(const double2* p) { a[0] = c2_in<dd>(__ldcs(p)); }
    __device__ __forceinline__ void st(double2* p) const { __stcs(p, c2_out<dd>(a[0])); }
};
// raw (hi, lo) pairs in a workspace buffer between double-float passes: no
// conversion (the conversions run on the FP64 units, a pass's slowest work)
struct Vec16Raw {
    dd2 a[1];
    __device__ __forceinline__ void ld(const double2* p) {
        const float4 v = __ldcs(reinterpret_cast<const float4*>(p));
        a[0].x = dd(v.x, v.y);
        a[0].y = dd(v.z, v.w);
    }
    __device__ __forceinline__ void st(double2* p) const {
        __stcs(reinterpret_cast<float4*>(p), make_float4(a[0].x.hi, a[0].x.lo, a[0].y.hi, a[0].y.lo));
    }
};
template <typename R, bool RAW> struct VecSel { using t = Vec16<R>; };
template <> struct VecSel<dd, true> { using t = Vec16Raw; };

// Tile copies between HBM and shared memory.  A CTA-thread t moves vectors
// v = t + k*T; the tile-local index of v splits into disjoint bit fields of t
// and of k, and both the index deposit into global qubits and the swizzle are
// linear in those fields, so each is a per-thread part XOR a per-k part
// (tabulated once per pass in shared memory: koff[k] = (global, slot)).
template <typename R, bool RAW = false, int U = 8>
__device__ __forceinline__ void tile_gather(C2<R>* sm, const SC2<R>* gs, uint32_t gt, uint32_t st,
                                            const uint2* koff, int nk, int T, int t) {
    using V = typename VecSel<R, RAW>::t;
    constexpr int APV = 16 / sizeof(C2<R>);
    int k = 0;
    for (; k + U <= nk; k += U) {
        V v[U];
#pragma unroll
        for (int j = 0; j < U; ++j) v[j].ld(gs + (gt | koff[k + j].x));
#pragma unroll
        for (int j = 0; j < U; ++j) {
            const uint32_t sl = st ^ koff[k + j].y;
#pragma unroll
            for (int e = 0; e < APV; ++e) sm[sl ^ e] = v[j].a[e];
        }
    }
    for (; k < nk; ++k) {
        V v;
        v.ld(gs + (gt | koff[k].x));
        const uint32_t sl = st ^ koff[k].y;
#pragma unroll
        for (int e = 0; e < APV; ++e) sm[sl ^ e] = v.a[e];
    }
}

template <typename R, bool RAW = false>
__device__ __forceinline__ void tile_scatter(const C2<R>* sm, SC2<R>* gs, uint32_t gt, uint32_t st,
                                             const uint2* koff, int nk, int T, int t) {
    using V = typename VecSel<R, RAW>::t;
    constexpr int APV = 16 / sizeof(C2<R>);
    for (int k = 0; k < nk; ++k) {
        V v;
        const uint32_t sl = st ^ koff[k].y;
#pragma unroll
        for (int e = 0; e < APV; ++e) v.a[e] = sm[sl ^ e];
        v.st(gs + (gt | koff[k].x));
    }
}

// Bring a tile's 128-byte lines into L2 ahead of its gather (a hint: no result,
// no wait).  With T >= 8 (every production tile) vectors t .. t+7 of one k
// share a line, so every eighth thread takes the lines; smaller groups touch
// some lines more than once.
template <typename R>
__device__ __forceinline__ void tile_prefetch(const SC2<R>* gs, uint32_t gt, const uint2* koff, int nk,
                                              int t) {
    if (t & 7) return;
    for (int k = 0; k < nk; ++k)
        asm volatile("prefetch.global.L2 [%0];" ::"l"(gs + (gt | koff[k].x)));
}

// FULL: tile groups span whole warps (2^(m-K) >= 32 threads; every production
// tile), see sweep_kernel.
template <typename R, int K, int MODE, bool FULL, bool PH2 = true>
__global__ void __launch_bounds__(256, 2) pass_kernel(const __grid_constant__ PArgs<St<R>> A) {
    if (geometry_bad(blockDim.x != (unsigned)(A.S << A.tbits) || A.tbits != A.m - K ||
                         A.stage_end <= A.stage_begin,
                     A.err, kErrPassGeometry))
        return;
    extern __shared__ __align__(16) unsigned char smem[];
    R* sh_tab = reinterpret_cast<R*>(smem + A.sm_sh);
    R* ps_all = reinterpret_cast<R*>(smem + A.sm_ps);
    C2<R>* psi_all = reinterpret_cast<C2<R>*>(smem + A.sm_psi);
    C2<R>* lam_all = reinterpret_cast<C2<R>*>(smem + A.sm_lam);
    R* acc_all = reinterpret_cast<R*>(smem + A.sm_acc);
    R* red_all = reinterpret_cast<R*>(smem + A.sm_red);

    const unsigned char* smt = nullptr;
    const unsigned char* sms = nullptr;
    if (A.plan_smem) {
        unsigned char* t = smem + A.sm_plan;
        unsigned char* u = t + ((A.tab_bytes + 15) & ~15);
        copy_region(t, A.plan + A.tab_off, A.tab_bytes);
        copy_region(u, A.plan + A.sched_off, A.sched_bytes);
        smt = t;
        sms = u;
    }
    grid_dep_wait();
    grid_dep_launch();
    const DOp* P_ops = rebase(A.ops, A.plan, A.sched_off, sms);
    const DStage* P_stages = rebase(A.stages, A.plan, A.sched_off, sms);
    const int32_t* P_pass_entries = rebase(A.pass_entries, A.plan, A.sched_off, sms);
    const int32_t* P_pass_accs = rebase(A.pass_accs, A.plan, A.sched_off, sms);
    const DEntry* P_entries = rebase(A.entries, A.plan, A.tab_off, smt);
    const DConst* P_consts = rebase(A.consts, A.plan, A.tab_off, smt);
    const R* P_cmat = reinterpret_cast<const R*>(
        rebase(reinterpret_cast<const unsigned char*>(A.cmat), A.plan, A.tab_off, smt));
    const R* P_cang = reinterpret_cast<const R*>(
        rebase(reinterpret_cast<const unsigned char*>(A.cang), A.plan, A.tab_off, smt));
    if (A.plan_smem) __syncthreads();

    const int n = A.n, G = A.G, tdim = 1 << A.m;
    const long long total_tiles = (long long)A.B * A.ntiles;
    constexpr bool DDK = !std::is_same<St<R>, R>::value;   // double-float kernel
    Geo q;
    q.T = 1 << A.tbits;
    q.lanes = q.T < 32 ? q.T : 32;
    q.wg = q.T > 32 ? q.T / 32 : 1;
    q.g = threadIdx.x / q.T;
    q.t = threadIdx.x % q.T;
    q.h = 0;
    if (A.tbits < G) q.h = ((q.g & ((1 << (G - A.tbits)) - 1)) << A.tbits) & (tdim - 1);
    q.mask = blockDim.x >= 32 ? 0xffffffffu : ((1u << blockDim.x) - 1u);
    const int lane = q.t & 31;
    const int warp_in_group = q.t >> 5;
    const int nthr = blockDim.x;

    // Tile copy geometry: vectors v = t + k*T of APV amplitudes.
    constexpr int APV = 16 / sizeof(C2<R>);
    const int nvec = tdim / APV;
    const int nk = (nvec + q.T - 1) / q.T;
    uint2* koff = reinterpret_cast<uint2*>(smem + A.sm_koff);
    for (int k = threadIdx.x; k < nk; k += nthr) {
        const uint32_t u = (uint32_t)k * q.T * APV;
        koff[k] = make_uint2(tile_global(u, 0, A.tile_q, G), swz(u, G));
    }
    const uint32_t u_t = (uint32_t)q.t * APV;
    const uint32_t st_t = swz(u_t, G) ^ (uint32_t)q.h;

    for (int i = threadIdx.x; i < A.sh_count; i += nthr) {
        const DEntry e = P_entries[vqc_ld(&P_pass_entries[A.sh_begin + i])];
        eval_entry<R>(e, P_consts, static_cast<const St<R>*>(nullptr), A.w, P_cang, P_cmat,
                      sh_tab + EntryWords<R>::value * i);
    }
    __syncthreads();

    C2<R>* psi = psi_all + (size_t)q.g * tdim;
    C2<R>* lam = lam_all + (size_t)q.g * tdim;
    R* ps_tab = ps_all + (size_t)q.g * A.ps_count * EntryWords<R>::value;
    R* acc = acc_all + (size_t)q.g * A.acc_count * q.wg * 8;

    for (long long unit = blockIdx.x; unit < A.nunits; unit += gridDim.x) {
        const long long tid_raw = unit * A.S + q.g;
        const bool valid = tid_raw < total_tiles;
        const long long tile_id = valid ? tid_raw : total_tiles - 1;
        const int b = (int)(tile_id / A.ntiles);
        const int tau = (int)(tile_id % A.ntiles);
        uint32_t tile_base = 0;
        for (int j = 0; j < A.nout; ++j)
            if ((tau >> j) & 1) tile_base |= 1u << A.out_q[j];

        if (MODE == 1 && std::is_same<R, float>::value) {
            // the complex64 backward evaluates its per-sample entries itself: with
            // the table copy instead its register allocation spilled more and it
            // measured 0.7% slower (the other kernels read the table)
            for (int i = threadIdx.x; i < A.S * A.ps_count; i += nthr) {
                const int gg = i / A.ps_count, k = i % A.ps_count;
                const long long tt = min(unit * A.S + gg, total_tiles - 1);
                const int bb = (int)(tt / A.ntiles);
                const DEntry e = P_entries[vqc_ld(&P_pass_entries[A.ps_begin + k])];
                eval_entry<R>(e, P_consts, A.x + (size_t)bb * A.Px, A.w, P_cang, P_cmat,
                              ps_all + ((size_t)gg * A.ps_count + k) * EntryWords<R>::value);
            }
        } else if (A.ps_count) {   // the pass's per-sample entries, copied from the sample's precomputed table
            constexpr int V = EntryWords<R>::value * (int)sizeof(R) / 16;   // 16-byte vectors per entry
            const int4* gtab = static_cast<const int4*>(A.ps_g);
            int4* stab = reinterpret_cast<int4*>(ps_all);
            const int per = A.ps_count * V;
            for (int i = threadIdx.x; i < A.S * per; i += nthr) {
                const int gg = i / per, r = i - gg * per, k = r / V, v = r - k * V;
                const int bb = (int)(min(unit * A.S + gg, total_tiles - 1) / A.ntiles);
                const int slot = P_entries[vqc_ld(&P_pass_entries[A.ps_begin + k])].slot;
                stab[((size_t)gg * A.ps_count + k) * V + v] = gtab[((size_t)bb * A.n_ps + slot) * V + v];
            }
        }
        const size_t sbase = (size_t)b << n;
        const uint32_t gt = tile_global(u_t, tile_base, A.tile_q, G);
        if (A.src_psi) {
            if (DDK && A.src_raw) tile_gather<R, DDK>(psi, A.src_psi + sbase, gt, st_t, koff, nk, q.T, q.t);
            else   // 16 loads in flight where one state is gathered, 8 beside lam's registers
                tile_gather<R, false, MODE == 0 ? 16 : 8>(psi, A.src_psi + sbase, gt, st_t, koff, nk, q.T, q.t);
        }
        if (MODE == 1 && A.src_lam) {
            if (DDK && A.lam_raw) tile_gather<R, DDK>(lam, A.src_lam + sbase, gt, st_t, koff, nk, q.T, q.t);
            else tile_gather<R>(lam, A.src_lam + sbase, gt, st_t, koff, nk, q.T, q.t);
        }
        if (unit + gridDim.x < A.nunits) {   // the CTA's next tile into L2 during this one's stages
            const long long nt = min((unit + gridDim.x) * A.S + q.g, total_tiles - 1);
            const int nb = (int)(nt / A.ntiles), ntau = (int)(nt % A.ntiles);
            uint32_t nbase = 0;
            for (int j = 0; j < A.nout; ++j)
                if ((ntau >> j) & 1) nbase |= 1u << A.out_q[j];
            const uint32_t ngt = tile_global(u_t, nbase, A.tile_q, G);
            const size_t nsb = (size_t)nb << n;
            if (A.src_psi) tile_prefetch<R>(A.src_psi + nsb, ngt, koff, nk, q.t);
            if (MODE == 1 && A.src_lam) tile_prefetch<R>(A.src_lam + nsb, ngt, koff, nk, q.t);
        }
        __syncthreads();

        C2<R> a[1 << K];
        int32_t sg[K];
        StageView v{0, 0};
        if (MODE == 0) {
            for (int s = A.stage_begin; s < A.stage_end; ++s) {
                const DStage* sp = P_stages + s;
                v = stage_view<K>(sp, q.t, q.h, sg);
                v.pb |= tile_base;
                if (s == A.stage_begin && !A.src_psi) {
#pragma unroll
                    for (int r = 0; r < (1 << K); ++r) a[r] = cm<R>(0, 0);
                    if (v.pb == 0) a[0] = cm<R>(1, 0);
                } else {
                    block_load<R, K>(a, psi, v.swb, sg);
                }
                run_ops<R, K, 0, true, FULL, PH2>(P_ops, vqc_ld(&sp->op_begin), vqc_ld(&sp->op_end), v.pb, a, a,
                                 sh_tab, ps_tab, nullptr, q, lane, warp_in_group);
                if (s + 1 < A.stage_end || A.dst_psi) {   // store map: absorbed CX gates
                    if (vqc_ld(&sp->nperm)) group_sync<R>(q);   // all loads of the stage first
                    int32_t s2[K];
                    const uint32_t b2 = map_base<K, true>(sp, q.t, q.h, s2);
                    block_store<R, K>(a, psi, b2, s2);
                    group_sync<R>(q);
                }
            }
            if (A.E_part) {
                R* red = red_all + (size_t)q.g * q.wg * n;
                expz_partials<R, K>(P_stages + (A.stage_end - 1), v.pb, a, n, red, q, warp_in_group);
                __syncthreads();
                if (valid)
                    for (int j = q.t; j < n; j += q.T) {
                        R e = 0;
                        for (int k = 0; k < q.wg; ++k) e += red[k * n + j];
                        A.E_part[tile_id * n + j] = as_out<St<R>>(e);
                    }
            }
            __syncthreads();
            if (A.dst_psi && valid) {
                if (DDK && A.dst_raw) tile_scatter<R, DDK>(psi, A.dst_psi + sbase, gt, st_t, koff, nk, q.T, q.t);
                else tile_scatter<R>(psi, A.dst_psi + sbase, gt, st_t, koff, nk, q.T, q.t);
            }
            __syncthreads();
            continue;
        }

        // backward: stages of the pass in reverse
        for (int s = A.stage_end - 1; s >= A.stage_begin; --s) {
            const DStage* sp = P_stages + s;
            C2<R> l[1 << K];
            v = stage_view<K>(sp, q.t, q.h, sg);
            v.pb |= tile_base;
            {   // the forward left this stage's output in its store map
                int32_t s2[K];
                const uint32_t b2 = map_base<K, true>(sp, q.t, q.h, s2);
                block_load<R, K>(a, psi, b2, s2);
                if (s == A.stage_end - 1 && !A.src_lam)
                    lambda_init<R, K>(sp, v.pb, A.gE + (size_t)b * n, n, a, l);
                else
                    block_load<R, K>(l, lam, b2, s2);
            }
            run_ops<R, K, 1, true, FULL, PH2>(P_ops, vqc_ld(&sp->op_begin), vqc_ld(&sp->op_end), v.pb, a, l, sh_tab,
                             ps_tab, acc, q, lane, warp_in_group);
            if (s > A.stage_begin || A.dst_psi) {   // back to the stage's load map
                if (vqc_ld(&sp->nperm)) group_sync<R>(q);   // all loads of the stage first
                int32_t s2[K];
                const uint32_t b2 = map_base<K, false>(sp, q.t, q.h, s2);
                block_store<R, K>(a, psi, b2, s2);
                block_store<R, K>(l, lam, b2, s2);
            }
            group_sync<R>(q);
        }
        __syncthreads();
        if (valid && A.dst_psi) {
            if (DDK && A.dst_raw) {
                tile_scatter<R, DDK>(psi, A.dst_psi + sbase, gt, st_t, koff, nk, q.T, q.t);
                tile_scatter<R, DDK>(lam, A.dst_lam + sbase, gt, st_t, koff, nk, q.T, q.t);
            } else {
                tile_scatter<R>(psi, A.dst_psi + sbase, gt, st_t, koff, nk, q.T, q.t);
                tile_scatter<R>(lam, A.dst_lam + sbase, gt, st_t, koff, nk, q.T, q.t);
            }
        }
        // the tile's rho sums (warps in order), in parallel over accumulators and
        // components; the per-sample turn into terms is reduce_terms' work
        for (int i = threadIdx.x; i < A.S * A.acc_count * 3; i += nthr) {
            const int gg = i / (A.acc_count * 3), r = i % (A.acc_count * 3), k = r / 3, c = r % 3;
            const long long tt = unit * A.S + gg;
            if (tt >= total_tiles) continue;
            const R* ap = acc_all + ((size_t)gg * A.acc_count + k) * q.wg * 8 + c;
            R sum = 0;
            for (int wi = 0; wi < q.wg; ++wi) sum += ap[wi * 8];
            A.rho[((size_t)tt * A.n_accs + vqc_ld(&P_pass_accs[A.acc_begin + k])) * 4 + c] = as_out<St<R>>(sum);
        }
        __syncthreads();
    }
}

// E[b, j] = sum over tiles of E_part[b * ntiles + tau, j]  (fixed order).
template <typename R>
__global__ void reduce_expz(const R* E_part, int B, int ntiles, int n, R* E) {
    grid_dep_wait();
    grid_dep_launch();
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < (long long)B * n;
         i += (long long)gridDim.x * blockDim.x) {
        const long long b = i / n, j = i % n;
        R s = 0;
        for (int t = 0; t < ntiles; ++t) s += E_part[(b * ntiles + t) * n + j];
        E[i] = s;
    }
}

// Per-sample table entries of every sample (the x-dependent runs), evaluated
// once per call for all passes: out [B][n_ps][entry words], in the kernels'
// real type R (slot order = ps_list order).
template <typename R>
__global__ void __launch_bounds__(256) ps_tables(const DEntry* entries, const int32_t* ps_list,
                                                 const DConst* consts, const R* cang, const R* cmat,
                                                 const St<R>* x, int Px, const St<R>* w, int B, int n_ps,
                                                 R* out) {
    grid_dep_wait();
    grid_dep_launch();
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < (long long)B * n_ps;
         i += (long long)gridDim.x * blockDim.x) {
        const long long b = i / n_ps;
        const DEntry e = entries[vqc_ld(&ps_list[i % n_ps])];
        eval_entry<R>(e, consts, x + b * Px, w, cang, cmat,
                      out + ((size_t)b * n_ps + e.slot) * EntryWords<R>::value);
    }
}

// Gradient terms of every accumulator of every sample: the sample's per-tile
// rho sums added in tile order, then the constituent walk of acc_terms (one
// partial), in the kernels' arithmetic R (the plan's constants are stored as R:
// (hi, lo) float pairs for double-float plans).  terms: [B, n_terms].
template <typename R>
__global__ void __launch_bounds__(256) reduce_terms(const St<R>* rho, int B, int ntiles, int n_accs,
                                                    const DAcc* accs, const DEntry* entries,
                                                    const DConst* consts, const R* cang, const R* cmat,
                                                    const St<R>* x, int Px, const St<R>* w, int n_terms,
                                                    St<R>* terms) {
    grid_dep_wait();
    grid_dep_launch();
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < (long long)B * n_accs;
         i += (long long)gridDim.x * blockDim.x) {
        const long long b = i / n_accs;
        const int k = (int)(i % n_accs);
        R t[4] = {0, 0, 0, 0};
        for (int tau = 0; tau < ntiles; ++tau) {
            const St<R>* r = rho + ((b * ntiles + tau) * n_accs + k) * 4;
            t[0] += as_r<R>(r[0]);
            t[1] += as_r<R>(r[1]);
            t[2] += as_r<R>(r[2]);
        }
        const DAcc ac = accs[k];
        acc_terms<R>(ac, entries[ac.entry], t, 1, consts,
                     x ? x + b * Px : static_cast<const St<R>*>(nullptr), w, cang, cmat, terms + b * n_terms);
    }
}

// dx[b, p] = sum_tau sum_{terms j of x column p} terms[b * ntiles + tau, j]
template <typename R>
__global__ void reduce_dx(const R* terms, int B, int ntiles, int nt, const int32_t* ptr,
                          const int32_t* occ, int Px, R* dx) {
    grid_dep_wait();
    grid_dep_launch();
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < (long long)B * Px;
         i += (long long)gridDim.x * blockDim.x) {
        const long long b = i / Px;
        const int p = (int)(i % Px);
        R s = 0;
        for (int t = 0; t < ntiles; ++t) {
            const R* row = terms + (b * ntiles + t) * nt;
            for (int k = vqc_ld(&ptr[p]); k < vqc_ld(&ptr[p + 1]); ++k) s += row[vqc_ld(&occ[k])];
        }
        dx[i] = s;
    }
}

// dw[p] = sum over every tile row of the terms of w index p: one block per p,
// fixed strided partial sums then a fixed-shape tree.
template <typename R>
__global__ void __launch_bounds__(256) reduce_dw(const R* terms, long long rows, int nt,
                                                 const int32_t* ptr, const int32_t* occ, R* dw) {
    __shared__ R part[256];
    const int p = blockIdx.x;
    grid_dep_wait();
    grid_dep_launch();
    const int k0 = vqc_ld(&ptr[p]), k1 = vqc_ld(&ptr[p + 1]);
    R s = 0;
    for (long long r = threadIdx.x; r < rows; r += 256) {
        const R* row = terms + r * nt;
        for (int k = k0; k < k1; ++k) s += row[vqc_ld(&occ[k])];
    }
    part[threadIdx.x] = s;
    __syncthreads();
    for (int w = 128; w >= 1; w >>= 1) {
        if (threadIdx.x < w) part[threadIdx.x] += part[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) dw[p] = part[0];
}

// probs[i] = |psi[i]|^2 over count amplitudes (the probabilities output).
template <typename R>
__global__ void __launch_bounds__(256) abs2_kernel(const C2<R>* psi, long long count, R* probs) {
    grid_dep_wait();
    grid_dep_launch();
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < count;
         i += (long long)gridDim.x * blockDim.x) {
        const C2<R> v = psi[i];
        probs[i] = fma(v.x, v.x, v.y * v.y);
    }
}

}  // namespace vqc
