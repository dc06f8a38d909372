// capi.cu -- the C ABI declared in include/vqc.h: plan lifetime, launch
// geometry, workspace layout and kernel launches.  No exception crosses the
// ABI; every entry point returns a vqc_status and records a thread-local
// message on failure.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdlib>
#include <cstring>
#include <initializer_list>
#include <map>
#include <memory>
#include <mutex>
#include <new>
#include <set>
#include <string>
#include <vector>

#include "engine.h"
#include "kernels.h"
#include "pass.cuh"
#include "sweep.cuh"

namespace vqc {
namespace {
// Launch geometry depends only on (plan, mode, batch, device): cache it so a
// call does not repeat the attribute and occupancy queries.
struct GeoKey {
    const void* plan;
    int mode, batch, dev, hbm;
    bool operator<(const GeoKey& o) const {
        if (plan != o.plan) return plan < o.plan;
        if (mode != o.mode) return mode < o.mode;
        if (batch != o.batch) return batch < o.batch;
        if (dev != o.dev) return dev < o.dev;
        return hbm < o.hbm;
    }
};
}  // namespace
}  // namespace vqc

namespace vqc {
namespace {

thread_local std::string g_err;

vqc_status fail(vqc_status s, const std::string& msg) {
    g_err = msg;
    return s;
}

vqc_status cuda_fail(cudaError_t e, const char* what) {
    return fail(VQC_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

#define VQC_CUDA(call)                                          \
    do {                                                        \
        cudaError_t e_ = (call);                                \
        if (e_ != cudaSuccess) return cuda_fail(e_, #call);     \
    } while (0)

struct DevInfo {
    int sms = 0, smem_optin = 0;
    bool ok = false;
};

std::mutex g_mu;
std::vector<DevInfo> g_dev;

vqc_status device_info(int dev, DevInfo& out) {
    std::lock_guard<std::mutex> lk(g_mu);
    if ((int)g_dev.size() <= dev) g_dev.resize(dev + 1);
    if (!g_dev[dev].ok) {
        VQC_CUDA(cudaDeviceGetAttribute(&g_dev[dev].sms, cudaDevAttrMultiProcessorCount, dev));
        VQC_CUDA(cudaDeviceGetAttribute(&g_dev[dev].smem_optin,
                                        cudaDevAttrMaxSharedMemoryPerBlockOptin, dev));
        g_dev[dev].ok = true;
    }
    out = g_dev[dev];
    return VQC_OK;
}

// Let `fn` take up to the device's opt-in shared memory per CTA, once per
// (kernel, device).  The attribute is per kernel, not per launch geometry:
// setting it to each geometry's own need would let a later, smaller geometry of
// the same kernel (another plan, batch or environment setting) lower it below a
// cached larger geometry's need, whose launch would then fail.
std::mutex g_smem_attr_mu;
std::set<std::pair<const void*, int>> g_smem_attr_done;

vqc_status allow_max_smem(const void* fn, int dev, int smem_optin) {
    std::lock_guard<std::mutex> lk(g_smem_attr_mu);
    if (g_smem_attr_done.count({fn, dev})) return VQC_OK;
    VQC_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_optin));
    g_smem_attr_done.insert({fn, dev});
    return VQC_OK;
}

// mode 2: the backward with the forward sweep and E inside (vqc_forward_backward)
const void* kernel_ptr(int dtype, bool dfloat, int mode, int K, bool full, bool ph2) {
    // complex64 sweeps of plans without CRZ / RZZ: the instantiations without
    // the phase cases (fewer spills)
    if (!dfloat && dtype == VQC_C64 && !ph2)
        return mode == 0 ? sweep_ptr_f32_fwd_nph(K, full)
             : mode == 1 ? sweep_ptr_f32_bwd_nph(K, full) : sweep_ptr_f32_fused_nph(K, full);
    if (dfloat)
        return mode == 2 ? sweep_ptr_dd_fused(K, full) : mode == 0 ? sweep_ptr_dd_fwd(K, full) : sweep_ptr_dd_bwd(K, full);
    if (mode == 2) return dtype == VQC_C64 ? sweep_ptr_f32_fused(K, full) : sweep_ptr_f64_fused(K, full);
    if (full) {
        if (dtype == VQC_C64) return mode == 0 ? sweep_ptr_f32_fwd(K) : sweep_ptr_f32_bwd(K);
        return mode == 0 ? sweep_ptr_f64_fwd(K) : sweep_ptr_f64_bwd(K);
    }
    if (dtype == VQC_C64) return mode == 0 ? sweep_ptr_f32_fwd_small(K) : sweep_ptr_f32_bwd_small(K);
    return mode == 0 ? sweep_ptr_f64_fwd_small(K) : sweep_ptr_f64_bwd_small(K);
}

size_t align16(size_t v) { return (v + 15) & ~size_t(15); }
size_t align256(size_t v) { return (v + 255) & ~size_t(255); }

// Launch geometry of one call.
struct Launch {
    const Schedule* s = nullptr;
    int K = 0, T = 0, S = 0, block = 0, grid = 0, nunits = 0, wg = 1, bpt = 1;
    size_t smem = 0;
    int sm_sh = 0, sm_ps = 0, sm_psi = 0, sm_lam = 0, sm_acc = 0, sm_terms = 0, sm_dw = 0,
        sm_red = 0, sm_plan = 0, sm_w = 0, sm_xg = 0;
    int cl = 0, sm_ecl = 0;   // cluster path: log2 CTAs per sample, <Z> gather area
    bool plan_smem = false;
    const void* fn = nullptr;
};

int env_int(const char* name, int dflt) {
    const char* v = std::getenv(name);
    return v && *v ? std::atoi(v) : dflt;
}

// Launch with programmatic stream serialisation: the kernel may be scheduled
// while the previous kernel in the stream finishes, and waits for it (every
// kernel calls grid_dep_wait() before touching caller memory), which hides most
// of the launch gap between the back-to-back kernels of one call and between
// consecutive calls.  VQC_PDL=0 turns it off (plain stream order).
cudaError_t launch(const void* fn, dim3 grid, dim3 block, void** args, size_t smem,
                   cudaStream_t stream) {
    static const bool pdl = env_int("VQC_PDL", 1) != 0;
    if (!pdl) return cudaLaunchKernel(fn, grid, block, args, smem, stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelExC(&cfg, fn, args);
}

int cta_threads() {
    const int t = env_int("VQC_CTA_THREADS", 128);
    return t >= 32 && t <= 512 ? t : 128;
}

// Pick the register-block size: the largest K that still gives the batch
// enough threads to cover every SM's schedulers (SMs x 4 warps), but not below
// 3 (a block of 8 amplitudes) where the circuit allows it.  A forced-K sweep on
// GB300 (8-qubit batch 1024 and 8192, 12-qubit batch 4096; forward, backward
// and the fused call) found no smaller K faster than this choice: smaller
// blocks add stages (shared-memory round trips and barriers) faster than the
// extra warps hide latency.
int choose_k(const HostPlan& p, int mode, int B, int sms) {
    int forced = env_int(mode == 0 ? "VQC_FORCE_K_FWD" : "VQC_FORCE_K_BWD", 0);
    if (forced > 0 && find_schedule(p, mode, forced)) return forced;
    int kmax = 0;
    for (const auto& s : p.scheds)
        if (s.mode == mode && s.path == VQC_PATH_RESIDENT) kmax = std::max(kmax, s.K);
    if (kmax == 0) return 0;
    const int kmin = std::min(kmax, 3);
    const double want = (double)sms * 4 * 32;
    int K = kmax;
    while (K > kmin && (double)B * std::ldexp(1.0, p.n - K) < want && find_schedule(p, mode, K - 1))
        --K;
    return K;
}

vqc_status plan_launch_uncached(const HostPlan& p, int launch_mode, int B, Launch& L) {
    // mode 2 (fused) has the backward's schedule and layout, its own kernel
    const int mode = launch_mode == 2 ? 1 : launch_mode;
    int dev = 0;
    VQC_CUDA(cudaGetDevice(&dev));
    DevInfo di;
    vqc_status st = device_info(dev, di);
    if (st != VQC_OK) return st;
    L.K = choose_k(p, mode, B, di.sms);
    L.s = L.K ? find_schedule(p, mode, L.K) : nullptr;
    if (!L.s)
        return fail(VQC_ERR_UNSUPPORTED, "no resident schedule for this circuit (n = " +
                                             std::to_string(p.n) + ")");
    const bool dbl = p.dtype == VQC_C128;
    const size_t rs = dbl ? 8 : 4, cs = 2 * rs;
    // A sample needs 2^(n-K) register blocks; a group of at most 256 threads
    // holds them, bpt blocks per thread.
    L.T = std::min(1 << (p.n - L.K), sweep_max_threads(dbl, mode, L.K));
    L.bpt = (1 << (p.n - L.K)) / L.T;
    L.wg = L.T > 32 ? L.T / 32 : 1;
    // Shared memory: a fixed part per CTA and a part per resident sample.
    const size_t dim = (size_t)1 << p.n;
    const size_t ew = dbl ? 8 : 32;   // reals per table entry
    const size_t fixed = align16((size_t)p.n_sh * ew * rs) + align16(mode == 1 ? (size_t)p.num_w * rs : 0) +
                         align16((size_t)p.num_w * rs) + 10 * 16;
    const size_t per_sample = (size_t)p.n_ps * ew * rs + dim * cs * (mode == 1 ? 2 : 1) +
                              (size_t)(p.num_x + p.n) * rs +
                              (mode == 1 ? p.accs.size() * L.wg * 8 * rs + p.term_src.size() * rs : 0) +
                              (size_t)L.wg * p.n * rs;
    // samples per CTA: groups up to VQC_CTA_THREADS (default 128) threads
    int S = std::max(1, cta_threads() / L.T);
    if ((size_t)di.smem_optin > fixed) {
        size_t fit = ((size_t)di.smem_optin - fixed) / per_sample;
        S = (int)std::min<size_t>((size_t)S, fit);
    } else {
        S = 0;
    }
    if (S < 1)
        return fail(VQC_ERR_UNSUPPORTED,
                    "state does not fit in shared memory on the resident path (" +
                        std::to_string(fixed + per_sample) + " > " +
                        std::to_string(di.smem_optin) + " bytes)");
    // Groups smaller than a warp fill whole warps when the CTA spans more than one.
    if (L.T < 32 && S * L.T > 32) S -= S % (32 / L.T);
    L.S = S;
    L.block = L.S * L.T;
    if (L.block > sweep_max_threads(dbl, mode, L.K))
        return fail(VQC_ERR_UNSUPPORTED, "thread group too large for this kernel");
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t o = off;
        off = align16(off + bytes);
        return (int)o;
    };
    L.sm_sh = take((size_t)p.n_sh * ew * rs);
    L.sm_ps = take((size_t)L.S * p.n_ps * ew * rs);
    L.sm_psi = take((size_t)L.S * dim * cs);
    L.sm_lam = take(mode == 1 ? (size_t)L.S * dim * cs : 0);
    L.sm_acc = take(mode == 1 ? (size_t)L.S * p.accs.size() * L.wg * 8 * rs : 0);
    L.sm_terms = take(mode == 1 ? (size_t)L.S * p.term_src.size() * rs : 0);
    L.sm_dw = take(mode == 1 ? (size_t)p.num_w * rs : 0);
    L.sm_red = take((size_t)L.S * L.wg * p.n * rs);   // <Z> partials (forward, or recompute with E)
    L.sm_w = take((size_t)p.num_w * rs);
    L.sm_xg = take((size_t)L.S * (p.num_x + p.n) * rs);
    // the plan's table data and this schedule go to shared memory when they fit
    const size_t plan_bytes = align16(p.dev_tab_end - p.dev_tab_begin) +
                              (L.s->dev_region_end - L.s->dev_region_begin);
    L.plan_smem = off + plan_bytes <= (size_t)di.smem_optin && env_int("VQC_PLAN_IN_SMEM", 1) != 0;
    L.sm_plan = L.plan_smem ? take(plan_bytes) : 0;
    L.smem = off;
    if (L.smem > (size_t)di.smem_optin)
        return fail(VQC_ERR_UNSUPPORTED, "shared-memory layout exceeds the per-CTA limit");
    L.fn = kernel_ptr(p.dtype, p.dfloat, launch_mode, L.K, L.T >= 32, p.has_ph2);
    if (!L.fn) return fail(VQC_ERR_UNSUPPORTED, "kernel not instantiated for this K");
    st = allow_max_smem(L.fn, dev, di.smem_optin);
    if (st != VQC_OK) return st;
    int per_sm = 0;
    VQC_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, L.fn, L.block, L.smem));
    if (per_sm < 1) return fail(VQC_ERR_UNSUPPORTED, "kernel cannot be resident with this geometry");
    L.nunits = (B + L.S - 1) / L.S;
    L.grid = std::max(1, std::min(L.nunits, per_sm * di.sms));
    return VQC_OK;
}

std::mutex g_geo_mu;
std::map<GeoKey, Launch> g_launch_cache;
std::map<GeoKey, Launch> g_cluster_cache;   // cluster-path geometry (forget_plan clears it too)

GeoKey geo_key(const HostPlan& p, int mode, int B, int hbm) {
    int dev = -1;
    cudaGetDevice(&dev);
    // environment switches that change the geometry are part of the key
    const int env = env_int("VQC_FORCE_K_FWD", 0) * 1000 + env_int("VQC_FORCE_K_BWD", 0) * 10 +
                    (env_int("VQC_PLAN_IN_SMEM", 1) != 0 ? 1 : 0) + cta_threads() * 1000000;
    return GeoKey{&p, mode, B, dev, hbm * 100000 + env};
}

vqc_status plan_launch(const HostPlan& p, int mode, int B, Launch& L) {
    const GeoKey k = geo_key(p, mode, B, 0);
    {
        std::lock_guard<std::mutex> lk(g_geo_mu);
        auto it = g_launch_cache.find(k);
        if (it != g_launch_cache.end()) {
            L = it->second;
            return VQC_OK;
        }
    }
    vqc_status st = plan_launch_uncached(p, mode, B, L);
    if (st == VQC_OK) {
        std::lock_guard<std::mutex> lk(g_geo_mu);
        g_launch_cache[k] = L;
    }
    return st;
}

template <typename R>
void fill_plan_args(const HostPlan& p, const Launch& L, KArgs<R>& a) {
    const char* base = static_cast<const char*>(p.dbuf);
    a.ops = reinterpret_cast<const DOp*>(base + L.s->dev_ops);
    a.stages = reinterpret_cast<const DStage*>(base + L.s->dev_stages);
    a.nstages = (int)L.s->stages.size();
    a.entries = reinterpret_cast<const DEntry*>(base + p.dev_entries);
    a.ps_list = reinterpret_cast<const int32_t*>(base + p.dev_ps_list);
    a.sh_list = reinterpret_cast<const int32_t*>(base + p.dev_sh_list);
    a.consts = reinterpret_cast<const DConst*>(base + p.dev_consts);
    a.cmat = reinterpret_cast<const R*>(base + p.dev_cmat);
    a.cang = reinterpret_cast<const R*>(base + p.dev_cang);
    a.accs = reinterpret_cast<const DAcc*>(base + p.dev_accs);
    a.xocc_ptr = reinterpret_cast<const int32_t*>(base + p.dev_xocc_ptr);
    a.xocc = reinterpret_cast<const int32_t*>(base + p.dev_xocc);
    a.wocc_ptr = reinterpret_cast<const int32_t*>(base + p.dev_wocc_ptr);
    a.wocc = reinterpret_cast<const int32_t*>(base + p.dev_wocc);
    a.err = p.dev_error;
    a.n = p.n;
    a.K = L.K;
    a.tbits = p.n - L.K;
    a.G = p.G_swz;
    a.S = L.S;
    a.tpg = L.T;
    a.bpt = L.bpt;
    a.n_ps = p.n_ps;
    a.n_sh = p.n_sh;
    a.n_accs = (int)p.accs.size();
    a.n_ps = p.n_ps;
    a.n_terms = (int)p.term_src.size();
    a.Px = p.num_x;
    a.Pw = p.num_w;
    a.sm_sh = L.sm_sh; a.sm_ps = L.sm_ps; a.sm_psi = L.sm_psi; a.sm_lam = L.sm_lam;
    a.sm_acc = L.sm_acc; a.sm_terms = L.sm_terms; a.sm_dw = L.sm_dw; a.sm_red = L.sm_red;
    a.sm_w = L.sm_w; a.sm_xg = L.sm_xg;
    a.plan = static_cast<const unsigned char*>(p.dbuf);
    a.tab_off = (int)p.dev_tab_begin;
    a.tab_bytes = (int)(p.dev_tab_end - p.dev_tab_begin);
    a.sched_off = (int)L.s->dev_region_begin;
    a.sched_bytes = (int)(L.s->dev_region_end - L.s->dev_region_begin);
    a.sm_plan = L.sm_plan;
    a.plan_smem = L.plan_smem ? 1 : 0;
    a.cl = L.cl;
    a.sm_ecl = L.sm_ecl;
}

// Device buffer layout of a plan (all sections 16-byte aligned).
// Uploaded plans (their device error words are read by vqc_sync_check).
std::mutex g_plans_mu;
std::set<const HostPlan*> g_plans;

vqc_status upload(HostPlan& p) {
    const bool dbl = p.dtype == VQC_C128;
    std::vector<uint8_t> blob;
    auto put = [&](const void* src, size_t bytes) {
        size_t off = blob.size();
        blob.resize(align16(off + bytes), 0);
        if (bytes && src) std::memcpy(blob.data() + off, src, bytes);
        return off;
    };
    std::vector<int32_t> ps_list, sh_list;
    for (size_t i = 0; i < p.entries.size(); ++i)
        (p.entries[i].per_sample ? ps_list : sh_list).push_back((int32_t)i);
    // the kernels index lists by slot order, which is entry order within each list
    std::vector<double> cm_d = p.cmat, ca_d = p.cang;
    std::vector<float> cm_f(cm_d.begin(), cm_d.end()), ca_f(ca_d.begin(), ca_d.end());
    if (p.dfloat) {
        // double-float kernels read constants as (hi, lo) float pairs in the 8
        // bytes a double takes: hi = the double rounded to float, lo = the rest
        auto split = [](std::vector<double>& v) {
            for (double& d : v) {
                const float hi = (float)d, lo = (float)(d - (double)hi);
                std::memcpy(reinterpret_cast<char*>(&d), &hi, 4);
                std::memcpy(reinterpret_cast<char*>(&d) + 4, &lo, 4);
            }
        };
        split(cm_d);
        split(ca_d);
    }
    p.dev_entries = put(p.entries.data(), p.entries.size() * sizeof(DEntry));
    p.dev_ps_list = put(ps_list.data(), ps_list.size() * 4);
    p.dev_sh_list = put(sh_list.data(), sh_list.size() * 4);
    p.dev_consts = put(p.consts.data(), p.consts.size() * sizeof(DConst));
    p.dev_cmat = dbl ? put(cm_d.data(), cm_d.size() * 8) : put(cm_f.data(), cm_f.size() * 4);
    p.dev_cang = dbl ? put(ca_d.data(), ca_d.size() * 8) : put(ca_f.data(), ca_f.size() * 4);
    p.dev_accs = put(p.accs.data(), p.accs.size() * sizeof(DAcc));
    p.dev_xocc_ptr = put(p.xocc_ptr.data(), p.xocc_ptr.size() * 4);
    p.dev_xocc = put(p.xocc.data(), p.xocc.size() * 4);
    p.dev_wocc_ptr = put(p.wocc_ptr.data(), p.wocc_ptr.size() * 4);
    p.dev_wocc = put(p.wocc.data(), p.wocc.size() * 4);
    p.dev_tab_begin = p.dev_entries;
    p.dev_tab_end = blob.size();
    for (auto& s : p.scheds) {
        s.dev_region_begin = blob.size();
        s.dev_ops = put(s.ops.data(), s.ops.size() * sizeof(DOp));
        s.dev_stages = put(s.stages.data(), s.stages.size() * sizeof(DStage));
        s.dev_passes = put(s.passes.data(), s.passes.size() * sizeof(DPass));
        s.dev_pass_entries = put(s.pass_entries.data(), s.pass_entries.size() * 4);
        s.dev_pass_accs = put(s.pass_accs.data(), s.pass_accs.size() * 4);
        s.dev_region_end = blob.size();
    }
    size_t err_off = put(nullptr, 16);
    blob.resize(align256(blob.size()), 0);
    VQC_CUDA(cudaGetDevice(&p.device));
    void* d = nullptr;
    cudaError_t e = cudaMalloc(&d, blob.size());
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return fail(VQC_ERR_OUT_OF_MEMORY, "cudaMalloc of the plan failed");
    }
    e = cudaMemcpy(d, blob.data(), blob.size(), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
        cudaFree(d);
        return cuda_fail(e, "cudaMemcpy(plan)");
    }
    p.dbuf = d;
    p.dbytes = blob.size();
    p.dev_error = reinterpret_cast<unsigned*>(static_cast<char*>(d) + err_off);
    std::lock_guard<std::mutex> lk(g_plans_mu);
    g_plans.insert(&p);
    return VQC_OK;
}

// Workspace of a backward call: [0, 256) control block (counter), then the
// per-CTA dw partials [grid, num_w].
size_t bwd_workspace(const HostPlan& p, const Launch& L) {
    const size_t rs = p.dtype == VQC_C128 ? 8 : 4;
    return 256 + align256((size_t)L.grid * std::max(p.num_w, 1) * rs);
}

bool misaligned(const void* ptr, size_t a) {
    return (reinterpret_cast<uintptr_t>(ptr) & (a - 1)) != 0;
}

template <typename R>
vqc_status run(const HostPlan& p, int mode, int B, const void* x, const void* w, const void* psi0,
               const void* psi_final, const void* gE, void* E, void* state_out, void* dx, void* dw,
               void* ws, size_t ws_bytes, cudaStream_t stream) {
    using C = C2<R>;
    Launch L;
    vqc_status st = plan_launch(p, mode, B, L);
    if (st != VQC_OK) return st;
    KArgs<R> a{};
    fill_plan_args<R>(p, L, a);
    a.B = B;
    a.nunits = L.nunits;
    a.x = static_cast<const R*>(x);
    a.w = static_cast<const R*>(w);
    a.psi0 = static_cast<const C*>(psi0);
    a.psi_final = static_cast<const C*>(psi_final);
    a.gE = static_cast<const R*>(gE);
    a.E = static_cast<R*>(E);
    a.state_out = static_cast<C*>(state_out);
    a.dx = static_cast<R*>(dx);
    a.dw = static_cast<R*>(dw);
    if (mode >= 1) {
        size_t need = bwd_workspace(p, L);
        if (!ws || ws_bytes < need || misaligned(ws, 256))
            return fail(VQC_ERR_WORKSPACE, "backward workspace must be >= " + std::to_string(need) +
                                               " bytes and 256-byte aligned");
        a.counter = static_cast<unsigned*>(ws);
        a.dw_part = reinterpret_cast<R*>(static_cast<char*>(ws) + 256);
    }
    void* args[] = {&a};
    VQC_CUDA(launch(L.fn, dim3(L.grid), dim3(L.block), args, L.smem, stream));
    if (mode >= 1 && dw && p.num_w > 0) {
        const R* part = a.dw_part;
        int rows = L.grid, cols = p.num_w;
        R* out = static_cast<R*>(dw);
        void* rargs[] = {&part, &rows, &cols, &out};
        VQC_CUDA(launch(reduce_cols_ptr(p.dtype == VQC_C128), dim3(cols), dim3(256), rargs,
                                  0, stream));
    }
    return VQC_OK;
}


// ---------------------------------------------------------------- cluster path

vqc_status plan_cluster(const HostPlan& p, int mode, int B, Launch& L) {
    const GeoKey k = geo_key(p, mode, B, 2);
    {
        std::lock_guard<std::mutex> lk(g_geo_mu);
        auto it = g_cluster_cache.find(k);
        if (it != g_cluster_cache.end()) {
            L = it->second;
            return VQC_OK;
        }
    }
    L = Launch();
    L.s = find_cluster_schedule(p, mode);
    if (!L.s) return fail(VQC_ERR_UNSUPPORTED, "no cluster schedule for this circuit");
    int dev = 0;
    VQC_CUDA(cudaGetDevice(&dev));
    DevInfo di;
    vqc_status st = device_info(dev, di);
    if (st != VQC_OK) return st;
    const bool dbl = p.dtype == VQC_C128;
    const size_t rs = dbl ? 8 : 4, cs = 2 * rs, ew = dbl ? 8 : 32;
    L.K = L.s->K;
    L.cl = p.n - L.K - L.s->cta_bits;
    L.T = 1 << (p.n - L.K);           // threads of a sample group, over the whole cluster
    L.block = L.T >> L.cl;            // 2^cta_bits: 256 or 512
    L.S = 1;
    L.bpt = 1;
    L.wg = L.block / 32;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t o = off;
        off = align16(off + bytes);
        return (int)o;
    };
    const size_t slice = ((size_t)1 << (p.n - L.cl)) * cs;
    L.sm_sh = take((size_t)p.n_sh * ew * rs);
    L.sm_ps = take((size_t)p.n_ps * ew * rs);
    L.sm_psi = take(slice);
    if (mode == 0) {
        L.sm_red = take((size_t)L.wg * p.n * rs);
        L.sm_ecl = take(((size_t)1 << L.cl) * p.n * rs);
        L.sm_w = take((size_t)p.num_w * rs);
        L.sm_xg = take((size_t)p.num_x * rs);
    } else {   // lam, rho partials [accs][warps][4], terms, dw partial, x and gE rows
        L.sm_lam = take(slice);
        L.sm_acc = take(std::max<size_t>(p.accs.size(), 1) * L.wg * 4 * rs);
        L.sm_terms = take(std::max<size_t>(p.term_src.size(), 1) * rs);
        L.sm_dw = take((size_t)std::max(p.num_w, 1) * rs);
        L.sm_w = take((size_t)std::max(p.num_w, 1) * rs);
        L.sm_xg = take((size_t)(p.num_x + p.n) * rs);
    }
    const size_t plan_bytes = align16(p.dev_tab_end - p.dev_tab_begin) +
                              (L.s->dev_region_end - L.s->dev_region_begin);
    L.plan_smem = off + plan_bytes <= (size_t)di.smem_optin && env_int("VQC_PLAN_IN_SMEM", 1) != 0;
    L.sm_plan = L.plan_smem ? take(plan_bytes) : 0;
    L.smem = off;
    if (L.smem > (size_t)di.smem_optin)
        return fail(VQC_ERR_UNSUPPORTED, "cluster slice does not fit in shared memory");
    L.fn = mode == 0 ? (p.dfloat ? cluster_ptr_dd() : cluster_ptr(dbl)) : cluster_bwd_ptr(dbl, p.dfloat);
    st = allow_max_smem(L.fn, dev, di.smem_optin);
    if (st != VQC_OK) return st;
    cudaLaunchConfig_t cfg{};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1u << L.cl;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(1u << L.cl);
    cfg.blockDim = dim3(L.block);
    cfg.dynamicSmemBytes = L.smem;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int nclusters = 0;
    VQC_CUDA(cudaOccupancyMaxActiveClusters(&nclusters, L.fn, &cfg));
    if (nclusters < 1) return fail(VQC_ERR_UNSUPPORTED, "cluster kernel cannot be resident");
    L.nunits = B;
    L.grid = std::min(B, nclusters) << L.cl;
    std::lock_guard<std::mutex> lk(g_geo_mu);
    g_cluster_cache[k] = L;
    return VQC_OK;
}

// The cluster forward by default for 2-CTA clusters (complex64 15 qubits,
// complex128 14): measured 16-24% / ~5% faster than the HBM-tiled passes there.
// Larger clusters measured slower (0.7x at 16 qubits: one sample per cluster
// leaves too few warps per SM to hide the per-stage cluster barriers), so they
// run only when VQC_FORCE_PATH=cluster asks; VQC_FORCE_PATH=hbm turns it off.
// The cluster backward (psi and lam over the cluster) follows the same rule:
// by default for 2-CTA clusters (complex64 14 qubits, complex128 13), where it
// measured 1-7% faster than the backward passes, and 0.78-0.90x with 4-8 CTAs
// (0.80x on the 16-qubit / batch-512 workload); it also needs its shared-memory
// layout (two slices, the per-warp rho partials, the tables) to fit one CTA.
bool use_cluster(const HostPlan& p, int mode) {
    const Schedule* s = find_cluster_schedule(p, mode);
    if (!s) return false;
    const char* f = std::getenv("VQC_FORCE_PATH");
    const bool forced = f && std::string(f) == "cluster";
    if (f && std::string(f) == "hbm") return false;
    const bool two_cta = p.n - s->K - s->cta_bits == 1;
    if (mode == 0) return forced || two_cta;
    if (!forced && !two_cta) return false;
    Launch L;
    const std::string saved = g_err;
    const bool ok = plan_cluster(p, 1, 1, L) == VQC_OK;
    g_err = saved;
    return ok;
}

template <typename R>
vqc_status run_cluster_forward(const HostPlan& p, int B, const void* x, const void* w,
                               const void* psi0, void* E, void* state_out, cudaStream_t stream) {
    using C = C2<R>;
    Launch L;
    vqc_status st = plan_cluster(p, 0, B, L);
    if (st != VQC_OK) return st;
    KArgs<R> a{};
    fill_plan_args<R>(p, L, a);
    a.B = B;
    a.nunits = B;
    a.x = static_cast<const R*>(x);
    a.w = static_cast<const R*>(w);
    a.psi0 = static_cast<const C*>(psi0);
    a.E = static_cast<R*>(E);
    a.state_out = static_cast<C*>(state_out);
    void* args[] = {&a};
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1u << L.cl;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(L.grid);
    cfg.blockDim = dim3(L.block);
    cfg.dynamicSmemBytes = L.smem;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = env_int("VQC_PDL", 1) != 0 ? 2 : 1;
    VQC_CUDA(cudaLaunchKernelExC(&cfg, L.fn, args));
    return VQC_OK;
}

// Workspace of a cluster backward: [0, 256) control block, then the per-cluster
// dw partials [clusters, num_w].
size_t cluster_bwd_workspace(const HostPlan& p, const Launch& L) {
    const size_t rs = p.dtype == VQC_C128 ? 8 : 4;
    return 256 + align256((size_t)(L.grid >> L.cl) * std::max(p.num_w, 1) * rs);
}

template <typename R>
vqc_status run_cluster_backward(const HostPlan& p, int B, const void* x, const void* w,
                                const void* psi0, const void* psi_final, const void* gE, void* dx,
                                void* dw, void* ws, size_t ws_bytes, cudaStream_t stream) {
    using C = C2<R>;
    Launch L;
    vqc_status st = plan_cluster(p, 1, B, L);
    if (st != VQC_OK) return st;
    const size_t need = cluster_bwd_workspace(p, L);
    if (!ws || ws_bytes < need || misaligned(ws, 256))
        return fail(VQC_ERR_WORKSPACE, "backward workspace must be >= " + std::to_string(need) +
                                           " bytes and 256-byte aligned");
    KArgs<R> a{};
    fill_plan_args<R>(p, L, a);
    a.B = B;
    a.nunits = B;
    a.x = static_cast<const R*>(x);
    a.w = static_cast<const R*>(w);
    a.psi0 = static_cast<const C*>(psi0);
    a.psi_final = static_cast<const C*>(psi_final);
    a.gE = static_cast<const R*>(gE);
    a.dx = static_cast<R*>(dx);
    a.dw = static_cast<R*>(dw);
    a.counter = static_cast<unsigned*>(ws);
    a.dw_part = reinterpret_cast<R*>(static_cast<char*>(ws) + 256);
    void* args[] = {&a};
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1u << L.cl;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(L.grid);
    cfg.blockDim = dim3(L.block);
    cfg.dynamicSmemBytes = L.smem;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = env_int("VQC_PDL", 1) != 0 ? 2 : 1;
    VQC_CUDA(cudaLaunchKernelExC(&cfg, L.fn, args));
    if (dw && p.num_w > 0) {
        const R* part = a.dw_part;
        int rows = L.grid >> L.cl, cols = p.num_w;
        R* out = static_cast<R*>(dw);
        void* rargs[] = {&part, &rows, &cols, &out};
        VQC_CUDA(launch(reduce_cols_ptr(p.dtype == VQC_C128), dim3(cols), dim3(256), rargs, 0, stream));
    }
    return VQC_OK;
}

// ---------------------------------------------------------------- HBM path
struct PassGeo {
    const Schedule* s = nullptr;
    int K = 0, T = 0, S = 0, block = 0, grid = 0, wg = 1, ntiles = 1;
    long long nunits = 0;
    size_t smem = 0;
    int sm_sh = 0, sm_ps = 0, sm_psi = 0, sm_lam = 0, sm_acc = 0, sm_red = 0, sm_plan = 0,
        sm_koff = 0;
    bool plan_smem = false;
    const void* fn = nullptr;
};

vqc_status plan_hbm_uncached(const HostPlan& p, int mode, int B, PassGeo& L) {
    L.s = find_hbm_schedule(p, mode);
    if (!L.s) return fail(VQC_ERR_UNSUPPORTED, "no HBM-tiled schedule for this circuit");
    int dev = 0;
    VQC_CUDA(cudaGetDevice(&dev));
    DevInfo di;
    vqc_status st = device_info(dev, di);
    if (st != VQC_OK) return st;
    const bool dbl = p.dtype == VQC_C128;
    const size_t rs = dbl ? 8 : 4, cs = 2 * rs;
    const int m = L.s->m;
    L.K = L.s->K;
    L.T = 1 << (m - L.K);
    L.wg = L.T > 32 ? L.T / 32 : 1;
    L.ntiles = 1 << (p.n - m);
    int ps_max = 0, sh_max = 0, acc_max = 0;
    for (const DPass& ps : L.s->passes) {
        ps_max = std::max(ps_max, ps.ps_count);
        sh_max = std::max(sh_max, ps.sh_count);
        acc_max = std::max(acc_max, ps.acc_count);
    }
    const size_t tdim = (size_t)1 << m;
    const size_t ew = dbl ? 8 : 32;   // reals per table entry
    const size_t fixed = align16((size_t)sh_max * ew * rs) + 8 * 16 + 1024;   // + tile-copy offsets
    const size_t per_tile = (size_t)ps_max * ew * rs + tdim * cs * (mode == 1 ? 2 : 1) +
                            (mode == 1 ? (size_t)acc_max * L.wg * 8 * rs : (size_t)L.wg * p.n * rs);
    int S = std::max(1, 128 / L.T);
    if ((size_t)di.smem_optin <= fixed + per_tile)
        S = (size_t)di.smem_optin >= fixed + per_tile ? 1 : 0;
    else
        S = (int)std::min<size_t>((size_t)S, ((size_t)di.smem_optin - fixed) / per_tile);
    if (S < 1) return fail(VQC_ERR_UNSUPPORTED, "HBM tile does not fit in shared memory");
    if (L.T < 32 && S * L.T > 32) S -= S % (32 / L.T);
    L.S = S;
    L.block = S * L.T;
    if (L.block > 512) return fail(VQC_ERR_UNSUPPORTED, "HBM tile group too large");
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t o = off;
        off = align16(off + bytes);
        return (int)o;
    };
    L.sm_sh = take((size_t)sh_max * ew * rs);
    L.sm_ps = take((size_t)S * ps_max * ew * rs);
    L.sm_psi = take((size_t)S * tdim * cs);
    L.sm_lam = take(mode == 1 ? (size_t)S * tdim * cs : 0);
    L.sm_acc = take(mode == 1 ? (size_t)S * acc_max * L.wg * 8 * rs : 0);
    L.sm_red = take(mode == 0 ? (size_t)S * L.wg * p.n * rs : 0);
    {   // tile-copy offsets: one uint2 per vector round of a tile
        const size_t apv = 16 / cs, nvec = tdim / apv;
        L.sm_koff = take(((nvec + L.T - 1) / L.T) * 8);
    }
    const size_t plan_bytes = align16(p.dev_tab_end - p.dev_tab_begin) +
                              (L.s->dev_region_end - L.s->dev_region_begin);
    L.plan_smem = off + plan_bytes <= (size_t)di.smem_optin && plan_bytes <= 48 * 1024;
    L.sm_plan = L.plan_smem ? take(plan_bytes) : 0;
    L.smem = off;
    L.fn = p.dfloat ? pass_ptr_dd(mode, L.K, L.T >= 32)
           : (!dbl && mode == 0 && !p.has_ph2) ? pass_ptr_f32_fwd_nph(L.K, L.T >= 32)   // no phase cases
                                               : pass_ptr(dbl, mode, L.K, L.T >= 32);
    if (!L.fn) return fail(VQC_ERR_UNSUPPORTED, "pass kernel not instantiated for this K");
    st = allow_max_smem(L.fn, dev, di.smem_optin);
    if (st != VQC_OK) return st;
    int per_sm = 0;
    VQC_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, L.fn, L.block, L.smem));
    if (per_sm < 1) return fail(VQC_ERR_UNSUPPORTED, "pass kernel cannot be resident");
    L.nunits = ((long long)B * L.ntiles + S - 1) / S;
    L.grid = (int)std::max<long long>(1, std::min<long long>(L.nunits, (long long)per_sm * di.sms));
    return VQC_OK;
}

std::map<GeoKey, PassGeo> g_pass_cache;

vqc_status plan_hbm(const HostPlan& p, int mode, int B, PassGeo& L) {
    const GeoKey k = geo_key(p, mode, B, 1);
    {
        std::lock_guard<std::mutex> lk(g_geo_mu);
        auto it = g_pass_cache.find(k);
        if (it != g_pass_cache.end()) {
            L = it->second;
            return VQC_OK;
        }
    }
    vqc_status st = plan_hbm_uncached(p, mode, B, L);
    if (st == VQC_OK) {
        std::lock_guard<std::mutex> lk(g_geo_mu);
        g_pass_cache[k] = L;
    }
    return st;
}

void forget_plan(const HostPlan* p) {
    std::lock_guard<std::mutex> lk(g_geo_mu);
    for (auto it = g_launch_cache.begin(); it != g_launch_cache.end();)
        it = it->first.plan == p ? g_launch_cache.erase(it) : std::next(it);
    for (auto it = g_pass_cache.begin(); it != g_pass_cache.end();)
        it = it->first.plan == p ? g_pass_cache.erase(it) : std::next(it);
    for (auto it = g_cluster_cache.begin(); it != g_cluster_cache.end();)
        it = it->first.plan == p ? g_cluster_cache.erase(it) : std::next(it);
}

// Workspace of the HBM path.  Forward: [control | working state | <Z> partials].
// Backward: [control | psi | lam | gradient-term partials].
struct HbmWs {
    size_t state = 0, lam = 0, part = 0, terms = 0, ps = 0, total = 0;
};

HbmWs hbm_layout(const HostPlan& p, int mode, int B, int ntiles) {
    const size_t rs = p.dtype == VQC_C128 ? 8 : 4, cs = 2 * rs;
    const size_t sbytes = align256((size_t)B * ((size_t)1 << p.n) * cs);
    HbmWs w;
    w.state = 256;
    if (mode == 0) {
        w.part = w.state + sbytes;
        w.ps = w.part + align256((size_t)B * ntiles * p.n * rs);
    } else {   // per-tile rho sums [B * ntiles][accs][4], then the per-sample terms [B][terms]
        w.lam = w.state + sbytes;
        w.part = w.lam + sbytes;
        w.terms = w.part + align256((size_t)B * ntiles * std::max<size_t>(p.accs.size(), 1) * 4 * rs);
        w.ps = w.terms + align256((size_t)B * std::max<size_t>(p.term_src.size(), 1) * rs);
    }
    // every sample's per-sample table entries [B][n_ps][entry words]
    w.total = w.ps + align256((size_t)B * p.n_ps * (p.dtype == VQC_C128 ? 8 : 32) * rs);
    return w;
}

// Every sample's per-sample table entries into `out` (ps_tables), read by the
// passes instead of evaluating them once per tile.
template <typename R>
vqc_status launch_ps_tables(const HostPlan& p, int B, const void* x, const void* w, void* out,
                            cudaStream_t stream) {
    if (p.n_ps == 0) return VQC_OK;
    const char* base = static_cast<const char*>(p.dbuf);
    const DEntry* entries = reinterpret_cast<const DEntry*>(base + p.dev_entries);
    const int32_t* ps_list = reinterpret_cast<const int32_t*>(base + p.dev_ps_list);
    const DConst* consts = reinterpret_cast<const DConst*>(base + p.dev_consts);
    const R* cang = reinterpret_cast<const R*>(base + p.dev_cang);
    const R* cmat = reinterpret_cast<const R*>(base + p.dev_cmat);
    const R* xr = static_cast<const R*>(x);
    const R* wr = static_cast<const R*>(w);
    int Px = p.num_x, Bi = B, nps = p.n_ps;
    void* args[] = {&entries, &ps_list, &consts, &cang, &cmat, &xr, &Px, &wr, &Bi, &nps, &out};
    const int blocks = (int)std::min<long long>(4096, ((long long)B * nps + 255) / 256);
    VQC_CUDA(launch(p.dfloat ? ps_tables_ptr_dd() : ps_tables_ptr(p.dtype == VQC_C128), dim3(std::max(blocks, 1)),
                    dim3(256), args, 0, stream));
    return VQC_OK;
}

template <typename R>
void fill_pass_args(const HostPlan& p, const PassGeo& L, const DPass& ps, PArgs<R>& a) {
    const char* base = static_cast<const char*>(p.dbuf);
    a.ops = reinterpret_cast<const DOp*>(base + L.s->dev_ops);
    a.stages = reinterpret_cast<const DStage*>(base + L.s->dev_stages);
    a.err = p.dev_error;
    a.pass_entries = reinterpret_cast<const int32_t*>(base + L.s->dev_pass_entries);
    a.pass_accs = reinterpret_cast<const int32_t*>(base + L.s->dev_pass_accs);
    a.entries = reinterpret_cast<const DEntry*>(base + p.dev_entries);
    a.consts = reinterpret_cast<const DConst*>(base + p.dev_consts);
    a.cmat = reinterpret_cast<const R*>(base + p.dev_cmat);
    a.cang = reinterpret_cast<const R*>(base + p.dev_cang);
    a.accs = reinterpret_cast<const DAcc*>(base + p.dev_accs);
    a.n = p.n;
    a.m = L.s->m;
    a.K = L.K;
    a.tbits = L.s->m - L.K;
    a.G = p.G_swz;
    a.S = L.S;
    a.nout = p.n - L.s->m;
    a.ntiles = L.ntiles;
    a.stage_begin = ps.stage_begin;
    a.stage_end = ps.stage_end;
    a.ps_begin = ps.ps_begin;
    a.ps_count = ps.ps_count;
    a.sh_begin = ps.sh_begin;
    a.sh_count = ps.sh_count;
    a.acc_begin = ps.acc_begin;
    a.acc_count = ps.acc_count;
    a.n_accs = (int)p.accs.size();
    a.n_ps = p.n_ps;
    a.Px = p.num_x;
    a.nunits = L.nunits;
    for (int i = 0; i < 24; ++i) {
        a.tile_q[i] = ps.tile_q[i];
        a.out_q[i] = ps.out_q[i];
    }
    a.sm_sh = L.sm_sh; a.sm_ps = L.sm_ps; a.sm_psi = L.sm_psi; a.sm_lam = L.sm_lam;
    a.sm_acc = L.sm_acc; a.sm_red = L.sm_red; a.sm_koff = L.sm_koff;
    a.plan = static_cast<const unsigned char*>(p.dbuf);
    a.tab_off = (int)p.dev_tab_begin;
    a.tab_bytes = (int)(p.dev_tab_end - p.dev_tab_begin);
    a.sched_off = (int)L.s->dev_region_begin;
    a.sched_bytes = (int)(L.s->dev_region_end - L.s->dev_region_begin);
    a.sm_plan = L.sm_plan;
    a.plan_smem = L.plan_smem ? 1 : 0;
}

template <typename R>
vqc_status run_hbm_forward(const HostPlan& p, int B, const void* x, const void* w,
                           const void* psi0, void* E, void* state_out, void* ws, size_t ws_bytes,
                           cudaStream_t stream, bool want_E) {
    using C = C2<R>;
    PassGeo L;
    vqc_status st = plan_hbm(p, 0, B, L);
    if (st != VQC_OK) return st;
    const HbmWs lay = hbm_layout(p, 0, B, L.ntiles);
    if (!ws || ws_bytes < lay.total || misaligned(ws, 256))
        return fail(VQC_ERR_WORKSPACE, "forward workspace must be >= " + std::to_string(lay.total) +
                                           " bytes and 256-byte aligned");
    char* wsc = static_cast<char*>(ws);
    C* W = state_out ? static_cast<C*>(state_out) : reinterpret_cast<C*>(wsc + lay.state);
    R* E_part = reinterpret_cast<R*>(wsc + lay.part);
    void* ps_g = wsc + lay.ps;
    st = launch_ps_tables<R>(p, B, x, w, ps_g, stream);
    if (st != VQC_OK) return st;
    const int np = (int)L.s->passes.size();
    for (int i = 0; i < np; ++i) {
        PArgs<R> a{};
        fill_pass_args<R>(p, L, L.s->passes[i], a);
        a.ps_g = ps_g;
        a.B = B;
        a.x = static_cast<const R*>(x);
        a.w = static_cast<const R*>(w);
        a.src_psi = i == 0 ? static_cast<const C*>(psi0) : W;
        const bool last = i == np - 1;
        a.dst_psi = (last && want_E && !state_out) ? nullptr : W;
        a.E_part = (last && want_E) ? E_part : nullptr;
        // double-float: raw pairs between passes, complex128 in and out (a
        // pass reads its whole tile before writing it, so W may change format
        // in place)
        a.src_raw = i > 0;
        a.dst_raw = !last;
        void* args[] = {&a};
        VQC_CUDA(launch(L.fn, dim3(L.grid), dim3(L.block), args, L.smem, stream));
    }
    if (want_E) {
        const R* Ep = E_part;
        R* Eo = static_cast<R*>(E);
        int Bi = B, nt = L.ntiles, n = p.n;
        void* args[] = {&Ep, &Bi, &nt, &n, &Eo};
        const int blocks = (int)std::min<long long>(4096, ((long long)B * n + 255) / 256);
        VQC_CUDA(launch(reduce_expz_ptr(p.dtype == VQC_C128), dim3(std::max(blocks, 1)),
                                  dim3(256), args, 0, stream));
    }
    return VQC_OK;
}

template <typename R>
vqc_status run_hbm_backward(const HostPlan& p, int B, const void* x, const void* w,
                            const void* psi0, const void* psi_final, const void* gE, void* dx,
                            void* dw, void* ws, size_t ws_bytes, cudaStream_t stream) {
    using C = C2<R>;
    PassGeo L;
    vqc_status st = plan_hbm(p, 1, B, L);
    if (st != VQC_OK) return st;
    const HbmWs lay = hbm_layout(p, 1, B, L.ntiles);
    size_t need = lay.total;
    if (!ws || ws_bytes < need || misaligned(ws, 256))
        return fail(VQC_ERR_WORKSPACE, "backward workspace must be >= " + std::to_string(need) +
                                           " bytes and 256-byte aligned");
    char* wsc = static_cast<char*>(ws);
    C* Psi = reinterpret_cast<C*>(wsc + lay.state);
    C* Lam = reinterpret_cast<C*>(wsc + lay.lam);
    R* rho = reinterpret_cast<R*>(wsc + lay.part);
    R* terms = reinterpret_cast<R*>(wsc + lay.terms);
    void* ps_g = wsc + lay.ps;
    if (p.dtype == VQC_C128 || !psi_final) {   // complex64 backward passes evaluate their own entries
        st = launch_ps_tables<R>(p, B, x, w, ps_g, stream);
        if (st != VQC_OK) return st;
    }
    const C* src0 = static_cast<const C*>(psi_final);
    if (!src0) {
        // recompute the final state into Psi (the forward passes need no <Z>)
        PassGeo Lf;
        st = plan_hbm(p, 0, B, Lf);
        if (st != VQC_OK) return st;
        const int npf = (int)Lf.s->passes.size();
        for (int i = 0; i < npf; ++i) {
            PArgs<R> a{};
            fill_pass_args<R>(p, Lf, Lf.s->passes[i], a);
            a.ps_g = ps_g;
            a.B = B;
            a.x = static_cast<const R*>(x);
            a.w = static_cast<const R*>(w);
            a.src_psi = i == 0 ? static_cast<const C*>(psi0) : Psi;
            a.dst_psi = Psi;
            a.src_raw = i > 0;
            a.dst_raw = 1;   // read only by the backward passes below
            void* args[] = {&a};
            VQC_CUDA(launch(Lf.fn, dim3(Lf.grid), dim3(Lf.block), args, Lf.smem, stream));
        }
        src0 = Psi;
    }
    const int np = (int)L.s->passes.size();
    for (int i = np - 1; i >= 0; --i) {
        PArgs<R> a{};
        fill_pass_args<R>(p, L, L.s->passes[i], a);
        a.ps_g = ps_g;
        a.B = B;
        a.x = static_cast<const R*>(x);
        a.w = static_cast<const R*>(w);
        a.gE = static_cast<const R*>(gE);
        const bool first = i == np - 1, last = i == 0;
        a.src_psi = first ? src0 : Psi;
        a.src_lam = first ? nullptr : Lam;
        a.dst_psi = last ? nullptr : Psi;
        a.dst_lam = last ? nullptr : Lam;
        a.src_raw = first ? psi_final == nullptr : 1;   // recomputed states are raw
        a.lam_raw = 1;
        a.dst_raw = 1;
        a.rho = rho;
        void* args[] = {&a};
        VQC_CUDA(launch(L.fn, dim3(L.grid), dim3(L.block), args, L.smem, stream));
    }
    const char* base = static_cast<const char*>(p.dbuf);
    const bool dbl = p.dtype == VQC_C128;
    int nt = (int)p.term_src.size();
    const bool want = (dx && p.num_x > 0) || (dw && p.num_w > 0);
    if (want && !p.accs.empty()) {   // per-sample gradient terms from the per-tile rho sums
        const R* r = rho;
        int Bi = B, ntl = L.ntiles, na = (int)p.accs.size(), Px = p.num_x;
        const DAcc* accs = reinterpret_cast<const DAcc*>(base + p.dev_accs);
        const DEntry* entries = reinterpret_cast<const DEntry*>(base + p.dev_entries);
        const DConst* consts = reinterpret_cast<const DConst*>(base + p.dev_consts);
        const R* cang = reinterpret_cast<const R*>(base + p.dev_cang);
        const R* cmat = reinterpret_cast<const R*>(base + p.dev_cmat);
        const R* xr = static_cast<const R*>(x);
        const R* wr = static_cast<const R*>(w);
        R* o = terms;
        void* args[] = {&r, &Bi, &ntl, &na, &accs, &entries, &consts, &cang, &cmat, &xr, &Px, &wr, &nt, &o};
        const int blocks = (int)std::min<long long>(4096, ((long long)B * na + 255) / 256);
        VQC_CUDA(launch(p.dfloat ? reduce_terms_ptr_dd() : reduce_terms_ptr(dbl), dim3(std::max(blocks, 1)),
                        dim3(256), args, 0, stream));
    }
    if (dx && p.num_x > 0) {
        const R* t = terms;
        int Bi = B, ntl = 1, Px = p.num_x;
        const int32_t* ptr = reinterpret_cast<const int32_t*>(base + p.dev_xocc_ptr);
        const int32_t* occ = reinterpret_cast<const int32_t*>(base + p.dev_xocc);
        R* o = static_cast<R*>(dx);
        void* args[] = {&t, &Bi, &ntl, &nt, &ptr, &occ, &Px, &o};
        const int blocks = (int)std::min<long long>(4096, ((long long)B * Px + 255) / 256);
        VQC_CUDA(launch(reduce_dx_ptr(dbl), dim3(std::max(blocks, 1)), dim3(256), args, 0,
                                  stream));
    }
    if (dw && p.num_w > 0) {
        const R* t = terms;
        long long rows = B;
        const int32_t* ptr = reinterpret_cast<const int32_t*>(base + p.dev_wocc_ptr);
        const int32_t* occ = reinterpret_cast<const int32_t*>(base + p.dev_wocc);
        R* o = static_cast<R*>(dw);
        void* args[] = {&t, &rows, &nt, &ptr, &occ, &o};
        VQC_CUDA(launch(reduce_dw_ptr(dbl), dim3(p.num_w), dim3(256), args, 0, stream));
    }
    return VQC_OK;
}

// The resident path when it can take the batch (and VQC_FORCE_PATH does not
// ask for the HBM path), else the HBM path.
bool use_hbm(const HostPlan& p, int mode, int B) {
    const char* f = std::getenv("VQC_FORCE_PATH");
    if (f && std::string(f) == "hbm" && find_hbm_schedule(p, mode)) return true;
    Launch L;
    std::string saved = g_err;
    if (plan_launch(p, mode, B, L) == VQC_OK) return false;
    g_err = saved;
    return find_hbm_schedule(p, mode) != nullptr;
}

// vqc_forward_backward on the resident path: one launch of the fused kernel,
// unless the forward takes a larger register block than the backward.  The
// fused kernel sweeps forward with the backward's schedule, so then the
// forward call (its own, larger blocks) followed by the backward from the saved
// states is faster (12-qubit workload, batch 4096: 2.25 ms against 2.40 ms).
bool resident_two_calls(const HostPlan& p, int B) {
    Launch Lf, Lb;
    const std::string saved = g_err;
    const bool ok = plan_launch(p, 0, B, Lf) == VQC_OK && plan_launch(p, 1, B, Lb) == VQC_OK;
    g_err = saved;
    return ok && Lf.K > Lb.K;
}

// Workspace of the two-call form: [backward workspace | final states].
size_t two_call_state_offset(const HostPlan& p, int B) {
    Launch Lb;
    const std::string saved = g_err;
    const vqc_status st = plan_launch(p, 1, B, Lb);
    g_err = saved;
    return st == VQC_OK ? align256(bwd_workspace(p, Lb)) : 0;
}

std::mutex g_upload_mu;

vqc_status check_common(const vqc_plan* plan, int32_t batch) {
    if (!plan) return fail(VQC_ERR_INVALID_ARG, "plan is NULL");
    if (batch < 0) return fail(VQC_ERR_INVALID_ARG, "batch must be >= 0");
    int dev = -1;
    VQC_CUDA(cudaGetDevice(&dev));
    {
        std::lock_guard<std::mutex> lk(g_upload_mu);
        if (!plan->hp.dbuf) {
            vqc_status st = upload(const_cast<vqc_plan*>(plan)->hp);
            if (st != VQC_OK) return st;
        }
    }
    if (dev != plan->hp.device)
        return fail(VQC_ERR_INVALID_ARG, "plan was compiled for device " +
                                             std::to_string(plan->hp.device) +
                                             " but the current device is " + std::to_string(dev));
    return VQC_OK;
}

// Real arrays (E, gE, dx, dw, probabilities) must be aligned to the real type,
// state arrays to the complex type; NULL passes (each call checks presence).
vqc_status check_out_ptrs(const HostPlan& p, std::initializer_list<const void*> reals,
                          std::initializer_list<const void*> states) {
    const size_t rs = p.dtype == VQC_C128 ? 8 : 4;
    for (const void* q : reals)
        if (q && misaligned(q, rs)) return fail(VQC_ERR_INVALID_ARG, "real arrays must be aligned to the real type");
    for (const void* q : states)
        if (q && misaligned(q, 2 * rs))
            return fail(VQC_ERR_INVALID_ARG, "state arrays must be aligned to the complex type");
    return VQC_OK;
}

vqc_status check_ptrs(const HostPlan& p, const void* x, const void* w, const void* psi0,
                      const void* psi_final) {
    const size_t rs = p.dtype == VQC_C128 ? 8 : 4;
    if (p.num_x > 0 && !x) return fail(VQC_ERR_INVALID_ARG, "x is NULL but the circuit uses x");
    if (p.num_w > 0 && !w) return fail(VQC_ERR_INVALID_ARG, "w is NULL but the circuit uses w");
    if ((x && misaligned(x, rs)) || (w && misaligned(w, rs)))
        return fail(VQC_ERR_INVALID_ARG, "x / w must be aligned to the real type");
    if ((psi0 && misaligned(psi0, 2 * rs)) || (psi_final && misaligned(psi_final, 2 * rs)))
        return fail(VQC_ERR_INVALID_ARG, "state arrays must be aligned to the complex type");
    return VQC_OK;
}

}  // namespace

vqc_status set_error(vqc_status s, const std::string& msg) { return fail(s, msg); }

// tc_stage.cu: the error word of vqc_stage_apply's kernels (read and cleared).
vqc_status stage_error_check();

// host_eval.cu: the per-plan arena of vqc_evaluate_host.
void release_host_arena(const vqc_plan* plan);

// The backward with an explicit scratch buffer, for vqc_backward_noalloc: the
// scratch must hold the same layout as a vqc_backward workspace; with
// clear_control the control block is zeroed on `stream` before the launch.
vqc_status backward_with_scratch(const vqc_plan* plan, int32_t batch, const void* x,
                                 const void* w, const void* psi0, const void* psi_final,
                                 const void* grad_expz, void* grad_x, void* grad_w, void* scratch,
                                 size_t scratch_bytes, void* stream, bool clear_control) {
    vqc_status st = check_common(plan, batch);
    if (st != VQC_OK) return st;
    const HostPlan& p = plan->hp;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (batch == 0) {
        if (grad_w && p.num_w > 0)
            VQC_CUDA(cudaMemsetAsync(grad_w, 0, (size_t)p.num_w * (p.dtype == VQC_C128 ? 8 : 4), s));
        return VQC_OK;
    }
    st = check_ptrs(p, x, w, psi0, psi_final);
    if (st != VQC_OK) return st;
    if (!grad_expz) return fail(VQC_ERR_INVALID_ARG, "grad_expz is NULL");
    st = check_out_ptrs(p, {grad_expz, grad_x, grad_w}, {});
    if (st != VQC_OK) return st;
    // the same path choice as vqc_backward: the cluster backward when the
    // environment asks for it, resident when the batch fits a resident launch,
    // else the HBM-tiled passes (each with its own workspace layout)
    const bool clu = use_cluster(p, 1);
    const bool hbm = !clu && use_hbm(p, 1, batch);
    size_t need = 0;
    if (clu) {
        Launch L;
        st = plan_cluster(p, 1, batch, L);
        if (st != VQC_OK) return st;
        need = cluster_bwd_workspace(p, L);
    } else if (hbm) {
        PassGeo L;
        st = plan_hbm(p, 1, batch, L);
        if (st != VQC_OK) return st;
        need = hbm_layout(p, 1, batch, L.ntiles).total;
    } else {
        Launch L;
        st = plan_launch(p, 1, batch, L);
        if (st != VQC_OK) return st;
        need = bwd_workspace(p, L);
    }
    if (need > scratch_bytes)
        return fail(VQC_ERR_WORKSPACE, "this batch needs " + std::to_string(need) +
                                           " bytes of scratch; the built-in scratch holds " +
                                           std::to_string(scratch_bytes));
    if (clear_control) VQC_CUDA(cudaMemsetAsync(scratch, 0, 256, s));
    if (clu) {
        if (p.dtype == VQC_C64)
            return run_cluster_backward<float>(p, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                               grad_w, scratch, scratch_bytes, s);
        return run_cluster_backward<double>(p, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                            grad_w, scratch, scratch_bytes, s);
    }
    if (hbm) {
        if (p.dtype == VQC_C64)
            return run_hbm_backward<float>(p, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                           grad_w, scratch, scratch_bytes, s);
        return run_hbm_backward<double>(p, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                        grad_w, scratch, scratch_bytes, s);
    }
    if (p.dtype == VQC_C64)
        return run<float>(p, 1, batch, x, w, psi0, psi_final, grad_expz, nullptr, nullptr, grad_x,
                          grad_w, scratch, scratch_bytes, s);
    return run<double>(p, 1, batch, x, w, psi0, psi_final, grad_expz, nullptr, nullptr, grad_x,
                       grad_w, scratch, scratch_bytes, s);
}

}  // namespace vqc

using namespace vqc;

extern "C" {

vqc_status vqc_compile(const vqc_gate* gates, int32_t num_gates, int32_t num_qubits,
                       int32_t num_x, int32_t num_w, vqc_dtype dtype, vqc_plan** out_plan) {
    try {
        if (!out_plan) return fail(VQC_ERR_INVALID_ARG, "out_plan is NULL");
        *out_plan = nullptr;
        if (num_gates < 0 || num_x < 0 || num_w < 0 || (num_gates > 0 && !gates))
            return fail(VQC_ERR_INVALID_ARG, "negative count or NULL gate list");
        if (dtype != VQC_C64 && dtype != VQC_C128 && dtype != VQC_C128_DF)
            return fail(VQC_ERR_INVALID_ARG, "bad dtype");
        if (num_qubits < 1 || num_qubits > VQC_MAX_QUBITS)
            return fail(VQC_ERR_TOO_MANY_QUBITS, "num_qubits must be in 1.." +
                                                     std::to_string(VQC_MAX_QUBITS));
        std::unique_ptr<vqc_plan> p(new vqc_plan());
        std::string err;
        // VQC_C128_DF plans are complex128 plans (same layouts and schedules)
        // whose kernels compute in double-float
        const vqc_dtype store = dtype == VQC_C128_DF ? VQC_C128 : dtype;
        vqc_status st = compile_host(gates, num_gates, num_qubits, num_x, num_w, store, p->hp, err);
        if (st != VQC_OK) return fail(st, err);
        p->hp.dfloat = dtype == VQC_C128_DF;
        // Upload now when a CUDA device is present; a host-only plan (no device
        // in this process) still serves vqc_plan_export and vqc_plan_info, and
        // is uploaded by the first launching call.
        int ndev = 0;
        if (cudaGetDeviceCount(&ndev) != cudaSuccess) {
            (void)cudaGetLastError();
            ndev = 0;
        }
        if (ndev > 0) {
            st = upload(p->hp);
            if (st != VQC_OK) return st;
        }
        *out_plan = p.release();
        return VQC_OK;
    } catch (const std::bad_alloc&) {
        return fail(VQC_ERR_OUT_OF_MEMORY, "host allocation failed");
    } catch (...) {
        return fail(VQC_ERR_INVALID_ARG, "internal error in vqc_compile");
    }
}

void vqc_free(vqc_plan* plan) {
    if (!plan) return;
    {
        std::lock_guard<std::mutex> lk(g_plans_mu);
        g_plans.erase(&plan->hp);
    }
    forget_plan(&plan->hp);
    release_host_arena(plan);
    if (plan->hp.dbuf) {
        int cur = -1;
        cudaGetDevice(&cur);
        if (cur != plan->hp.device) cudaSetDevice(plan->hp.device);
        cudaFree(plan->hp.dbuf);
        if (cur != plan->hp.device && cur >= 0) cudaSetDevice(cur);
    }
    delete plan;
}

size_t vqc_workspace_bytes(const vqc_plan* plan, int32_t batch, int32_t mode) {
    if (!plan) return (size_t)-1;
    if (mode == 3) {   // vqc_forward_backward: its one-launch form, or either call's workspace
        size_t need = std::max(vqc_workspace_bytes(plan, batch, 0), vqc_workspace_bytes(plan, batch, 1));
        const HostPlan& p = plan->hp;
        Launch L;
        const std::string saved = g_err;
        if (batch > 0 && !use_cluster(p, 0) && !use_hbm(p, 0, batch) && !use_hbm(p, 1, batch)) {
            if (resident_two_calls(p, batch)) {
                const size_t cs = p.dtype == VQC_C128 ? 16 : 8;
                need = std::max(need, two_call_state_offset(p, batch) + align256(((size_t)batch << p.n) * cs));
            } else if (plan_launch(p, 2, batch, L) == VQC_OK) {
                need = std::max(need, bwd_workspace(p, L));
            }
        }
        if (batch > 0 && use_cluster(p, 1)) {   // [either call's workspace | final states]
            const size_t cs = p.dtype == VQC_C128 ? 16 : 8;
            need = align256(need) + align256(((size_t)batch << p.n) * cs);
        }
        g_err = saved;
        return need;
    }
    if (mode == 2 && batch > 0) {   // vqc_probabilities: forward workspace + state + E
        const HostPlan& p = plan->hp;
        const size_t rs = p.dtype == VQC_C128 ? 8 : 4;
        return align256(vqc_workspace_bytes(plan, batch, 0)) +
               align256(((size_t)batch << p.n) * 2 * rs) + align256((size_t)batch * p.n * rs);
    }
    if ((mode != 0 && mode != 1) || batch <= 0) return 0;
    const HostPlan& p = plan->hp;
    if (use_cluster(p, mode)) {
        if (mode == 0) return 0;
        Launch L;
        if (plan_cluster(p, 1, batch, L) != VQC_OK) return 0;
        return cluster_bwd_workspace(p, L);
    }
    if (use_hbm(p, mode, batch)) {
        PassGeo L;
        if (plan_hbm(p, mode, batch, L) != VQC_OK) return 0;
        return hbm_layout(p, mode, batch, L.ntiles).total;
    }
    if (mode == 0) return 0;
    Launch L;
    if (plan_launch(p, 1, batch, L) != VQC_OK) return 0;
    return bwd_workspace(p, L);
}

vqc_status vqc_probabilities(const vqc_plan* plan, int32_t batch, const void* x, const void* w,
                             const void* psi0, void* probs_out, void* workspace,
                             size_t workspace_bytes, void* stream) {
    try {
        vqc_status st = check_common(plan, batch);
        if (st != VQC_OK) return st;
        if (batch == 0) return VQC_OK;
        const HostPlan& p = plan->hp;
        if (!probs_out) return fail(VQC_ERR_INVALID_ARG, "probs_out is NULL");
        st = check_out_ptrs(p, {probs_out}, {});
        if (st != VQC_OK) return st;
        const bool dbl = p.dtype == VQC_C128;
        const size_t rs = dbl ? 8 : 4;
        const size_t fws = vqc_workspace_bytes(plan, batch, 0);
        const size_t need = vqc_workspace_bytes(plan, batch, 2);
        if (!workspace || workspace_bytes < need || misaligned(workspace, 256))
            return fail(VQC_ERR_WORKSPACE, "probabilities workspace must be >= " + std::to_string(need) +
                                               " bytes and 256-byte aligned");
        char* base = static_cast<char*>(workspace);
        void* state = base + align256(fws);
        void* E = base + align256(fws) + align256(((size_t)batch << p.n) * 2 * rs);
        st = vqc_forward(plan, batch, x, w, psi0, E, state, fws ? workspace : nullptr, fws, stream);
        if (st != VQC_OK) return st;
        cudaStream_t s = static_cast<cudaStream_t>(stream);
        long long count = (long long)batch << p.n;
        int blocks = (int)std::min<long long>((count + 255) / 256, 152LL * 16);
        const void* src = state;
        void* dst = probs_out;
        void* args[] = {&src, &count, &dst};
        VQC_CUDA(launch(abs2_ptr(dbl), dim3(std::max(blocks, 1)), dim3(256), args, 0, s));
        return VQC_OK;
    } catch (...) {
        return fail(VQC_ERR_INVALID_ARG, "internal error in vqc_probabilities");
    }
}

vqc_status vqc_workspace_init(void* workspace, size_t workspace_bytes, void* stream) {
    if (!workspace || workspace_bytes < 256) return fail(VQC_ERR_WORKSPACE, "workspace too small");
    VQC_CUDA(cudaMemsetAsync(workspace, 0, 256, static_cast<cudaStream_t>(stream)));
    return VQC_OK;
}

vqc_status vqc_forward(const vqc_plan* plan, int32_t batch, const void* x, const void* w,
                       const void* psi0, void* expz_out, void* state_out, void* workspace,
                       size_t workspace_bytes, void* stream) {
    try {
        vqc_status st = check_common(plan, batch);
        if (st != VQC_OK) return st;
        if (batch == 0) return VQC_OK;
        const HostPlan& p = plan->hp;
        st = check_ptrs(p, x, w, psi0, nullptr);
        if (st != VQC_OK) return st;
        if (!expz_out) return fail(VQC_ERR_INVALID_ARG, "expz_out is NULL");
        st = check_out_ptrs(p, {expz_out}, {state_out});
        if (st != VQC_OK) return st;
        cudaStream_t s = static_cast<cudaStream_t>(stream);
        if (use_cluster(p, 0)) {
            if (p.dtype == VQC_C64)
                return run_cluster_forward<float>(p, batch, x, w, psi0, expz_out, state_out, s);
            return run_cluster_forward<double>(p, batch, x, w, psi0, expz_out, state_out, s);
        }
        if (use_hbm(p, 0, batch)) {
            if (p.dtype == VQC_C64)
                return run_hbm_forward<float>(p, batch, x, w, psi0, expz_out, state_out, workspace,
                                              workspace_bytes, s, true);
            return run_hbm_forward<double>(p, batch, x, w, psi0, expz_out, state_out, workspace,
                                           workspace_bytes, s, true);
        }
        if (p.dtype == VQC_C64)
            return run<float>(p, 0, batch, x, w, psi0, nullptr, nullptr, expz_out, state_out,
                              nullptr, nullptr, nullptr, 0, s);
        return run<double>(p, 0, batch, x, w, psi0, nullptr, nullptr, expz_out, state_out, nullptr,
                           nullptr, nullptr, 0, s);
    } catch (...) {
        return fail(VQC_ERR_INVALID_ARG, "internal error in vqc_forward");
    }
}

vqc_status vqc_backward(const vqc_plan* plan, int32_t batch, const void* x, const void* w,
                        const void* psi0, const void* psi_final, const void* grad_expz,
                        void* grad_x, void* grad_w, void* workspace, size_t workspace_bytes,
                        void* stream) {
    try {
        vqc_status st = check_common(plan, batch);
        if (st != VQC_OK) return st;
        const HostPlan& p = plan->hp;
        cudaStream_t s = static_cast<cudaStream_t>(stream);
        if (batch == 0) {
            if (grad_w && p.num_w > 0)
                VQC_CUDA(cudaMemsetAsync(grad_w, 0, (size_t)p.num_w * (p.dtype == VQC_C128 ? 8 : 4), s));
            return VQC_OK;
        }
        st = check_ptrs(p, x, w, psi0, psi_final);
        if (st != VQC_OK) return st;
        if (!grad_expz) return fail(VQC_ERR_INVALID_ARG, "grad_expz is NULL");
        st = check_out_ptrs(p, {grad_expz, grad_x, grad_w}, {});
        if (st != VQC_OK) return st;
        if (use_cluster(p, 1)) {
            if (p.dtype == VQC_C64)
                return run_cluster_backward<float>(p, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                                   grad_w, workspace, workspace_bytes, s);
            return run_cluster_backward<double>(p, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                                grad_w, workspace, workspace_bytes, s);
        }
        if (use_hbm(p, 1, batch)) {
            if (p.dtype == VQC_C64)
                return run_hbm_backward<float>(p, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                               grad_w, workspace, workspace_bytes, s);
            return run_hbm_backward<double>(p, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                            grad_w, workspace, workspace_bytes, s);
        }
        if (p.dtype == VQC_C64)
            return run<float>(p, 1, batch, x, w, psi0, psi_final, grad_expz, nullptr, nullptr,
                              grad_x, grad_w, workspace, workspace_bytes, s);
        return run<double>(p, 1, batch, x, w, psi0, psi_final, grad_expz, nullptr, nullptr, grad_x,
                           grad_w, workspace, workspace_bytes, s);
    } catch (...) {
        return fail(VQC_ERR_INVALID_ARG, "internal error in vqc_backward");
    }
}

vqc_status vqc_forward_backward(const vqc_plan* plan, int32_t batch, const void* x, const void* w,
                                const void* psi0, const void* grad_expz, void* expz_out, void* grad_x,
                                void* grad_w, void* workspace, size_t workspace_bytes, void* stream) {
    try {
        vqc_status st = check_common(plan, batch);
        if (st != VQC_OK) return st;
        const HostPlan& p = plan->hp;
        cudaStream_t s = static_cast<cudaStream_t>(stream);
        if (batch == 0) {
            if (grad_w && p.num_w > 0)
                VQC_CUDA(cudaMemsetAsync(grad_w, 0, (size_t)p.num_w * (p.dtype == VQC_C128 ? 8 : 4), s));
            return VQC_OK;
        }
        st = check_ptrs(p, x, w, psi0, nullptr);
        if (st != VQC_OK) return st;
        if (!grad_expz) return fail(VQC_ERR_INVALID_ARG, "grad_expz is NULL");
        if (!expz_out) return fail(VQC_ERR_INVALID_ARG, "expz_out is NULL");
        st = check_out_ptrs(p, {expz_out, grad_expz, grad_x, grad_w}, {});
        if (st != VQC_OK) return st;
        if (!use_cluster(p, 0) && !use_hbm(p, 0, batch) && !use_hbm(p, 1, batch) &&
            resident_two_calls(p, batch)) {
            // the forward (larger register blocks) saves the final states after the
            // backward's workspace; the backward starts from them
            const size_t need = vqc_workspace_bytes(plan, batch, 3);
            if (!workspace || workspace_bytes < need || misaligned(workspace, 256))
                return fail(VQC_ERR_WORKSPACE, "workspace must be >= " + std::to_string(need) +
                                                   " bytes and 256-byte aligned");
            void* psi_final = static_cast<char*>(workspace) + two_call_state_offset(p, batch);
            st = vqc_forward(plan, batch, x, w, psi0, expz_out, psi_final, nullptr, 0, stream);
            if (st != VQC_OK) return st;
            return vqc_backward(plan, batch, x, w, psi0, psi_final, grad_expz, grad_x, grad_w, workspace,
                                workspace_bytes, stream);
        }
        if (!use_cluster(p, 0) && !use_hbm(p, 0, batch) && !use_hbm(p, 1, batch)) {
            // one launch: the backward kernel sweeps forward itself (the state stays in
            // shared memory), writes E, then sweeps back
            if (p.dtype == VQC_C64)
                return run<float>(p, 2, batch, x, w, psi0, nullptr, grad_expz, expz_out, nullptr, grad_x,
                                  grad_w, workspace, workspace_bytes, s);
            return run<double>(p, 2, batch, x, w, psi0, nullptr, grad_expz, expz_out, nullptr, grad_x,
                               grad_w, workspace, workspace_bytes, s);
        }
        if (use_cluster(p, 1)) {
            // the forward leaves the final states after the larger of the two calls'
            // workspaces; the cluster backward starts from them
            const size_t need = vqc_workspace_bytes(plan, batch, 3);
            if (!workspace || workspace_bytes < need || misaligned(workspace, 256))
                return fail(VQC_ERR_WORKSPACE, "workspace must be >= " + std::to_string(need) +
                                                   " bytes and 256-byte aligned");
            const size_t cs = p.dtype == VQC_C128 ? 16 : 8;
            const size_t soff = need - align256(((size_t)batch << p.n) * cs);
            void* psi_final = static_cast<char*>(workspace) + soff;
            st = vqc_forward(plan, batch, x, w, psi0, expz_out, psi_final, workspace, soff, stream);
            if (st != VQC_OK) return st;
            return vqc_backward(plan, batch, x, w, psi0, psi_final, grad_expz, grad_x, grad_w, workspace,
                                soff, stream);
        }
        // states beyond one SM: the forward (passes or cluster) leaves the final
        // states in the psi region of the backward's HBM layout, in this
        // workspace, and the backward passes start from them (the forward's own
        // working state is that region too, and its <Z> partials sit where the
        // backward's lam goes: both are consumed before the backward starts)
        if (use_hbm(p, 1, batch)) {
            PassGeo Lb;
            st = plan_hbm(p, 1, batch, Lb);
            if (st != VQC_OK) return st;
            const HbmWs lay = hbm_layout(p, 1, batch, Lb.ntiles);
            const size_t need = vqc_workspace_bytes(plan, batch, 3);
            if (!workspace || workspace_bytes < need || misaligned(workspace, 256))
                return fail(VQC_ERR_WORKSPACE, "workspace must be >= " + std::to_string(need) +
                                                   " bytes and 256-byte aligned");
            void* psi_final = static_cast<char*>(workspace) + lay.state;
            st = vqc_forward(plan, batch, x, w, psi0, expz_out, psi_final, workspace, workspace_bytes,
                             stream);
            if (st != VQC_OK) return st;
            return vqc_backward(plan, batch, x, w, psi0, psi_final, grad_expz, grad_x, grad_w,
                                workspace, workspace_bytes, stream);
        }
        st = vqc_forward(plan, batch, x, w, psi0, expz_out, nullptr, workspace, workspace_bytes, stream);
        if (st != VQC_OK) return st;
        return vqc_backward(plan, batch, x, w, psi0, nullptr, grad_expz, grad_x, grad_w, workspace,
                            workspace_bytes, stream);
    } catch (...) {
        return fail(VQC_ERR_INVALID_ARG, "internal error in vqc_forward_backward");
    }
}

vqc_status vqc_plan_info(const vqc_plan* plan, int32_t batch, vqc_plan_stats* out) {
    if (!plan || !out) return fail(VQC_ERR_INVALID_ARG, "NULL argument");
    const HostPlan& p = plan->hp;
    std::memset(out, 0, sizeof(*out));
    out->num_qubits = p.n;
    out->num_x = p.num_x;
    out->num_w = p.num_w;
    out->dtype = p.dfloat ? VQC_C128_DF : p.dtype;
    out->num_gates_in = p.num_gates_in;
    out->num_ops = (int32_t)p.ops.size();
    out->num_runs = p.n_runs;
    out->num_terms = (int32_t)p.term_src.size();
    out->fwd_flops_per_eval = p.fwd_flops;
    out->bwd_flops_per_eval = p.bwd_flops;
    out->recompute_flops_per_eval = p.recompute_flops;
    const int B = std::max(batch, 1);
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess) {
        (void)cudaGetLastError();
        ndev = 0;
    }
    const std::string saved = g_err;
    int sms = 152;   // without a device: GB300's SM count
    if (ndev > 0) {
        int dev = 0;
        DevInfo di;
        if (cudaGetDevice(&dev) == cudaSuccess && device_info(dev, di) == VQC_OK) sms = di.sms;
        else (void)cudaGetLastError();
    }
    const double sbytes = std::ldexp(1.0, p.n) * (p.dtype == VQC_C128 ? 16.0 : 8.0);
    for (int mode = 0; mode < 2; ++mode) {
        int* path = mode == 0 ? &out->fwd_path : &out->bwd_path;
        int* kk = mode == 0 ? &out->fwd_k : &out->bwd_k;
        int* ns = mode == 0 ? &out->fwd_stages : &out->bwd_stages;
        int* np = mode == 0 ? &out->fwd_passes : &out->bwd_passes;
        int* tps = mode == 0 ? &out->fwd_threads_per_sample : &out->bwd_threads_per_sample;
        int* tq = mode == 0 ? &out->fwd_tile_qubits : &out->bwd_tile_qubits;
        double* hb = mode == 0 ? &out->fwd_hbm_bytes_per_eval : &out->bwd_hbm_bytes_per_eval;
        const int K = choose_k(p, mode, B, sms);
        const bool clu = use_cluster(p, mode);
        const bool hbm = !clu && (ndev > 0 ? use_hbm(p, mode, B)
                                           : (K == 0 && find_hbm_schedule(p, mode) != nullptr));
        const Schedule* s = clu ? find_cluster_schedule(p, mode)
                          : hbm ? find_hbm_schedule(p, mode) : (K ? find_schedule(p, mode, K) : nullptr);
        if (!s) {
            *path = -1;
            continue;
        }
        *path = s->path;
        *kk = s->K;
        *ns = (int)s->stages.size();
        *tq = s->m;
        if (hbm) {
            const int P = (int)s->passes.size();
            *np = P;
            *tps = (1 << (s->m - s->K)) << (p.n - s->m);
            // state traffic: forward reads and writes the state once per pass;
            // the backward reads psi (and lam after the first pass) and writes
            // both (except after the last pass)
            *hb = mode == 0 ? 2.0 * P * sbytes : (4.0 * P - 3.0) * sbytes;
        } else {
            *np = 1;
            *tps = 1 << (p.n - s->K);
        }
    }
    g_err = saved;
    return VQC_OK;
}

vqc_status vqc_plan_export(const vqc_plan* plan, void* buf, size_t* inout_bytes) {
    if (!plan || !inout_bytes) return fail(VQC_ERR_INVALID_ARG, "NULL argument");
    try {
        std::vector<uint8_t> b = export_plan(plan->hp);
        size_t cap = *inout_bytes;
        *inout_bytes = b.size();
        if (!buf) return VQC_OK;
        if (cap < b.size()) return fail(VQC_ERR_INVALID_ARG, "buffer too small");
        std::memcpy(buf, b.data(), b.size());
        return VQC_OK;
    } catch (...) {
        return fail(VQC_ERR_OUT_OF_MEMORY, "export failed");
    }
}

vqc_status vqc_sync_check(void* stream) {
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetLastError");
    // the kernels' launch self-checks: each plan's error word on this device
    int dev = -1;
    VQC_CUDA(cudaGetDevice(&dev));
    std::vector<const HostPlan*> plans;
    {
        std::lock_guard<std::mutex> lk(g_plans_mu);
        plans.assign(g_plans.begin(), g_plans.end());
    }
    unsigned tripped = 0;
    for (const HostPlan* p : plans) {
        if (p->device != dev || !p->dev_error) continue;
        unsigned w = 0;
        VQC_CUDA(cudaMemcpy(&w, p->dev_error, sizeof(w), cudaMemcpyDeviceToHost));
        if (w) {
            tripped |= w;
            VQC_CUDA(cudaMemset(p->dev_error, 0, sizeof(w)));
        }
    }
    if (tripped)
        return fail(VQC_ERR_DEVICE_CHECK,
                    std::string("a kernel's launch self-check tripped:") +
                        ((tripped & 1u) ? " resident sweep geometry" : "") +
                        ((tripped & 2u) ? " HBM pass geometry" : "") +
                        ((tripped & 4u) ? " cluster geometry" : "") + " (the work was skipped)");
    return stage_error_check();   // vqc_stage_apply's tensor-core waits
}

const char* vqc_last_error(void) { return g_err.c_str(); }

int32_t vqc_abi_version(void) { return VQC_ABI_VERSION; }

}  // extern "C"
