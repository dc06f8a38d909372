// host_eval.cu -- vqc_evaluate_host: one batched evaluation whose inputs and
// outputs are in host memory.
//
// A caller that holds its angles in host memory (a training loop on the CPU
// side, a service answering requests) would otherwise pay three host-to-device
// copies, the forward, the backward, three device-to-host copies and their
// per-call overheads.  Here the plan keeps a device arena (packed inputs,
// packed outputs, the workspace) and a pinned host mirror of the packed inputs
// and outputs, sized for the largest batch seen:
//   host x, w, gE  --memcpy-->  pinned [x | w | gE]  --1 copy-->  device
//   vqc_forward_backward (E, dx, dw; one launch on the resident path)
//   device [E | dx | dw]  --1 copy-->  pinned  --memcpy-->  host E, dx, dw
// and the call returns after the stream has finished.  Where the device can
// access pageable host memory coherently (cudaDevAttrPageableMemoryAccess, e.g.
// a Grace-Blackwell node over NVLink-C2C) there is no staging at all: the
// kernels read x, w, gE from and write E, dx, dw to the caller's arrays
// (VQC_HOST_DIRECT=0 forces the staged copies).  From the second call with the
// same batch and outputs (and, direct, the same arrays) on, the device part is
// one CUDA graph launch (captured once on a private stream; VQC_HOST_GRAPH=0
// turns this off).  The arena is released by vqc_free.
#include <cuda_runtime.h>

#include <cstdlib>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>
#include <string>

#include "engine.h"

namespace vqc {
vqc_status set_error(vqc_status s, const std::string& msg);
}  // namespace vqc

namespace {

size_t up256(size_t v) { return (v + 255) & ~(size_t)255; }

// Byte offsets of one batch size's layout.  The pinned mirror holds the
// input region [0, in_bytes) and the output region [out, out + out_bytes).
struct Layout {
    size_t x = 0, w = 0, g = 0, in_bytes = 0;
    size_t out = 0, E = 0, dx = 0, dw = 0, out_bytes = 0;
    size_t ws0 = 0, ws0_bytes = 0, ws1 = 0, ws1_bytes = 0, dev_bytes = 0;
    bool operator==(const Layout& o) const { return std::memcmp(this, &o, sizeof(Layout)) == 0; }
};

struct Arena {
    std::mutex mu;
    int device = -1;
    unsigned char* dev = nullptr;
    size_t dev_cap = 0;
    unsigned char* pin = nullptr;
    size_t pin_cap = 0;
    Layout last;          // layout whose workspaces were last initialised
    bool have_last = false;
    // The call's device work as a CUDA graph, captured on a private stream the
    // second time the same (batch, outputs) shape is seen and replayed after.
    cudaStream_t cap = nullptr;
    cudaGraphExec_t exec = nullptr;
    int shape_batch = -1, shape_flags = -1;   // shape of the previous call
    const void* shape_ptrs[6] = {};           // its host arrays (direct access: part of the shape)
    bool graph_failed = false;
    void drop_graph() {
        if (exec) cudaGraphExecDestroy(exec);
        exec = nullptr;
    }
    ~Arena() {
        drop_graph();
        if (cap) cudaStreamDestroy(cap);
        if (dev) cudaFree(dev);
        if (pin) cudaFreeHost(pin);
    }
};

std::mutex g_arena_mu;
std::map<const vqc_plan*, std::unique_ptr<Arena>> g_arenas;

Arena* arena_of(const vqc_plan* plan) {
    std::lock_guard<std::mutex> lk(g_arena_mu);
    std::unique_ptr<Arena>& a = g_arenas[plan];
    if (!a) a.reset(new Arena());
    return a.get();
}

Layout layout_for(const vqc_plan* plan, int B, bool bwd) {
    const vqc::HostPlan& p = plan->hp;
    const size_t rs = p.dtype == VQC_C128 ? 8 : 4;
    Layout L;
    size_t o = 0;
    L.x = o; o = up256(o + (size_t)B * p.num_x * rs);
    L.w = o; o = up256(o + (size_t)p.num_w * rs);
    L.g = o; o = up256(o + (bwd ? (size_t)B * p.n * rs : 0));
    L.in_bytes = o;
    L.out = o;
    L.E = o - L.out; o = up256(o + (size_t)B * p.n * rs);
    L.dx = o - L.out; o = up256(o + (bwd ? (size_t)B * p.num_x * rs : 0));
    L.dw = o - L.out; o = up256(o + (bwd ? (size_t)p.num_w * rs : 0));
    L.out_bytes = o - L.out;
    // forward only: vqc_forward's workspace; with gE: vqc_forward_backward's
    L.ws0_bytes = bwd ? 0 : vqc_workspace_bytes(plan, B, 0);
    L.ws0 = o; o = up256(o + L.ws0_bytes);
    L.ws1_bytes = bwd ? vqc_workspace_bytes(plan, B, 3) : 0;
    L.ws1 = o; o = up256(o + L.ws1_bytes);
    L.dev_bytes = o;
    return L;
}

vqc_status cuda_err(cudaError_t e, const char* what) {
    return vqc::set_error(VQC_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

bool env_flag(const char* name, bool dflt) {
    const char* v = std::getenv(name);
    return v ? std::atoi(v) != 0 : dflt;
}

// Whether kernels on `dev` may read and write pageable host memory directly
// (cudaDevAttrPageableMemoryAccess: coherent access through the host's page
// tables, as on Grace-Blackwell's NVLink-C2C).  Queried once per device.
bool host_direct(int dev) {
    static std::mutex mu;
    static int known[64];
    static bool init = false;
    if (dev < 0 || dev >= 64) return false;
    std::lock_guard<std::mutex> lk(mu);
    if (!init) {
        for (int& k : known) k = -1;
        init = true;
    }
    if (known[dev] < 0) {
        int v = 0;
        if (cudaDeviceGetAttribute(&v, cudaDevAttrPageableMemoryAccess, dev) != cudaSuccess) {
            (void)cudaGetLastError();
            v = 0;
        }
        known[dev] = v ? 1 : 0;
    }
    return known[dev] == 1;
}

// Capture enqueue() on the arena's private stream into an executable graph.
// Returns nullptr (and stops trying for this arena) when any step refuses to
// be captured; the caller then enqueues directly, as on the first call.
template <typename F>
cudaGraphExec_t capture(Arena* A, F& enqueue) {
    if (!A->cap && cudaStreamCreateWithFlags(&A->cap, cudaStreamNonBlocking) != cudaSuccess) {
        (void)cudaGetLastError();
        A->cap = nullptr;
        A->graph_failed = true;
        return nullptr;
    }
    cudaGraph_t g = nullptr;
    cudaGraphExec_t ex = nullptr;
    if (cudaStreamBeginCapture(A->cap, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
        (void)cudaGetLastError();
        A->graph_failed = true;
        return nullptr;
    }
    const std::string saved = vqc_last_error();
    const vqc_status st = enqueue(A->cap);
    const cudaError_t e1 = cudaStreamEndCapture(A->cap, &g);
    bool ok = st == VQC_OK && e1 == cudaSuccess && g;
    if (ok && cudaGraphInstantiate(&ex, g, 0) != cudaSuccess) ok = false;
    if (g) cudaGraphDestroy(g);
    if (!ok) {
        if (ex) cudaGraphExecDestroy(ex);
        ex = nullptr;
        (void)cudaGetLastError();
        vqc::set_error(VQC_OK, saved);   // a refused capture is not the caller's error
        A->graph_failed = true;
    }
    return ex;
}

}  // namespace

namespace vqc {
// Called by vqc_free: drop the plan's arena (its address may be reused).
void release_host_arena(const vqc_plan* plan) {
    std::unique_ptr<Arena> a;
    {
        std::lock_guard<std::mutex> lk(g_arena_mu);
        auto it = g_arenas.find(plan);
        if (it == g_arenas.end()) return;
        a = std::move(it->second);
        g_arenas.erase(it);
    }
    if (a && a->device >= 0) {
        const int owner = a->device;
        int cur = -1;
        cudaGetDevice(&cur);
        if (cur != owner) cudaSetDevice(owner);
        a.reset();   // frees on the owning device
        if (cur != owner && cur >= 0) cudaSetDevice(cur);
    }
}
}  // namespace vqc

extern "C" vqc_status vqc_evaluate_host(const vqc_plan* plan, int32_t batch, const void* x,
                                        const void* w, const void* grad_expz, void* expz_out,
                                        void* grad_x, void* grad_w, void* stream) {
    try {
        if (!plan) return vqc::set_error(VQC_ERR_INVALID_ARG, "plan is NULL");
        if (batch < 0) return vqc::set_error(VQC_ERR_INVALID_ARG, "batch must be >= 0");
        const vqc::HostPlan& p = plan->hp;
        const size_t rs = p.dtype == VQC_C128 ? 8 : 4;
        const bool bwd = grad_expz != nullptr;
        if (batch == 0) {
            if (bwd && grad_w && p.num_w > 0) std::memset(grad_w, 0, (size_t)p.num_w * rs);
            return VQC_OK;
        }
        if (p.num_x > 0 && !x) return vqc::set_error(VQC_ERR_INVALID_ARG, "x is NULL but the circuit uses x");
        if (p.num_w > 0 && !w) return vqc::set_error(VQC_ERR_INVALID_ARG, "w is NULL but the circuit uses w");
        if (!expz_out) return vqc::set_error(VQC_ERR_INVALID_ARG, "expz_out is NULL");
        int dev = -1;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return cuda_err(e, "cudaGetDevice");
        cudaStream_t s = static_cast<cudaStream_t>(stream);

        Arena* A = arena_of(plan);
        std::lock_guard<std::mutex> lk(A->mu);
        if (A->device >= 0 && A->device != dev)
            return vqc::set_error(VQC_ERR_INVALID_ARG, "vqc_evaluate_host: the plan's arena is on device " +
                                                           std::to_string(A->device) + ", current device is " +
                                                           std::to_string(dev));
        const bool direct = env_flag("VQC_HOST_DIRECT", true) && host_direct(dev);
        const int flags = (bwd ? 1 : 0) | (bwd && grad_x ? 2 : 0) | (bwd && grad_w ? 4 : 0) |
                          (direct ? 8 : 0);
        const void* ptrs[6] = {x, w, grad_expz, expz_out, grad_x, grad_w};
        bool same_shape = A->shape_batch == batch && A->shape_flags == flags;
        if (direct)
            for (int i = 0; i < 6; ++i) same_shape = same_shape && A->shape_ptrs[i] == ptrs[i];
        if (!same_shape) A->drop_graph();
        // A captured graph holds this shape's layout (the arena and workspaces it
        // was recorded on): reuse it instead of planning the launches again.
        const Layout L = (A->exec && A->have_last) ? A->last : layout_for(plan, batch, bwd);
        if (L.dev_bytes > A->dev_cap) {
            A->drop_graph();
            if (A->dev) {
                e = cudaStreamSynchronize(s);
                if (e != cudaSuccess) return cuda_err(e, "cudaStreamSynchronize");
                cudaFree(A->dev);
                A->dev = nullptr;
                A->dev_cap = 0;
            }
            e = cudaMalloc(reinterpret_cast<void**>(&A->dev), L.dev_bytes);
            if (e != cudaSuccess) {
                A->dev = nullptr;
                return vqc::set_error(VQC_ERR_OUT_OF_MEMORY, std::string("cudaMalloc(arena): ") +
                                                                 cudaGetErrorString(e));
            }
            A->dev_cap = L.dev_bytes;
            A->device = dev;
            A->have_last = false;
        }
        const size_t pin_need = direct ? 0 : L.in_bytes + L.out_bytes;
        if (pin_need > A->pin_cap) {
            if (A->pin) cudaFreeHost(A->pin);
            A->pin = nullptr;
            A->pin_cap = 0;
            e = cudaHostAlloc(reinterpret_cast<void**>(&A->pin), pin_need, cudaHostAllocDefault);
            if (e != cudaSuccess) {
                A->pin = nullptr;
                return vqc::set_error(VQC_ERR_OUT_OF_MEMORY, std::string("cudaHostAlloc(staging): ") +
                                                                 cudaGetErrorString(e));
            }
            A->pin_cap = pin_need;
        }
        unsigned char* D = A->dev;
        unsigned char* H = A->pin;
        if (!A->have_last || !(A->last == L)) {   // new workspace placement: initialise it
            if (L.ws0_bytes) {
                vqc_status st = vqc_workspace_init(D + L.ws0, L.ws0_bytes, stream);
                if (st != VQC_OK) return st;
            }
            if (L.ws1_bytes) {
                vqc_status st = vqc_workspace_init(D + L.ws1, L.ws1_bytes, stream);
                if (st != VQC_OK) return st;
            }
            A->last = L;
            A->have_last = true;
        }

        // Direct access: the kernels read x, w, gE and write E, dx, dw in the
        // caller's host arrays themselves; only the workspace is in the arena.
        auto enqueue_direct = [&](cudaStream_t q) -> vqc_status {
            const void* xh = p.num_x > 0 ? x : nullptr;
            const void* wh = p.num_w > 0 ? w : nullptr;
            if (!bwd)
                return vqc_forward(plan, batch, xh, wh, nullptr, expz_out, nullptr,
                                   L.ws0_bytes ? D + L.ws0 : nullptr, L.ws0_bytes, q);
            return vqc_forward_backward(plan, batch, xh, wh, nullptr, grad_expz, expz_out,
                                        (flags & 2) && p.num_x > 0 ? grad_x : nullptr,
                                        (flags & 4) && p.num_w > 0 ? grad_w : nullptr,
                                        L.ws1_bytes ? D + L.ws1 : nullptr, L.ws1_bytes, q);
        };

        // inputs: caller memory -> pinned mirror (one copy to the device below)
        if (!direct) {
            if (p.num_x > 0) std::memcpy(H + L.x, x, (size_t)batch * p.num_x * rs);
            if (p.num_w > 0) std::memcpy(H + L.w, w, (size_t)p.num_w * rs);
            if (bwd) std::memcpy(H + L.g, grad_expz, (size_t)batch * p.n * rs);
        }

        // The device work: input copy, forward, backward, output copy.
        auto enqueue_staged = [&](cudaStream_t q) -> vqc_status {
            cudaError_t ce = cudaMemcpyAsync(D, H, L.in_bytes, cudaMemcpyHostToDevice, q);
            if (ce != cudaSuccess) return cuda_err(ce, "cudaMemcpyAsync(inputs)");
            const void* xd = p.num_x > 0 ? D + L.x : nullptr;
            const void* wd = p.num_w > 0 ? D + L.w : nullptr;
            unsigned char* O = D + L.out;
            const vqc_status r =
                bwd ? vqc_forward_backward(plan, batch, xd, wd, nullptr, D + L.g, O + L.E,
                                           (flags & 2) && p.num_x > 0 ? O + L.dx : nullptr,
                                           (flags & 4) && p.num_w > 0 ? O + L.dw : nullptr,
                                           L.ws1_bytes ? D + L.ws1 : nullptr, L.ws1_bytes, q)
                    : vqc_forward(plan, batch, xd, wd, nullptr, O + L.E, nullptr,
                                  L.ws0_bytes ? D + L.ws0 : nullptr, L.ws0_bytes, q);
            if (r != VQC_OK) return r;
            ce = cudaMemcpyAsync(H + L.in_bytes, O, L.out_bytes, cudaMemcpyDeviceToHost, q);
            if (ce != cudaSuccess) return cuda_err(ce, "cudaMemcpyAsync(outputs)");
            return VQC_OK;
        };
        auto enqueue = [&](cudaStream_t q) -> vqc_status {
            return direct ? enqueue_direct(q) : enqueue_staged(q);
        };
        const bool graphs = !A->graph_failed && env_flag("VQC_HOST_GRAPH", true);
        if (graphs && same_shape && !A->exec) A->exec = capture(A, enqueue);
        A->shape_batch = batch;
        A->shape_flags = flags;
        for (int i = 0; i < 6; ++i) A->shape_ptrs[i] = ptrs[i];
        if (A->exec) {
            e = cudaGraphLaunch(A->exec, s);
            if (e != cudaSuccess) return cuda_err(e, "cudaGraphLaunch");
        } else {
            vqc_status st = enqueue(s);
            if (st != VQC_OK) return st;
        }
        e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) return cuda_err(e, "cudaStreamSynchronize");
        if (direct) return VQC_OK;

        const unsigned char* HO = H + L.in_bytes;
        std::memcpy(expz_out, HO + L.E, (size_t)batch * p.n * rs);
        if (bwd && grad_x && p.num_x > 0) std::memcpy(grad_x, HO + L.dx, (size_t)batch * p.num_x * rs);
        if (bwd && grad_w && p.num_w > 0) std::memcpy(grad_w, HO + L.dw, (size_t)p.num_w * rs);
        return VQC_OK;
    } catch (const std::bad_alloc&) {
        return vqc::set_error(VQC_ERR_OUT_OF_MEMORY, "host allocation failed");
    } catch (...) {
        return vqc::set_error(VQC_ERR_INVALID_ARG, "internal error in vqc_evaluate_host");
    }
}

extern "C" int32_t vqc_host_direct(int32_t device) {
    return env_flag("VQC_HOST_DIRECT", true) && host_direct(device) ? 1 : 0;
}
